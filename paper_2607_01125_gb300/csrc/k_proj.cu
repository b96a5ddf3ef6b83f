// Low-rank projection P = X U  (each row: p = U^T x, the factor (X V_r) of the
// perturbed forward pass in Section 3).
//
// X [rows, d_in] (fp32 / bf16 / fp16), U [d_in, r] fp32, P [rows, r] fp32.
// HBM-bound on X: every element of X is read once.  A block owns 128 rows and
// one K-range (split-K so the grid covers every SM); K is staged through shared
// memory in chunks of 32, converted to fp32, and each thread accumulates a 4x4
// register tile (4 rows x 4 basis columns) in fp32.  With more than one K-range
// the partial tiles go to scratch and a second kernel adds them in a fixed
// order, so the result does not depend on scheduling.
#include "internal.h"

namespace zoact {
namespace {

constexpr int PROJ_RB = 128;  // rows per block
constexpr int PROJ_KC = 32;   // K chunk

template <typename TX>
__device__ __forceinline__ void load_x_chunk(float (*Xs)[PROJ_KC + 1], const TX* __restrict__ X,
                                             int64_t rows, int ld, int k_lim, int64_t row0, int k0,
                                             int tid, int nthreads);

template <>
__device__ __forceinline__ void load_x_chunk<float>(float (*Xs)[PROJ_KC + 1], const float* __restrict__ X,
                                                    int64_t rows, int ld, int k_lim, int64_t row0, int k0,
                                                    int tid, int nthreads) {
  constexpr int VPR = PROJ_KC / 4;  // float4 vectors per row
  for (int v = tid; v < PROJ_RB * VPR; v += nthreads) {
    const int rr = v / VPR, kk = (v % VPR) * 4;
    const int64_t row = row0 + rr;
    const int k = k0 + kk;
    float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
    if (row < rows && k < k_lim) x = *reinterpret_cast<const float4*>(X + row * ld + k);
    Xs[rr][kk + 0] = x.x; Xs[rr][kk + 1] = x.y; Xs[rr][kk + 2] = x.z; Xs[rr][kk + 3] = x.w;
  }
}

template <typename T16>
__device__ __forceinline__ void load_x_chunk16(float (*Xs)[PROJ_KC + 1], const T16* __restrict__ X,
                                               int64_t rows, int ld, int k_lim, int64_t row0, int k0,
                                               int tid, int nthreads) {
  constexpr int VPR = PROJ_KC / 8;  // 16-byte vectors per row
  for (int v = tid; v < PROJ_RB * VPR; v += nthreads) {
    const int rr = v / VPR, kk = (v % VPR) * 8;
    const int64_t row = row0 + rr;
    const int k = k0 + kk;
    uint4 raw = make_uint4(0, 0, 0, 0);
    if (row < rows && k < k_lim) raw = *reinterpret_cast<const uint4*>(X + row * ld + k);
    const T16* e = reinterpret_cast<const T16*>(&raw);
#pragma unroll
    for (int i = 0; i < 8; ++i) Xs[rr][kk + i] = to_f32<T16>(e[i]);
  }
}

template <>
__device__ __forceinline__ void load_x_chunk<__nv_bfloat16>(float (*Xs)[PROJ_KC + 1],
                                                            const __nv_bfloat16* __restrict__ X, int64_t rows,
                                                            int ld, int k_lim, int64_t row0, int k0, int tid,
                                                            int nthreads) {
  load_x_chunk16(Xs, X, rows, ld, k_lim, row0, k0, tid, nthreads);
}
template <>
__device__ __forceinline__ void load_x_chunk<__half>(float (*Xs)[PROJ_KC + 1], const __half* __restrict__ X,
                                                     int64_t rows, int ld, int k_lim, int64_t row0, int k0,
                                                     int tid, int nthreads) {
  load_x_chunk16(Xs, X, rows, ld, k_lim, row0, k0, tid, nthreads);
}

// RPAD: basis columns padded to a power of two >= 4; blockDim = 32 * RPAD / 4.
// r columns of U (row stride ldu) -> out rows of stride ld_out (split s at out + s * rows * ld_out).
template <typename TX, int RPAD>
__global__ void __launch_bounds__(8 * RPAD)
proj_kernel(const TX* __restrict__ X, const float* __restrict__ U, float* __restrict__ out, int64_t rows,
            int d_in, int r, int k_per_split, int ldu, int ld_out) {
  constexpr int NCG = RPAD / 4;        // column groups
  constexpr int NT = 32 * NCG;         // threads
  __shared__ float Xs[PROJ_RB][PROJ_KC + 1];
  __shared__ __align__(16) float Us[PROJ_KC][RPAD];
  const int tid = threadIdx.x;
  const int cg = tid % NCG, rg = tid / NCG;  // 32 row groups of 4 rows
  const int64_t row0 = (int64_t)blockIdx.x * PROJ_RB;
  const int split = blockIdx.y;
  const int k_begin = split * k_per_split;
  const int k_end = min(d_in, k_begin + k_per_split);

  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int c = 0; c < 4; ++c) acc[i][c] = 0.f;

  for (int k0 = k_begin; k0 < k_end; k0 += PROJ_KC) {
    __syncthreads();
    load_x_chunk<TX>(Xs, X, rows, d_in, k_end, row0, k0, tid, NT);
    for (int v = tid; v < PROJ_KC * RPAD; v += NT) {
      const int kk = v / RPAD, j = v % RPAD;
      const int k = k0 + kk;
      Us[kk][j] = (k < k_end && j < r) ? U[(int64_t)k * ldu + j] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < PROJ_KC; ++kk) {
      const float4 u = *reinterpret_cast<const float4*>(&Us[kk][cg * 4]);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float x = Xs[rg * 4 + i][kk];
        acc[i][0] = fmaf(x, u.x, acc[i][0]);
        acc[i][1] = fmaf(x, u.y, acc[i][1]);
        acc[i][2] = fmaf(x, u.z, acc[i][2]);
        acc[i][3] = fmaf(x, u.w, acc[i][3]);
      }
    }
  }
  float* dst = out + (int64_t)split * rows * ld_out;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t row = row0 + rg * 4 + i;
    if (row >= rows) continue;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
      const int j = cg * 4 + c;
      if (j < r) dst[row * ld_out + j] = acc[i][c];
    }
  }
}

// P[t, j0 + j] (row stride ldp) = sum over splits of part[split][t][j], j < rg, in split order.
__global__ void splitk_reduce_kernel(const float* __restrict__ part, float* __restrict__ P, int64_t n,
                                     int splits, int rg, int ldp, int j0) {
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += part[(int64_t)k * n + i];
    const int64_t t = i / rg;
    P[t * ldp + j0 + (i - t * rg)] = s;
  }
}

template <typename TX>
int proj_dispatch(Ctx* ctx, const TX* X, int64_t rows, int d_in, const float* U, int r, float* P) {
  const int64_t row_blocks = (rows + PROJ_RB - 1) / PROJ_RB;
  // enough K-splits to give every SM about two blocks, each split >= 256 wide
  int splits = (int)((2LL * ctx->sm_count + row_blocks - 1) / row_blocks);
  const int max_splits = (d_in + 255) / 256;
  if (splits > max_splits) splits = max_splits;
  if (splits < 1) splits = 1;
  int k_per_split = (d_in + splits - 1) / splits;
  k_per_split = (k_per_split + PROJ_KC - 1) / PROJ_KC * PROJ_KC;
  splits = (d_in + k_per_split - 1) / k_per_split;
  dim3 grid((unsigned)row_blocks, (unsigned)splits);
  // groups of up to 32 basis columns, one launch each
  for (int j0 = 0; j0 < r; j0 += 32) {
    const int rg = r - j0 < 32 ? r - j0 : 32;
    float* out = P + j0;
    int ld_out = r;
    if (splits > 1) {
      out = static_cast<float*>(scratch(ctx, SLOT_SPLITK, (size_t)splits * rows * rg * sizeof(float)));
      if (!out) return ZOACT_ERR_NOMEM;
      ld_out = rg;
    }
    const float* Ug = U + j0;
    const int rp = rg <= 4 ? 4 : rg <= 8 ? 8 : rg <= 16 ? 16 : 32;
    switch (rp) {
      case 4: proj_kernel<TX, 4><<<grid, 32, 0, ctx->stream>>>(X, Ug, out, rows, d_in, rg, k_per_split, r, ld_out); break;
      case 8: proj_kernel<TX, 8><<<grid, 64, 0, ctx->stream>>>(X, Ug, out, rows, d_in, rg, k_per_split, r, ld_out); break;
      case 16: proj_kernel<TX, 16><<<grid, 128, 0, ctx->stream>>>(X, Ug, out, rows, d_in, rg, k_per_split, r, ld_out); break;
      default: proj_kernel<TX, 32><<<grid, 256, 0, ctx->stream>>>(X, Ug, out, rows, d_in, rg, k_per_split, r, ld_out); break;
    }
    ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
    if (splits > 1) {
      const int64_t n = rows * rg;
      int64_t blocks = (n + 255) / 256;
      if (blocks > 4LL * ctx->sm_count) blocks = 4LL * ctx->sm_count;
      splitk_reduce_kernel<<<(unsigned)blocks, 256, 0, ctx->stream>>>(out, P, n, splits, rg, r, j0);
      ++ctx->n_launch;
      ZOACT_CHECK_LAUNCH();
    }
  }
  return ZOACT_OK;
}

}  // namespace

int launch_lowrank_proj(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U, int r,
                        float* P) {
  if (rows <= 0) return ZOACT_OK;
  switch (xdtype) {
    case ZOACT_DT_FP32: return proj_dispatch(ctx, static_cast<const float*>(X), rows, d_in, U, r, P);
    case ZOACT_DT_BF16:
    case ZOACT_DT_FP16: return launch_lowrank_proj_tc(ctx, X, xdtype, rows, d_in, U, r, P);
    default: return ZOACT_ERR_INVALID_ARG;
  }
}

namespace {

// Same kernels, with the split-K partials in a caller-given buffer of part_floats
// floats (no allocation): as many K-splits as fit, at least one.
template <typename TX>
int proj_dispatch_into(Ctx* ctx, const TX* X, int64_t rows, int d_in, const float* U, int r, float* P, float* part,
                       int64_t part_floats) {
  const int64_t row_blocks = (rows + PROJ_RB - 1) / PROJ_RB;
  int splits = (int)((2LL * ctx->sm_count + row_blocks - 1) / row_blocks);
  const int max_splits = (d_in + 255) / 256;
  if (splits > max_splits) splits = max_splits;
  const int64_t fit = part ? part_floats / (rows * r) : 0;
  if (splits > fit) splits = (int)fit;
  if (splits < 1) splits = 1;
  int k_per_split = (d_in + splits - 1) / splits;
  k_per_split = (k_per_split + PROJ_KC - 1) / PROJ_KC * PROJ_KC;
  splits = (d_in + k_per_split - 1) / k_per_split;
  float* out = splits > 1 ? part : P;
  dim3 grid((unsigned)row_blocks, (unsigned)splits);
  const int rp = r <= 4 ? 4 : r <= 8 ? 8 : r <= 16 ? 16 : 32;
  switch (rp) {
    case 4: proj_kernel<TX, 4><<<grid, 32, 0, ctx->stream>>>(X, U, out, rows, d_in, r, k_per_split, r, r); break;
    case 8: proj_kernel<TX, 8><<<grid, 64, 0, ctx->stream>>>(X, U, out, rows, d_in, r, k_per_split, r, r); break;
    case 16: proj_kernel<TX, 16><<<grid, 128, 0, ctx->stream>>>(X, U, out, rows, d_in, r, k_per_split, r, r); break;
    default: proj_kernel<TX, 32><<<grid, 256, 0, ctx->stream>>>(X, U, out, rows, d_in, r, k_per_split, r, r); break;
  }
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  if (splits > 1) {
    const int64_t n = rows * r;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 4LL * ctx->sm_count) blocks = 4LL * ctx->sm_count;
    splitk_reduce_kernel<<<(unsigned)blocks, 256, 0, ctx->stream>>>(out, P, n, splits, r, r, 0);
    ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
  }
  return ZOACT_OK;
}

}  // namespace

int launch_lowrank_proj_into(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U, int r,
                             float* P, float* part, int64_t part_floats) {
  if (rows <= 0) return ZOACT_OK;
  switch (xdtype) {
    case ZOACT_DT_FP32:
      return proj_dispatch_into(ctx, static_cast<const float*>(X), rows, d_in, U, r, P, part, part_floats);
    case ZOACT_DT_BF16:
      return proj_dispatch_into(ctx, static_cast<const __nv_bfloat16*>(X), rows, d_in, U, r, P, part, part_floats);
    case ZOACT_DT_FP16:
      return proj_dispatch_into(ctx, static_cast<const __half*>(X), rows, d_in, U, r, P, part, part_floats);
    default: return ZOACT_ERR_INVALID_ARG;
  }
}

}  // namespace zoact
