// Subspace diagnostics of Section 5.3, on the device:
//   overlap  ||U_a^T U_b||_F^2 / r_a        (stability of the basis across training stages)
//   energy   ||U^T G||_F^2 / ||G||_F^2       (share of a weight gradient inside the basis)
// Both are the squared Frobenius norm of M = U^T G for a tall U [d, r] (fp32) and
// a matrix G [d, n] (fp32 / bf16 / fp16; for the overlap G = U_b).  Off the hot
// path: CUDA cores, deterministic.  Pass 1 (grid: 64-column tiles of G x
// K-splits): each block stages 32-row chunks of U and G in shared memory and
// accumulates its r x 64 slice of M in fp32 registers (thread (ty, tx) owns rows
// ty + 16a and columns tx + 16b), writes the K-split's partial M and its share of
// ||G||^2.  Pass 2: every element of M is the K-split partials added in split
// order, squared and summed in fp64; the last block (atomic ticket) adds the
// block sums in order and writes the results.
#include "internal.h"

namespace zoact {
namespace {

constexpr int DK = 32;     // rows of U and G per shared-memory chunk
constexpr int DCOLS = 64;  // columns of G per block

template <typename TG> __device__ __forceinline__ float gval(const TG* G, int64_t i) { return to_f32<TG>(G[i]); }

template <int RA, typename TG>
__global__ void __launch_bounds__(256)
utg_partial_kernel(const float* __restrict__ U, const TG* __restrict__ G, int d, int r, int64_t n, int kchunk,
                   float* __restrict__ Mpart, double* __restrict__ g2part) {
  __shared__ float Us[DK][RA * 16];
  __shared__ float Gs[DK][DCOLS + 1];
  __shared__ double red[8];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t col0 = (int64_t)blockIdx.x * DCOLS;
  const int k_begin = blockIdx.y * kchunk;
  const int k_end = min(d, k_begin + kchunk);
  float acc[RA][4];
#pragma unroll
  for (int a = 0; a < RA; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
  double g2 = 0.0;
  for (int k0 = k_begin; k0 < k_end; k0 += DK) {
    for (int idx = tid; idx < DK * RA * 16; idx += 256) {
      const int kk = idx / (RA * 16), i = idx % (RA * 16);
      Us[kk][i] = (k0 + kk < k_end && i < r) ? U[(int64_t)(k0 + kk) * r + i] : 0.f;
    }
    float gs = 0.f;
    for (int idx = tid; idx < DK * DCOLS; idx += 256) {
      const int kk = idx / DCOLS, j = idx % DCOLS;
      const float v = (k0 + kk < k_end && col0 + j < n) ? gval<TG>(G, (int64_t)(k0 + kk) * n + col0 + j) : 0.f;
      Gs[kk][j] = v;
      gs = fmaf(v, v, gs);
    }
    g2 += gs;
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < DK; ++kk) {
      float g[4];
#pragma unroll
      for (int b = 0; b < 4; ++b) g[b] = Gs[kk][tx + 16 * b];
#pragma unroll
      for (int a = 0; a < RA; ++a) {
        const float u = Us[kk][ty + 16 * a];
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(u, g[b], acc[a][b]);
      }
    }
    __syncthreads();
  }
  float* Mp = Mpart + (int64_t)blockIdx.y * r * n;
#pragma unroll
  for (int a = 0; a < RA; ++a) {
    const int i = ty + 16 * a;
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int64_t j = col0 + tx + 16 * b;
      if (i < r && j < n) Mp[(int64_t)i * n + j] = acc[a][b];
    }
  }
  // this block's share of ||G||^2 (every element of G is loaded by exactly one block)
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) g2 += __shfl_xor_sync(0xffffffffu, g2, o);
  if ((tid & 31) == 0) red[tid >> 5] = g2;
  __syncthreads();
  if (tid == 0) {
    double s = 0.0;
    for (int w = 0; w < 8; ++w) s += red[w];
    g2part[(int64_t)blockIdx.y * gridDim.x + blockIdx.x] = s;
  }
}

// out[0] = sum (sum_k Mpart[k])^2, out[1] = sum g2part, out[2] = out[0] * scale / (out[1] or 1)
__global__ void __launch_bounds__(256)
utg_finish_kernel(const float* __restrict__ Mpart, int ks, int64_t count, const double* __restrict__ g2part,
                  int n_g2, double* __restrict__ bsum, unsigned int* __restrict__ ticket, double scale, int ratio_by_g2,
                  double* __restrict__ out) {
  double s = 0.0;
  for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < count; e += (int64_t)gridDim.x * blockDim.x) {
    float m = 0.f;
    for (int k = 0; k < ks; ++k) m += Mpart[(int64_t)k * count + e];
    s += (double)m * (double)m;
  }
  __shared__ double red[8];
  __shared__ bool last;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    for (int w = 0; w < 8; ++w) t += red[w];
    bsum[blockIdx.x] = t;
    __threadfence();
    last = atomicAdd(ticket, 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!last || threadIdx.x != 0) return;
  __threadfence();
  double num = 0.0, den = 0.0;
  for (unsigned int b = 0; b < gridDim.x; ++b) num += __ldcg(bsum + b);
  for (int b = 0; b < n_g2; ++b) den += __ldcg(g2part + b);
  out[0] = num;
  out[1] = den;
  out[2] = ratio_by_g2 ? (den > 0.0 ? num / den : 0.0) : num * scale;
  *ticket = 0u;
}

template <typename TG>
int run_utg(Ctx* ctx, const float* U, const TG* G, int d, int r, int64_t n, double scale, int ratio_by_g2,
            double* out) {
  const int64_t col_tiles = (n + DCOLS - 1) / DCOLS;
  if (col_tiles > 65535 * 64LL) return ZOACT_ERR_UNSUPPORTED;
  int ks = (int)((2LL * ctx->sm_count + col_tiles - 1) / col_tiles);
  const int max_ks = (d + 255) / 256;
  if (ks > max_ks) ks = max_ks;
  if (ks < 1) ks = 1;
  int kchunk = (d + ks - 1) / ks;
  kchunk = (kchunk + DK - 1) / DK * DK;
  ks = (d + kchunk - 1) / kchunk;
  const int64_t count = (int64_t)r * n;
  int64_t fin_blocks = (count + 255) / 256;
  if (fin_blocks > 4LL * ctx->sm_count) fin_blocks = 4LL * ctx->sm_count;
  const size_t m_bytes = ((size_t)ks * count * sizeof(float) + 255) / 256 * 256;
  const size_t g_bytes = ((size_t)ks * col_tiles * sizeof(double) + 255) / 256 * 256;
  uint8_t* buf = static_cast<uint8_t*>(scratch(ctx, SLOT_DIAG, m_bytes + g_bytes + (size_t)fin_blocks * 8));
  if (!buf) return ZOACT_ERR_NOMEM;
  float* Mpart = reinterpret_cast<float*>(buf);
  double* g2part = reinterpret_cast<double*>(buf + m_bytes);
  double* bsum = reinterpret_cast<double*>(buf + m_bytes + g_bytes);
  const dim3 grid((unsigned)col_tiles, (unsigned)ks);
  const int ra = (r + 15) / 16;
#define ZOACT_UTG(RA)                                                                                    \
  utg_partial_kernel<RA, TG><<<grid, 256, 0, ctx->stream>>>(U, G, d, r, n, kchunk, Mpart, g2part)
  if (ra <= 1) ZOACT_UTG(1);
  else if (ra <= 2) ZOACT_UTG(2);
  else if (ra <= 4) ZOACT_UTG(4);
  else if (ra <= 8) ZOACT_UTG(8);
  else ZOACT_UTG(16);
#undef ZOACT_UTG
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  utg_finish_kernel<<<(unsigned)fin_blocks, 256, 0, ctx->stream>>>(Mpart, ks, count, g2part, (int)(ks * col_tiles), bsum,
                                                                   ctx->d_tickets + 2, scale, ratio_by_g2, out);
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace

int launch_subspace_overlap(Ctx* ctx, const float* Ua, const float* Ub, int d, int ra, int rb, double* out) {
  return run_utg<float>(ctx, Ua, Ub, d, ra, rb, 1.0 / ra, 0, out);
}

int launch_gradient_energy(Ctx* ctx, const float* U, int d_in, int r, const void* G, int gdtype, int64_t n,
                           double* out) {
  switch (gdtype) {
    case ZOACT_DT_FP32: return run_utg(ctx, U, static_cast<const float*>(G), d_in, r, n, 1.0, 1, out);
    case ZOACT_DT_BF16: return run_utg(ctx, U, static_cast<const __nv_bfloat16*>(G), d_in, r, n, 1.0, 1, out);
    case ZOACT_DT_FP16: return run_utg(ctx, U, static_cast<const __half*>(G), d_in, r, n, 1.0, 1, out);
    default: return ZOACT_ERR_INVALID_ARG;
  }
}

}  // namespace zoact
