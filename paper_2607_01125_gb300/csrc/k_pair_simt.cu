// Pair forward on CUDA cores for fp32 weights and activations (Section 3):
//   y(sigma) = W x + (C + sigma eps Z)(U^T x)
// fp32 inputs have no dense tensor-core path with fp32 accuracy (tf32 keeps a
// 10-bit mantissa), so this kernel serves the fp32 workloads (the 256-wide toy
// graph), which are latency-bound.  64x64 output tile per 256-thread block,
// 4x4 register tile per thread, K staged through shared memory in chunks of 16.
// The epilogue builds the tile's C and Z columns in shared memory once (Z from
// the shared Philox generator) and adds the low-rank term in fp32.
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

constexpr int SB = 64;   // tile rows and cols
constexpr int SK = 16;   // K chunk
constexpr int SR = 32;   // max rank

__global__ void __launch_bounds__(256)
pair_simt_kernel(const float* __restrict__ X, const float* __restrict__ W, const float* __restrict__ P,
                 const float* __restrict__ Cg, float* __restrict__ Y, int64_t rows, int64_t T, int d_in,
                 int d_out, int r, int shared_in, int act, float eps, uint64_t seed, uint64_t query,
                 uint32_t layer_id) {
  __shared__ float As[SK][SB + 4];
  __shared__ float Bs[SK][SB + 4];
  __shared__ float Ct[SB * SR];
  __shared__ float Zt[SB * SR];
  const int tid = threadIdx.x;
  const int tx = tid % 16, ty = tid / 16;
  const int64_t m0 = (int64_t)blockIdx.y * SB;
  const int n0 = blockIdx.x * SB;

  float acc[4][4] = {};
  for (int k0 = 0; k0 < d_in; k0 += SK) {
    __syncthreads();
    for (int v = tid; v < SB * SK; v += 256) {
      const int rr = v / SK, kk = v % SK;
      const int64_t m = m0 + rr;
      const int n = n0 + rr;
      const int k = k0 + kk;
      As[kk][rr] = (m < rows && k < d_in) ? X[m * d_in + k] : 0.f;
      Bs[kk][rr] = (n < d_out && k < d_in) ? W[(int64_t)n * d_in + k] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < SK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[kk][ty * 4 + i]; b[i] = Bs[kk][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
  }

  // ---- epilogue tables: C and Z for the tile's columns, [col][j] ----
  const int64_t e0 = (int64_t)n0 * r;  // multiple of 4 (n0 is a multiple of 64)
  const int n_cols = min(SB, d_out - n0);
  const int n_elem = n_cols * r;
  for (int g = tid; g < (n_elem + 3) / 4; g += 256) {
    const float4 z = z_normals4(seed, layer_id, query, (uint64_t)((e0 >> 2) + g));
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int idx = 4 * g + i;
      if (idx < n_elem) {
        Zt[idx] = z_select(z, i);
        Ct[idx] = Cg[e0 + idx];
      }
    }
  }
  __syncthreads();

  for (int i = 0; i < 4; ++i) {
    const int64_t m = m0 + ty * 4 + i;
    if (m >= rows) continue;
    float p[SR];
#pragma unroll
    for (int j = 0; j < SR; ++j) p[j] = j < r ? P[m * r + j] : 0.f;
    for (int jc = 0; jc < 4; ++jc) {
      const int c = tx * 4 + jc;
      const int n = n0 + c;
      if (n >= d_out) continue;
      float sC = 0.f, sZ = 0.f;
#pragma unroll
      for (int j = 0; j < SR; ++j) {
        if (j < r) {
          sC = fmaf(Ct[c * r + j], p[j], sC);
          sZ = fmaf(Zt[c * r + j], p[j], sZ);
        }
      }
      const float base = acc[i][jc] + sC;
      if (shared_in) {
        Y[m * d_out + n] = apply_act(base + eps * sZ, act);
        Y[(T + m) * d_out + n] = apply_act(base - eps * sZ, act);
      } else {
        const float sg = m < T ? eps : -eps;
        Y[m * d_out + n] = apply_act(base + sg * sZ, act);
      }
    }
  }
}

}  // namespace

int launch_pair_simt(Ctx* ctx, const PairArgs& a) {
  if (a.xdtype != ZOACT_DT_FP32 || a.wtype != ZOACT_DT_FP32 || a.ydtype != ZOACT_DT_FP32)
    return ZOACT_ERR_UNSUPPORTED;
  if (a.r > SR || a.W2) return ZOACT_ERR_UNSUPPORTED;
  dim3 grid((unsigned)((a.d_out + SB - 1) / SB), (unsigned)((a.rows + SB - 1) / SB));
  pair_simt_kernel<<<grid, 256, 0, ctx->stream>>>(
      static_cast<const float*>(a.X), static_cast<const float*>(a.W), a.P, a.C, static_cast<float*>(a.Y),
      a.rows, a.T, a.d_in, a.d_out, a.r, a.shared, a.act, a.eps, a.seed, a.query, a.layer_id); ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
