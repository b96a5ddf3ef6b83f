// Pair / multi-point forward on CUDA cores for fp32 weights and activations
// (Section 3; Algorithm 2):
//   y_b = W x + (C + c_b Z_b)(U^T x)      for the evaluation blocks b
// fp32 inputs have no dense tensor-core path with fp32 accuracy (tf32 keeps a
// 10-bit mantissa), so this kernel serves the fp32 workloads (the 256-wide toy
// graph), which are latency-bound.  64x64 output tile per 256-thread block,
// 4x4 register tile per thread, K staged through shared memory in chunks of 16.
// The epilogue builds the table C + c_b Z_b of the tile's columns in shared
// memory for one block and 32 ranks at a time (Z from the shared Philox
// generator) and adds the low-rank term in fp32: stacked rows use their own
// block, shared rows are written once per block.
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

constexpr int SB = 64;   // tile rows and cols
constexpr int SK = 16;   // K chunk
constexpr int SR = 32;   // ranks per epilogue table chunk

struct EvalBlocks {
  int nb;
  float coef[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t qry[ZOACT_MAX_EVAL_BLOCKS];
};

__global__ void __launch_bounds__(256)
pair_simt_kernel(const float* __restrict__ X, const float* __restrict__ W, const float* __restrict__ P,
                 const float* __restrict__ Cg, float* __restrict__ Y, int64_t rows, int64_t T, int d_in,
                 int d_out, int r, int shared_in, int act, const EvalBlocks blk, uint64_t seed,
                 uint32_t layer_id) {
  __shared__ float As[SK][SB + 4];
  __shared__ float Bs[SK][SB + 4];
  __shared__ float Tt[SB * SR];
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

  // blocks this tile's rows touch (all of them when the input is shared)
  int b_first = 0, b_last = blk.nb - 1;
  if (!shared_in) {
    const int64_t last = (m0 + SB < rows ? m0 + SB : rows) - 1;
    b_first = (int)(m0 / T);
    b_last = (int)(last / T);
  }
  const int n_cols = min(SB, d_out - n0);
  for (int b = b_first; b <= b_last; ++b) {
    const float cb = blk.coef[b];
    float sl[4][4] = {};
    // the low-rank term in chunks of SR ranks: table C + c_b Z_b of the tile's columns, [col][j]
    for (int jc = 0; jc < r; jc += SR) {
      const int rc = min(SR, r - jc);
      __syncthreads();
      for (int idx = tid; idx < n_cols * rc; idx += 256) {
        const int c = idx / rc, j = jc + idx % rc;
        const int64_t e = (int64_t)(n0 + c) * r + j;
        const float z = cb != 0.f ? z_select(z_normals4(seed, layer_id, blk.qry[b], (uint64_t)(e >> 2)), (int)(e & 3))
                                  : 0.f;
        Tt[c * SR + (j - jc)] = fmaf(cb, z, Cg[e]);
      }
      __syncthreads();
      for (int i = 0; i < 4; ++i) {
        const int64_t m = m0 + ty * 4 + i;
        if (m >= rows || (!shared_in && m / T != b)) continue;
        for (int jj = 0; jj < rc; ++jj) {
          const float pj = P[m * r + jc + jj];
#pragma unroll
          for (int jc4 = 0; jc4 < 4; ++jc4) {
            const int c = tx * 4 + jc4;
            if (c < n_cols) sl[i][jc4] = fmaf(Tt[c * SR + jj], pj, sl[i][jc4]);
          }
        }
      }
    }
    for (int i = 0; i < 4; ++i) {
      const int64_t m = m0 + ty * 4 + i;
      if (m >= rows || (!shared_in && m / T != b)) continue;
      const int64_t row = shared_in ? (int64_t)b * T + m : m;
      for (int jc4 = 0; jc4 < 4; ++jc4) {
        const int n = n0 + tx * 4 + jc4;
        if (n < d_out) Y[row * d_out + n] = apply_act(acc[i][jc4] + sl[i][jc4], act);
      }
    }
  }
}

}  // namespace

int launch_pair_simt(Ctx* ctx, const PairArgs& a) {
  if (a.nseg > 1) return ZOACT_ERR_UNSUPPORTED;     // layers run as one: 16-bit activations only
  if (a.xdtype != ZOACT_DT_FP32 || a.wtype != ZOACT_DT_FP32 || a.ydtype != ZOACT_DT_FP32)
    return ZOACT_ERR_UNSUPPORTED;
  if (a.W2) return ZOACT_ERR_UNSUPPORTED;
  EvalBlocks blk{};
  blk.nb = a.nb;
  for (int b = 0; b < a.nb; ++b) { blk.coef[b] = a.coef[b]; blk.qry[b] = a.qry[b]; }
  dim3 grid((unsigned)((a.d_out + SB - 1) / SB), (unsigned)((a.rows + SB - 1) / SB));
  pair_simt_kernel<<<grid, 256, 0, ctx->stream>>>(
      static_cast<const float*>(a.X), static_cast<const float*>(a.W), a.P, a.C, static_cast<float*>(a.Y),
      a.rows, a.T, a.d_in, a.d_out, a.r, a.shared, a.act, blk, a.seed, a.layer_id); ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
