// ZO-Adam and ZO-SGD over the flat coefficient arenas (Section 3: Adam on the
// estimated coefficient gradient; Table 1 "Full SGD"; Appendix B: weight decay 0).
//
//   g = (1/q) sum_j a_j Z(seed, layer_id, query_j)   (Z regenerated, never stored;
//                                                      q = 1, a = a_pair: the two-sided g = a Z)
//   m = b1 m + (1 - b1) g ;  v = b2 v + (1 - b2) g^2
//   C -= (lr / (1 - b1^t)) * m / (sqrt(v) / sqrt(1 - b2^t) + adam_eps)
//
// Purely HBM-bound: each coefficient costs 24 bytes (read and write C, m, v).
// A thread owns groups of 4 consecutive elements: one Philox call yields the 4
// normals, and C, m, v move as 16-byte vectors.  The layer table (offsets,
// layer ids) travels in the kernel parameters; a group finds its layer by binary
// search.  a is read from device memory (the loss kernel's output), so a whole
// ZO step runs without a host synchronisation.  With q queries every group
// draws q Philox groups (one per query) and sums a_j z_j in query order.
#include "internal.h"
#include "philox.cuh"

#include <cmath>

namespace zoact {
namespace {

constexpr int ADAM_TABLE = 256;  // layers per launch

struct QueryList {
  uint64_t q[ZOACT_MAX_EVAL_BLOCKS];
};

struct AdamTable {
  int64_t begin[ADAM_TABLE];
  int64_t end[ADAM_TABLE];
  uint32_t layer_id[ADAM_TABLE];
  int n;
};

__device__ __forceinline__ int find_block(const AdamTable& t, int64_t e) {
  int lo = 0, hi = t.n - 1;
  while (lo < hi) {                  // last block with begin <= e
    const int mid = (lo + hi + 1) >> 1;
    if (t.begin[mid] <= e) lo = mid; else hi = mid - 1;
  }
  return lo;
}

template <bool SGD>
__global__ void __launch_bounds__(256)
zo_update_kernel(float* __restrict__ C, float* __restrict__ m, float* __restrict__ v, const __grid_constant__ AdamTable tab,
                 int64_t g_begin, int64_t g_end, const double* __restrict__ a_dev, int nq,
                 const __grid_constant__ QueryList qs, float lr, float b1, float b2, float adam_eps, float step_size,
                 float inv_sqrt_bc2, uint64_t seed, int* __restrict__ status) {
  pdl_wait();                              // a (the loss kernel's output) is visible
  pdl_trigger();
  bool finite = true;
  for (int j = 0; j < nq; ++j) finite = finite && isfinite(a_dev[j]);
  if (!finite) {
    if (blockIdx.x == 0 && threadIdx.x == 0) record_error(status, ZOACT_ERR_NONFINITE);
    return;
  }
  const float a0 = (float)a_dev[0];
  const float inv_q = 1.0f / (float)nq;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g = g_begin + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < g_end; g += stride) {
    const int64_t e = 4 * g;
    const int b = find_block(tab, e);
    if (e >= tab.end[b]) continue;                       // gap between blocks
    const int64_t local = e - tab.begin[b];              // element index inside the layer's [d_out, r]
    float gz[4];
    {
      const float4 z = z_normals4(seed, tab.layer_id[b], qs.q[0], (uint64_t)(local >> 2));
      gz[0] = a0 * z.x; gz[1] = a0 * z.y; gz[2] = a0 * z.z; gz[3] = a0 * z.w;
    }
    if (nq > 1) {
      for (int j = 1; j < nq; ++j) {
        const float aj = (float)a_dev[j];
        const float4 z = z_normals4(seed, tab.layer_id[b], qs.q[j], (uint64_t)(local >> 2));
        gz[0] = fmaf(aj, z.x, gz[0]); gz[1] = fmaf(aj, z.y, gz[1]);
        gz[2] = fmaf(aj, z.z, gz[2]); gz[3] = fmaf(aj, z.w, gz[3]);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) gz[i] *= inv_q;
    }
    const bool full = e + 4 <= tab.end[b];
    if (SGD) {
      if (full) {
        float4 c = *reinterpret_cast<float4*>(C + e);
        c.x -= lr * gz[0]; c.y -= lr * gz[1]; c.z -= lr * gz[2]; c.w -= lr * gz[3];
        *reinterpret_cast<float4*>(C + e) = c;
      } else {
        for (int i = 0; i < 4 && e + i < tab.end[b]; ++i) C[e + i] -= lr * gz[i];
      }
      continue;
    }
    float cv[4], mv[4], vv[4];
    if (full) {
      const float4 c4 = *reinterpret_cast<const float4*>(C + e);
      const float4 m4 = *reinterpret_cast<const float4*>(m + e);
      const float4 v4 = *reinterpret_cast<const float4*>(v + e);
      cv[0] = c4.x; cv[1] = c4.y; cv[2] = c4.z; cv[3] = c4.w;
      mv[0] = m4.x; mv[1] = m4.y; mv[2] = m4.z; mv[3] = m4.w;
      vv[0] = v4.x; vv[1] = v4.y; vv[2] = v4.z; vv[3] = v4.w;
    } else {
      for (int i = 0; i < 4; ++i) {
        const bool in = e + i < tab.end[b];
        cv[i] = in ? C[e + i] : 0.f; mv[i] = in ? m[e + i] : 0.f; vv[i] = in ? v[e + i] : 0.f;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      mv[i] = b1 * mv[i] + (1.0f - b1) * gz[i];
      vv[i] = b2 * vv[i] + (1.0f - b2) * gz[i] * gz[i];
      const float denom = sqrtf(vv[i]) * inv_sqrt_bc2 + adam_eps;
      cv[i] = cv[i] - step_size * (mv[i] / denom);
    }
    if (full) {
      *reinterpret_cast<float4*>(C + e) = make_float4(cv[0], cv[1], cv[2], cv[3]);
      *reinterpret_cast<float4*>(m + e) = make_float4(mv[0], mv[1], mv[2], mv[3]);
      *reinterpret_cast<float4*>(v + e) = make_float4(vv[0], vv[1], vv[2], vv[3]);
    } else {
      for (int i = 0; i < 4 && e + i < tab.end[b]; ++i) { C[e + i] = cv[i]; m[e + i] = mv[i]; v[e + i] = vv[i]; }
    }
  }
}

}  // namespace

int launch_adam(Ctx* ctx, float* C, float* m, float* v, const zoact_coeff_block* blocks, int n_blocks,
                const double* a, int q, const uint64_t* queries, float lr, float b1, float b2, float adam_eps,
                int64_t step, uint64_t seed, int sgd) {
  if (q < 1 || q > ZOACT_MAX_EVAL_BLOCKS) return ZOACT_ERR_INVALID_ARG;
  QueryList qs{};
  for (int j = 0; j < q; ++j) qs.q[j] = queries[j];
  const double bc1 = 1.0 - std::pow((double)b1, (double)step);
  const double bc2 = 1.0 - std::pow((double)b2, (double)step);
  const float step_size = sgd ? 0.f : (float)((double)lr / bc1);
  const float inv_sqrt_bc2 = sgd ? 0.f : (float)(1.0 / std::sqrt(bc2));
  for (int base = 0; base < n_blocks; base += ADAM_TABLE) {
    AdamTable tab;
    tab.n = n_blocks - base < ADAM_TABLE ? n_blocks - base : ADAM_TABLE;
    int64_t lo = INT64_MAX, hi = 0;
    for (int i = 0; i < tab.n; ++i) {
      const zoact_coeff_block& bl = blocks[base + i];
      tab.begin[i] = bl.offset;
      tab.end[i] = bl.offset + (int64_t)bl.d_out * bl.r;
      tab.layer_id[i] = bl.layer_id;
      if (tab.begin[i] < lo) lo = tab.begin[i];
      if (tab.end[i] > hi) hi = tab.end[i];
    }
    if (hi <= lo) continue;
    const int64_t g_begin = lo / 4, g_end = (hi + 3) / 4;
    int64_t nb = (g_end - g_begin + 255) / 256;
    const int64_t cap = (int64_t)ctx->sm_count * 8;
    if (nb > cap) nb = cap;
    ZOACT_CUDA_TRY(launch_pdl(ctx, sgd ? zo_update_kernel<true> : zo_update_kernel<false>, dim3((unsigned)nb),
                              dim3(256), 0, C, m, v, tab, g_begin, g_end, a, q, qs, lr, b1, b2, adam_eps, step_size,
                              inv_sqrt_bc2, seed, ctx->d_status));
    ++ctx->n_launch;
  }
  return ZOACT_OK;
}

}  // namespace zoact
