// Operands of the low-rank term on the tensor cores (Section 3: the factor
// (X V_r)(B + mu Z) of the perturbed forward pass as extra K columns of the
// pair-forward MMA).
//
// The low-rank term of an output element is sum_j P[t, j] T[n, j] with P = X U
// (fp32) and T = C + c_b Z_b (fp32).  Both factors are split into 16-bit
// parts, v = hi + lo with hi = bf16(v) and lo = bf16(v - hi), and the three
// largest products are laid out as 3r extra K columns (padded with zeros to
// whole 64-column K-blocks):
//     A_aug row t = [ P_hi | P_hi | P_lo | 0 ]      B_aug row n = [ T_hi | T_lo | T_hi | 0 ]
// so the MMA adds P_hi T_hi + P_hi T_lo + P_lo T_hi, which differs from P T by
// the dropped P_lo T_lo and the rounding of the lo parts: below 2^-15 sum_j
// |P_j| |T_j|.  For a gated pair whose gate and up projections differ, A_aug
// holds both ([gate parts | up parts]) and each B_aug zero-fills the other half.
// B_aug holds one table per evaluation block when the whole term goes to the
// tensor cores (LOWRANK_ALL_ON_TC: T = C + c_b Z_b, Z_b from the same Philox
// stream as every other kernel), and the single table T = C otherwise.
// Purely memory-bound and small (rows x r and d_out x r inputs).
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

struct AugBlocks {
  float coef[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t qry[ZOACT_MAX_EVAL_BLOCKS];
};

// part index of K column k of one layer's aug columns: 0 -> hi, 1 -> hi (A) / lo (B), 2 -> lo (A) / hi (B)
__device__ __forceinline__ void split16(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__device__ __forceinline__ __nv_bfloat16 a_part(float v, int part) {
  __nv_bfloat16 hi, lo;
  split16(v, hi, lo);
  return part == 2 ? lo : hi;
}
__device__ __forceinline__ __nv_bfloat16 b_part(float v, int part) {
  __nv_bfloat16 hi, lo;
  split16(v, hi, lo);
  return part == 1 ? lo : hi;
}

// One thread writes 8 consecutive bf16 of one aug row (a 16-byte store).
// Work items: [0, nA) rows of A_aug, then [nA, nA + nB) rows of B_aug, then B_aug2.
__global__ void __launch_bounds__(256)
aug_prep_kernel(const float* __restrict__ P, const float* __restrict__ P2, const float* __restrict__ C,
                const float* __restrict__ C2, __nv_bfloat16* __restrict__ A, __nv_bfloat16* __restrict__ B,
                __nv_bfloat16* __restrict__ B2, int64_t rows, int d_out, int r, int ka, int distinct, int full,
                int nb, const __grid_constant__ AugBlocks blk, uint64_t seed, uint32_t lid, uint32_t lid2) {
  const int ka_tot = distinct ? 2 * ka : ka;
  const int cpr = ka_tot / 8;                         // 16-byte chunks per row
  const int64_t nA = rows * cpr;
  const int nbB = full ? nb : 1;
  const int64_t nB = (int64_t)nbB * d_out * cpr;
  const int64_t total = nA + (B2 ? 2 * nB : nB);
  for (int64_t it = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; it < total; it += (int64_t)gridDim.x * blockDim.x) {
    alignas(16) __nv_bfloat16 out[8];
    if (it < nA) {
      const int64_t t = it / cpr;
      const int k0 = (int)(it % cpr) * 8;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int k = k0 + i;
        const int half = k / ka, kk = k % ka;          // half 1: the up projection (distinct only)
        const int part = kk / r, j = kk % r;
        const float* src = half ? P2 : P;
        out[i] = part < 3 ? a_part(src[t * r + j], part) : __float2bfloat16_rn(0.f);
      }
      *reinterpret_cast<uint4*>(A + t * ka_tot + k0) = *reinterpret_cast<const uint4*>(out);
    } else {
      const int64_t ib = it - nA;
      const bool up = ib >= nB;
      const int64_t jb = up ? ib - nB : ib;
      const int64_t row = jb / cpr;                     // b * d_out + n
      const int k0 = (int)(jb % cpr) * 8;
      const int b = (int)(row / d_out), n = (int)(row % d_out);
      const float* Cs = up ? C2 : C;
      const uint32_t layer = up ? lid2 : lid;
      const float cb = full ? blk.coef[b] : 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int k = k0 + i;
        const int half = k / ka, kk = k % ka;
        const int part = kk / r, j = kk % r;
        // distinct projections: gate rows use the first half, up rows the second
        const bool live = part < 3 && (!distinct || half == (up ? 1 : 0));
        float v = 0.f;
        if (live) {
          const int64_t e = (int64_t)n * r + j;
          v = Cs[e];
          if (cb != 0.f) v = fmaf(cb, z_select(z_normals4(seed, layer, blk.qry[b], (uint64_t)(e >> 2)), (int)(e & 3)), v);
        }
        out[i] = live ? b_part(v, part) : __float2bfloat16_rn(0.f);
      }
      __nv_bfloat16* dst = up ? B2 : B;
      *reinterpret_cast<uint4*>(dst + row * ka_tot + k0) = *reinterpret_cast<const uint4*>(out);
    }
  }
}

}  // namespace

int launch_aug_prep(Ctx* ctx, const PairArgs& a, int mode, int ka, int distinct, void* A_aug, void* B_aug,
                    void* B_aug2) {
  AugBlocks blk{};
  for (int b = 0; b < a.nb; ++b) { blk.coef[b] = a.coef[b]; blk.qry[b] = a.qry[b]; }
  const int full = mode == LOWRANK_ALL_ON_TC;
  const int ka_tot = distinct ? 2 * ka : ka;
  const int64_t cpr = ka_tot / 8;
  const int64_t nbB = full ? a.nb : 1;
  const int64_t total = a.rows * cpr + (B_aug2 ? 2 : 1) * nbB * a.d_out * cpr;
  int64_t grid = (total + 255) / 256;
  const int64_t cap = (int64_t)ctx->sm_count * 16;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  aug_prep_kernel<<<(unsigned)grid, 256, 0, ctx->stream>>>(
      a.P, distinct ? a.P2 : nullptr, a.C, a.C2, static_cast<__nv_bfloat16*>(A_aug),
      static_cast<__nv_bfloat16*>(B_aug), static_cast<__nv_bfloat16*>(B_aug2), a.rows, a.d_out, a.r, ka, distinct,
      full, a.nb, blk, a.seed, a.layer_id, a.layer_id2);
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
