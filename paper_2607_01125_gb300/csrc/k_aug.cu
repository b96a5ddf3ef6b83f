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
// stream as every other kernel; when a tile's rows span up to S blocks, A_aug
// has S K slots and row t fills slot block(t) mod S, so each slot meets the
// table of the tile's block congruent to it), and the single table T = C otherwise.  With C
// on the tensor cores the epilogue still adds c_b Z_b p: for it this kernel
// also writes Z of every distinct query transposed, Zt[q][j][n] (fp32), so the
// pair kernel copies its tile's columns instead of regenerating them per tile.
// Purely memory-bound and small (rows x r and d_out x r inputs).
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

struct AugBlocks {
  float coef[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t qry[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t zq[ZOACT_MAX_EVAL_BLOCKS];   // distinct queries whose Z is written transposed
  int nzq;
};

// v = hi + lo (+ what bf16 cannot hold): hi = bf16(v), lo = bf16(v - hi); v - hi is exact in fp32.
__device__ __forceinline__ void split16(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__device__ __forceinline__ uint32_t pack_bf16x2(__nv_bfloat16 a, __nv_bfloat16 b) {
  return (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16);
}

// One warp per output row: rows [0, nA) of A_aug, then the nB rows of B_aug
// (block b, column n), then those of B_aug2.  The warp stages the row's r source
// values (and those of the second projection, distinct gated A rows only) in its
// slice of shared memory, then writes the row as bf16 pairs, each lane splitting
// its K columns' source values into hi/lo.  r <= 256.
__global__ void __launch_bounds__(256)
aug_prep_kernel(const float* __restrict__ P, const float* __restrict__ P2, const float* __restrict__ C,
                const float* __restrict__ C2, __nv_bfloat16* __restrict__ A, __nv_bfloat16* __restrict__ B,
                __nv_bfloat16* __restrict__ B2, int64_t rows, int d_out, int r, int ka, int distinct, int full,
                int nb, const __grid_constant__ AugBlocks blk, uint64_t seed, uint32_t lid, uint32_t lid2,
                float* __restrict__ Zt, float* __restrict__ Zt2, int slots, int64_t T) {
  __shared__ float stage[8][2][256];
  const int lane = threadIdx.x & 31;
  float* s0 = stage[threadIdx.x >> 5][0];
  float* s1 = stage[threadIdx.x >> 5][1];
  const int ka_row = distinct ? 2 * ka : ka;          // columns of one slot
  const int ka_tot_a = slots * ka_row;                // A_aug row width
  const int ka_tot = ka_row;                          // B_aug row width
  const int nbB = full ? nb : 1;
  const int64_t nA = rows;
  const int64_t nB = (int64_t)nbB * d_out;
  const int64_t total = nA + (B2 ? 2 * nB : nB);
  const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
  for (int64_t w = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; w < total; w += nwarps) {
    const bool is_a = w < nA;
    bool up = false;
    int64_t orow;
    __syncwarp();                                    // the previous row's readers are done with the stage
    if (is_a) {
      orow = w;
      for (int j = lane; j < r; j += 32) {
        s0[j] = P[w * r + j];
        if (distinct) s1[j] = P2[w * r + j];
      }
    } else {
      const int64_t ib = w - nA;
      up = ib >= nB;
      orow = up ? ib - nB : ib;                      // b * d_out + n
      const int b = (int)(orow / d_out), n = (int)(orow - (int64_t)b * d_out);
      const float cb = full ? blk.coef[b] : 0.f;
      for (int j = lane; j < r; j += 32) {
        const int64_t e = (int64_t)n * r + j;
        float v = (up ? C2 : C)[e];
        if (cb != 0.f)
          v = fmaf(cb, z_select(z_normals4(seed, up ? lid2 : lid, blk.qry[b], (uint64_t)(e >> 2)), (int)(e & 3)), v);
        s0[j] = v;
      }
    }
    __syncwarp();
    __nv_bfloat16* dst = is_a ? A : (up ? B2 : B);
    const int row_w = is_a ? ka_tot_a : ka_tot;
    const int my_slot = (is_a && slots > 1) ? (int)((orow / T) % slots) : 0;
    uint32_t* drow = reinterpret_cast<uint32_t*>(dst + orow * row_w);
    for (int wd = lane; wd < row_w / 2; wd += 32) {
      __nv_bfloat16 o[2];
#pragma unroll
      for (int e2 = 0; e2 < 2; ++e2) {
        const int slot = (2 * wd + e2) / ka_row;
        const int k = 2 * wd + e2 - slot * ka_row;
        const int half = k >= ka ? 1 : 0, kk = k - half * ka;
        const int part = kk / r, j = kk - part * r;
        // A: [hi | hi | lo], B: [hi | lo | hi]
        const bool want_lo = is_a ? part == 2 : part == 1;
        const bool second = is_a && half == 1;       // distinct A: the up projection's parts
        // distinct gated B: gate rows fill the first half, up rows the second
        const bool live = part < 3 && slot == my_slot && (is_a || !distinct || half == (up ? 1 : 0));
        __nv_bfloat16 hi = __float2bfloat16_rn(0.f), lo = hi;
        if (live) split16(second ? s1[j] : s0[j], hi, lo);
        o[e2] = live ? (want_lo ? lo : hi) : __float2bfloat16_rn(0.f);
      }
      drow[wd] = pack_bf16x2(o[0], o[1]);
    }
  }
  // transposed Z tables: Zt[q][j][n] for each distinct query (gate, then up); one thread per
  // (matrix, query, group of 4 ranks, column n), columns fastest so that the stores coalesce
  if (Zt && blk.nzq > 0) {
    const int groups = (r + 3) / 4;
    const int n_mat = Zt2 ? 2 : 1;
    const int64_t items = (int64_t)n_mat * blk.nzq * groups * d_out;
    for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items;
         it += (int64_t)gridDim.x * blockDim.x) {
      const int n = (int)(it % d_out);
      int64_t rest = it / d_out;
      const int jg = (int)(rest % groups);
      rest /= groups;
      const int qi = (int)(rest % blk.nzq);
      const int mat = (int)(rest / blk.nzq);
      float* dst = (mat ? Zt2 : Zt) + (int64_t)qi * r * d_out;
      const uint32_t layer = mat ? lid2 : lid;
      if ((r & 3) == 0) {
        // the four ranks are one Philox group
        const float4 z = z_normals4(seed, layer, blk.zq[qi], (uint64_t)(((int64_t)n * r + 4 * jg) >> 2));
        dst[(int64_t)(4 * jg) * d_out + n] = z.x;
        dst[(int64_t)(4 * jg + 1) * d_out + n] = z.y;
        dst[(int64_t)(4 * jg + 2) * d_out + n] = z.z;
        dst[(int64_t)(4 * jg + 3) * d_out + n] = z.w;
      } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int j = 4 * jg + i;
          if (j < r) {
            const int64_t e = (int64_t)n * r + j;
            dst[(int64_t)j * d_out + n] =
                z_select(z_normals4(seed, layer, blk.zq[qi], (uint64_t)(e >> 2)), (int)(e & 3));
          }
        }
      }
    }
  }
}

}  // namespace

int launch_aug_prep(Ctx* ctx, const PairArgs& a, int mode, int ka, int distinct, int slots, void* A_aug,
                    void* B_aug, void* B_aug2, float* Zt, float* Zt2, const uint64_t* zq, int nzq) {
  AugBlocks blk{};
  for (int b = 0; b < a.nb; ++b) { blk.coef[b] = a.coef[b]; blk.qry[b] = a.qry[b]; }
  for (int i = 0; i < nzq; ++i) blk.zq[i] = zq[i];
  blk.nzq = Zt ? nzq : 0;
  const int full = mode == LOWRANK_ALL_ON_TC;
  const int ka_tot = distinct ? 2 * ka : ka;
  (void)ka_tot;
  const int64_t nbB = full ? a.nb : 1;
  const int64_t total_rows = a.rows + (B_aug2 ? 2 : 1) * nbB * a.d_out;   // one warp per row, 8 per block
  int64_t grid = (total_rows + 7) / 8;
  const int64_t cap = (int64_t)ctx->sm_count * 16;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  aug_prep_kernel<<<(unsigned)grid, 256, 0, ctx->stream>>>(
      a.P, distinct ? a.P2 : nullptr, a.C, a.C2, static_cast<__nv_bfloat16*>(A_aug),
      static_cast<__nv_bfloat16*>(B_aug), static_cast<__nv_bfloat16*>(B_aug2), a.rows, a.d_out, a.r, ka, distinct,
      full, a.nb, blk, a.seed, a.layer_id, a.layer_id2, Zt, Zt2, slots, a.T);
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
