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
  // layers run as one (B rows only): row n of the table belongs to layer s with seg_off[s] <= n <
  // seg_off[s + 1]; its T = C_s + c_b Z_b takes C_s and Z from that layer's own rows and Philox stream
  int nseg;
  int seg_off[ZOACT_MAX_GROUP + 1];
  const float* seg_C[ZOACT_MAX_GROUP];
  uint32_t seg_lid[ZOACT_MAX_GROUP];
};

// v = hi + lo (+ what bf16 cannot hold): hi = bf16(v), lo = bf16(v - hi); v - hi is exact in fp32.
__device__ __forceinline__ void split16(float v, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(v);
  lo = __float2bfloat16_rn(v - __bfloat162float(hi));
}

__device__ __forceinline__ uint32_t pack_bf16x2(__nv_bfloat16 a, __nv_bfloat16 b) {
  return (uint32_t)__bfloat16_as_ushort(a) | ((uint32_t)__bfloat16_as_ushort(b) << 16);
}

// The split parts of four consecutive ranks j0..j0+3 of one source row: hi
// (want_lo false) or lo, packed as bf16 pairs.
__device__ __forceinline__ uint2 split_quad(float4 v, bool want_lo) {
  __nv_bfloat16 h[4], l[4];
  split16(v.x, h[0], l[0]);
  split16(v.y, h[1], l[1]);
  split16(v.z, h[2], l[2]);
  split16(v.w, h[3], l[3]);
  const __nv_bfloat16* o = want_lo ? l : h;
  return make_uint2(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]));
}

// One thread per 16-byte chunk (8 K columns) of an output row: rows [0, nA)
// of A_aug, then the nB rows of B_aug (block b, column n), then those of
// B_aug2.  Each column k of a row maps to (slot, half, part, rank j); the chunk
// is built from the source values it needs (P or P2 for A rows, T = C + c_b Z_b
// for B rows; source rows are re-read from L1/L2 by the row's chunks).  With
// QUAD (r a multiple of 4 and 16-byte aligned sources) every 4 columns are one
// part of one slot: one float4 load and one Philox call per 4 columns.
template <bool QUAD>
__global__ void __launch_bounds__(256)
aug_prep_kernel(const float* __restrict__ P, const float* __restrict__ P2, const float* __restrict__ C,
                const float* __restrict__ C2, __nv_bfloat16* __restrict__ A, __nv_bfloat16* __restrict__ B,
                __nv_bfloat16* __restrict__ B2, int64_t rows, int d_out, int r, int ka, int distinct, int full,
                int nb, const __grid_constant__ AugBlocks blk, uint64_t seed, uint32_t lid, uint32_t lid2,
                float* __restrict__ Zt, float* __restrict__ Zt2, int slots, int64_t T) {
  pdl_wait();                                         // P and C written by the previous kernels
  pdl_trigger();
  const int ka_row = distinct ? 2 * ka : ka;          // columns of one slot (= B_aug row width)
  const int cA = slots * ka_row / 8, cB = ka_row / 8; // 16-byte chunks per A / B row
  const int nbB = full ? nb : 1;
  const int64_t nB = (int64_t)nbB * d_out;
  const int64_t itA = rows * cA;
  const int64_t items = itA + (B2 ? 2 : 1) * nB * cB;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t it = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; it < items; it += stride) {
    const bool is_a = it < itA;
    bool up = false;
    int64_t orow;
    int c;
    if (is_a) {
      orow = it / cA;
      c = (int)(it - orow * cA);
    } else {
      const int64_t ib = it - itA;
      const int64_t rb = ib / cB;
      c = (int)(ib - rb * cB);
      up = rb >= nB;
      orow = up ? rb - nB : rb;                      // b * d_out + n
    }
    int my_slot = 0, n = 0;
    float cb = 0.f;
    uint64_t q = 0;
    uint32_t layer = up ? lid2 : lid;
    const float* Cs = up ? C2 : C;      // the coefficients row n indexes (a grouped layer's own)
    if (is_a) {
      if (slots > 1) my_slot = (int)((orow / T) % slots);
    } else {
      const int b = (int)(orow / d_out);
      n = (int)(orow - (int64_t)b * d_out);
      if (full) { cb = blk.coef[b]; q = blk.qry[b]; }
      if (blk.nseg > 1) {
        int sg = 0;
        while (sg + 1 < blk.nseg && n >= blk.seg_off[sg + 1]) ++sg;
        n -= blk.seg_off[sg];
        Cs = blk.seg_C[sg];
        layer = blk.seg_lid[sg];
      }
    }
    uint32_t w[4];
#pragma unroll
    for (int h4 = 0; h4 < 2; ++h4) {
      if (QUAD) {
        const int k0 = 8 * c + 4 * h4;
        const int slot = k0 / ka_row;
        const int kk = k0 - slot * ka_row;
        const int half = kk >= ka ? 1 : 0, kq = kk - half * ka;
        const int part = kq / r, j0 = kq - part * r;
        // A: [hi | hi | lo], B: [hi | lo | hi]; distinct gated A: [gate parts | up parts];
        // distinct gated B: gate rows fill the first half, up rows the second
        const bool live = part < 3 && slot == my_slot && (is_a || !distinct || half == (up ? 1 : 0));
        uint2 o = make_uint2(0u, 0u);
        if (live) {
          float4 v;
          if (is_a) {
            v = *reinterpret_cast<const float4*>((distinct && half ? P2 : P) + orow * r + j0);
          } else {
            const int64_t e = (int64_t)n * r + j0;
            v = *reinterpret_cast<const float4*>(Cs + e);
            if (cb != 0.f) {
              const float4 z = z_normals4(seed, layer, q, (uint64_t)(e >> 2));
              v.x = fmaf(cb, z.x, v.x); v.y = fmaf(cb, z.y, v.y);
              v.z = fmaf(cb, z.z, v.z); v.w = fmaf(cb, z.w, v.w);
            }
          }
          o = split_quad(v, is_a ? part == 2 : part == 1);
        }
        w[2 * h4] = o.x;
        w[2 * h4 + 1] = o.y;
      } else {
        __nv_bfloat16 e4[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int k = 8 * c + 4 * h4 + i;
          const int slot = k / ka_row;
          const int kk = k - slot * ka_row;
          const int half = kk >= ka ? 1 : 0, kq = kk - half * ka;
          const int part = kq / r, j = kq - part * r;
          const bool live = part < 3 && slot == my_slot && (is_a || !distinct || half == (up ? 1 : 0));
          __nv_bfloat16 hi = __float2bfloat16_rn(0.f), lo = hi;
          if (live) {
            float v;
            if (is_a) {
              v = (distinct && half ? P2 : P)[orow * r + j];
            } else {
              const int64_t e = (int64_t)n * r + j;
              v = Cs[e];
              if (cb != 0.f) v = fmaf(cb, z_select(z_normals4(seed, layer, q, (uint64_t)(e >> 2)), (int)(e & 3)), v);
            }
            split16(v, hi, lo);
          }
          e4[i] = live ? ((is_a ? part == 2 : part == 1) ? lo : hi) : __float2bfloat16_rn(0.f);
        }
        w[2 * h4] = pack_bf16x2(e4[0], e4[1]);
        w[2 * h4 + 1] = pack_bf16x2(e4[2], e4[3]);
      }
    }
    __nv_bfloat16* dst = is_a ? A : (up ? B2 : B);
    const int64_t row_w = 8 * (int64_t)(is_a ? cA : cB);
    *reinterpret_cast<uint4*>(dst + orow * row_w + 8 * c) = make_uint4(w[0], w[1], w[2], w[3]);
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

bool aligned16_or_null(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace

int launch_aug_prep(Ctx* ctx, const PairArgs& a, int mode, int ka, int distinct, int slots, void* A_aug,
                    void* B_aug, void* B_aug2, float* Zt, float* Zt2, const uint64_t* zq, int nzq) {
  AugBlocks blk{};
  for (int b = 0; b < a.nb; ++b) { blk.coef[b] = a.coef[b]; blk.qry[b] = a.qry[b]; }
  blk.nseg = a.nseg > 1 ? a.nseg : 0;
  for (int g = 0; g < blk.nseg; ++g) {
    blk.seg_off[g] = a.seg_off[g];
    blk.seg_C[g] = a.seg_C[g];
    blk.seg_lid[g] = a.seg_lid[g];
  }
  blk.seg_off[blk.nseg] = a.d_out;
  // the operand rows of a grouped launch come from the layers' own coefficients (Z tables: one layer only)
  if (blk.nseg > 1 && (Zt || B_aug2)) return ZOACT_ERR_UNSUPPORTED;
  for (int i = 0; i < nzq; ++i) blk.zq[i] = zq[i];
  blk.nzq = Zt ? nzq : 0;
  const int full = mode == LOWRANK_ALL_ON_TC;
  const int ka_row = distinct ? 2 * ka : ka;
  const int64_t nbB = full ? a.nb : 1;
  const int64_t items = a.rows * (slots * ka_row / 8) + (B_aug2 ? 2 : 1) * nbB * a.d_out * (ka_row / 8);
  const int64_t z_items = Zt ? (int64_t)(Zt2 ? 2 : 1) * blk.nzq * ((a.r + 3) / 4) * a.d_out : 0;
  const int64_t work = items > z_items ? items : z_items;
  int64_t grid = (work + 255) / 256;
  const int64_t cap = (int64_t)ctx->sm_count * 32;
  if (grid > cap) grid = cap;
  if (grid < 1) grid = 1;
  // float4 source loads need 16-byte aligned rows: r a multiple of 4 and aligned bases (null: unused)
  bool quad = a.r % 4 == 0 && aligned16_or_null(a.P) && aligned16_or_null(distinct ? a.P2 : nullptr) &&
              aligned16_or_null(a.C) && aligned16_or_null(a.C2);
  for (int g = 0; g < blk.nseg; ++g) quad = quad && aligned16_or_null(a.seg_C[g]);
  auto kern = quad ? aug_prep_kernel<true> : aug_prep_kernel<false>;
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3((unsigned)grid), dim3(256), 0, a.P, distinct ? a.P2 : nullptr, a.C,
                            a.C2, static_cast<__nv_bfloat16*>(A_aug), static_cast<__nv_bfloat16*>(B_aug),
                            static_cast<__nv_bfloat16*>(B_aug2), a.rows, a.d_out, a.r, ka, distinct, full, a.nb, blk,
                            a.seed, a.layer_id, a.layer_id2, Zt, Zt2, slots, a.T));
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
