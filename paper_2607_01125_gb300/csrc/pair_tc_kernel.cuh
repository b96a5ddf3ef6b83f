// Pair forward on the 5th-generation tensor cores (Section 3, the perturbed
// forward pass; Algorithm 2 evaluates it at +eps and -eps):
//
//   Y[t, n] = act( sum_k X[t, k] W[n, k] + sum_j (C[n, j] + c_b Z_b[n, j]) P[t, j] )
//
// with P = X U (computed before) and Z_b regenerated from Philox inside the
// epilogue.  The evaluation points b (the two signs +eps / -eps of the pair,
// or Algorithm 2's unperturbed pass and its q forward-perturbed passes) are
// stacked along the token axis in blocks of T rows, so every W tile is fetched
// once for all of them; when all blocks share the input (the first layer, or
// gate/up of an MLP) the product is computed once and each accumulator row is
// written once per block.
//
// Structure (one persistent CTA per SM, 320 threads):
//   warp 0      TMA producer: X and W tiles (128x64 and 256x64, bf16/fp16,
//               128-byte swizzle) into a 4-stage shared-memory ring;
//   warp 1      MMA issuer: tcgen05.mma 128x256x16 into a TMEM accumulator,
//               two accumulators (512 TMEM columns) so the epilogue of one
//               tile overlaps the main loop of the next;
//   warps 2-9   epilogue, two warpgroups: warp w reads TMEM lanes
//               32*(w%4) .. +31 (its rows) and warpgroup h the h-th half of
//               the tile's columns.  Per tile and block they build the table
//               C + c_b Z_b of the tile's columns in shared memory (Z from
//               Philox; two blocks per pass), tcgen05.ld the accumulator 16
//               columns at a time, add the low-rank term with packed fp32x2
//               FMAs (column pairs), apply the activation and store from
//               registers.
// Gated mode (SiLU MLP gate/up): the 256-row W tile is 128 rows of W_gate and
// the same 128 rows of W_up; the epilogue writes silu(gate) * up for 128 columns.
// Plain mode (no P): the accumulator is stored as fp32 (used for X^T X).
//
// Low-rank term on the tensor cores (Params::aug_mode, operands from
// k_aug.cu): after a tile's d_in / 64 K-blocks the producer loads aug_kb more,
// from A_aug (16-bit split of P) and B_aug (16-bit split of C, or of C + c_b Z_b
// for the tile's block), and the MMA adds them as bf16 products.  With the whole
// term there (stacked rows whose tiles lie in one block) the epilogue only
// converts and stores; with C p there the epilogue adds c_b Z_b p from Z tables,
// once for both signs of a shared-input pair (y+- = acc +- eps Z p).
//
// INT4 weights (W4): the frozen W is symmetric INT4 in groups of 128 along d_in
// with fp16 scales.  Four more warps (448 threads in all) dequantise it: per
// K-block each thread loads 2 rows x 32 packed bytes and their scales with
// plain global loads (prefetched one K-block ahead), turns every nibble q into
// bf16 q * s (magic-number conversion 0x4300 | (q ^ 8) = 128 + q + 8, minus
// 136, times the scale, in bf16x2 arithmetic) and writes the 128-byte-swizzled
// bf16 tile straight into the MMA's shared-memory stage, then fences the
// async proxy and arrives on the stage's barrier.  Only X comes by TMA.  With
// 14 warps the registers per thread drop to 128, so the epilogue works on
// 8-column chunks.
#pragma once
#include "internal.h"
#include "philox.cuh"
#include "tc_common.cuh"

namespace zoact {
namespace pairtc {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int BK_AUG = BK;   // K columns per low-rank K-block
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
// Epilogue tables: C + c_b Z_b for the tile's columns, one [RT][slots + 4]
// table per evaluation block of a pass (two blocks per pass; gated mode keeps
// gate and up tables, four in all).  The 4-float row padding spreads the
// table writes over the banks and keeps rows 16-byte aligned.
constexpr int TBL_FLOATS = 8448;
constexpr int TPAD = 4;
__host__ __device__ constexpr int pair_slots(int rt) {
  return (2 * rt * (BN + TPAD) <= TBL_FLOATS) ? BN : (2 * rt * (BN / 2 + TPAD) <= TBL_FLOATS ? BN / 2 : BN / 4);
}
// gated tiles: four tables (gate and up, two blocks) over at most BN / 2 columns
__host__ __device__ constexpr int gated_slots(int rt) {
  return (4 * rt * (BN / 2 + TPAD) <= TBL_FLOATS) ? BN / 2 : (4 * rt * (BN / 4 + TPAD) <= TBL_FLOATS ? BN / 4 : BN / 8);
}
constexpr int EPI_WARPS = 8;
constexpr int EPI_THREADS = 32 * EPI_WARPS;
constexpr int DQ_THREADS = 128;                     // INT4 dequantisation warps
__host__ __device__ constexpr int num_threads(bool w4) { return 64 + EPI_THREADS + (w4 ? DQ_THREADS : 0); }
__host__ __device__ constexpr int epi_base(bool w4) { return 64 + (w4 ? DQ_THREADS : 0); }
constexpr int TMEM_COLS = 512;
constexpr int SMEM_BYTES = 1024 /*align slack*/ + STAGES * STAGE_BYTES + TBL_FLOATS * 4 + 256;
constexpr int GROUP_M = 8;
static_assert(SMEM_BYTES <= 232448, "dynamic shared memory above the 227 KB a CTA may use");

enum Mode { MODE_PAIR = 0, MODE_GATED = 1, MODE_PLAIN = 2 };

// Tensor maps of one launch: X, W (gate), W up, and the low-rank K columns
// A_aug, B_aug, B_aug up (unused ones are copies of a valid map).
// Output staging of a CTA-pair launch (Params::y_staged, the kernel's SMODE): none, the whole
// low-rank term on the MMA, the two signs of one query on a shared input (row per thread, or
// four rows per thread when the rank tile is <= 16 and a gated pair shares one projection), or
// other evaluation blocks on a shared input (four rows per thread, same conditions), or no output at
// all: the loss pair of the rounded outputs, fused (zoact_pair_forward_loss).
enum StageMode { STAGE_NONE = 0, STAGE_ALL = 1, STAGE_MIRROR = 2, STAGE_MIRROR4 = 3, STAGE_MULTI4 = 4,
                 STAGE_LOSS = 5 };

struct TmaSet {
  CUtensorMap a, b, b2, aa, ba, ba2;
  CUtensorMap y, y16;   // output Y for staged bulk stores: 128-byte swizzled rows, and 16-column boxes
  // INT4 on CTA pairs: b / b2 map the packed weights ([d_out, d_in/2] bytes, 32 x 128 boxes), s / s2 their
  // fp16 scales ([d_out, d_in/128], 8 x 128 boxes)
  CUtensorMap s, s2;
};

struct Params {
  const float* P;
  const float* C;
  const float* P2;   // gated: up
  const float* C2;
  void* Y;
  int64_t rows;      // rows of X
  int64_t T;
  int d_in, d_out, r;
  int shared;
  int act;
  int nb;                                   // evaluation blocks (rows [b T, (b+1) T) of Y)
  float coef[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t qry[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t seed;
  uint32_t layer_id, layer_id2;
  int num_m, num_n, num_k, num_tiles;
  int aug_mode;      // LowrankMode
  int y_staged;      // StageMode: tm.y / tm.y16 hold Y's store maps for the CTA-pair kernel's staged epilogue
  int aug_kb;        // extra K-blocks per tile from A_aug / B_aug (0 with LOWRANK_EPILOGUE)
  int aug_kb_slot;   // K-blocks of one slot (B_aug row width / 64)
  int aug_slots;     // LOWRANK_ALL_ON_TC: 1, or S when a tile spans up to S evaluation blocks (slot = block mod S)
  int64_t aug_block_rows;   // rows of one block's table in B_aug (LOWRANK_ALL_ON_TC)
  // LOWRANK_C_ON_TC: Z of each distinct query, transposed [q][r][d_out] (gate / up), and the table of each block
  const float* Zt;
  const float* Zt2;
  int64_t zt_qstride;       // floats per query table (r * d_out)
  int zq[ZOACT_MAX_EVAL_BLOCKS];   // block b's table in Zt (-1: coefficient 0)
  int64_t ldy;       // plain mode: row stride of D
  int vec_ok;        // C, C2, P, P2 and ldy allow 16-byte vector access
  int bn;            // N-tile width of pair / plain tiles (multiple of 32, <= BN); gated tiles use BN
  // INT4 weights: packed [d_out, d_in/2] bytes and fp16 scales [d_out, d_in/128]
  const uint8_t* Wq;
  const __half* Ws;
  const uint8_t* Wq2;
  const __half* Ws2;
  int* status;
  // fused loss pair (STAGE_LOSS): target [T, d_out] of Y's type through tm.y / tm.y16 (or none: mean of
  // squares), per-CTA partial sums, the ticket of the last CTA, and out[4] = {L+, L-, D, a}
  int has_target;
  float loss_eps;
  double* loss_part;
  unsigned int* loss_ticket;
  double* loss_out;
  // split tail (CTA-pair kernel): tiles [sk_first, sk_first + sk_tiles) are each cut into sk_split equal
  // K ranges, one per pair (sk_tiles = 0: every tile whole); sk_part holds one 128 x BN fp32 partial
  // accumulator per pair and CTA, sk_ticket one counter per tail tile and CTA (zero between launches)
  // row scales (CTA-pair staged epilogue of stacked rows only): in_scale [rows] multiplies every accumulator row
  // before the activation (an RMS-normalised input given unnormalised); out_sumsq [ceil(d_out / 64), rows]
  // receives, per 64-column part, the row's sum of squares of the stored (rounded) outputs
  const float* in_scale;
  float* out_sumsq;
  int group_m;       // M-tiles per group of the tile order (0: GROUP_M)
  int sk_first, sk_tiles, sk_split;
  float* sk_part;
  unsigned int* sk_ticket;
};

struct SharedState {
  uint64_t full[STAGES];
  uint64_t empty[STAGES];
  uint64_t tmem_full[2];
  uint64_t tmem_empty[2];
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
  int epi_ok;
};
static_assert(sizeof(SharedState) <= 256, "barrier block outgrew its shared-memory slot");

// TMA coordinates of low-rank K-block `ka` (0 .. aug_kb) of a tile whose rows start at tile_row0:
// x in A_aug (slots side by side), x in B_aug (one slot wide), and the first B_aug row of the table the
// slot meets -- the tile's block (one slot), or the tile's block congruent to the slot mod S (S slots;
// a slot no block of the tile maps to has zero A columns and reads any table).
__device__ __forceinline__ void aug_coords(const Params& prm, int64_t tile_row0, int tile_rows, int ka, int& kx_a,
                                           int& kx_b, int& y_b) {
  const int slot = ka / prm.aug_kb_slot;
  kx_a = ka * BK_AUG;
  kx_b = (ka - slot * prm.aug_kb_slot) * BK_AUG;
  y_b = 0;
  if (prm.aug_mode == LOWRANK_ALL_ON_TC) {
    const int b_lo = (int)(tile_row0 / prm.T);
    const int b_hi = (int)((min(tile_row0 + tile_rows, prm.rows) - 1) / prm.T);
    const int S = prm.aug_slots;
    int blk = b_lo + ((slot - b_lo % S) % S + S) % S;
    if (blk > b_hi) blk = b_lo;
    y_b = (int)(blk * prm.aug_block_rows);
  }
}

// Grouped tile order: groups of group_m M-tiles (0: GROUP_M), every N-tile of a group before the next group,
// the M-tiles of one N-tile consecutive -- a wave reads each W panel once per group while the group's X rows
// stay in L2.
__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int& m_blk, int& n_blk, int group_m = 0) {
  const int G = group_m > 0 ? group_m : GROUP_M;
  const int per_group = G * num_n;
  const int group = tile / per_group;
  const int first_m = group * G;
  const int gm = min(G, num_m - first_m);
  const int in_group = tile - group * per_group;
  m_blk = first_m + in_group % gm;
  n_blk = in_group / gm;
}

// Fill the tables of one layer for output columns [col0, col0 + ncols) at two
// evaluation points (tb1 may be null):
//   tb0[j * stride + s] = C[col0 + s][j] + c0 Z(q0)[col0 + s][j]   (tb1: c1, q1)
// (without the C term when Cg is null), zero where col0 + s >= d_out or j >= r.
// A point with coefficient 0 draws no Z; when both points use the same query
// (the two signs of the pair) Z is drawn once.
template <int RT>
__device__ __forceinline__ void build_tables(float* tb0, float* tb1, int stride, const float* __restrict__ Cg,
                                             uint32_t layer_id, int col0, int ncols, int d_out, int r,
                                             uint64_t seed, float c0, uint64_t q0, float c1, uint64_t q1, int tid,
                                             bool vec_ok) {
  const int valid_cols = max(0, min(ncols, d_out - col0));
  const bool z0_on = c0 != 0.f, z1_on = tb1 != nullptr && c1 != 0.f;
  const bool z1_same = z1_on && z0_on && q1 == q0;
  if (r == RT && vec_ok) {
    // one thread per 4 consecutive ranks of one column: one float4 of C, one Philox group
    constexpr int GPC = RT / 4;                          // groups per column
    const int n_groups = ncols * GPC;
    for (int g = tid; g < n_groups; g += EPI_THREADS) {
      const int s = g / GPC, jg = g % GPC;
      float4 c = make_float4(0.f, 0.f, 0.f, 0.f), z0 = c, z1 = c;
      if (s < valid_cols) {
        const int64_t e = (int64_t)(col0 + s) * RT + 4 * jg;
        if (Cg) c = *reinterpret_cast<const float4*>(Cg + e);
        if (z0_on) z0 = z_normals4(seed, layer_id, q0, (uint64_t)(e >> 2));
        if (z1_on) z1 = z1_same ? z0 : z_normals4(seed, layer_id, q1, (uint64_t)(e >> 2));
      }
      float* d0 = tb0 + (4 * jg) * stride + s;
      d0[0] = fmaf(c0, z0.x, c.x);
      d0[stride] = fmaf(c0, z0.y, c.y);
      d0[2 * stride] = fmaf(c0, z0.z, c.z);
      d0[3 * stride] = fmaf(c0, z0.w, c.w);
      if (tb1) {
        float* d1 = tb1 + (4 * jg) * stride + s;
        d1[0] = fmaf(c1, z1.x, c.x);
        d1[stride] = fmaf(c1, z1.y, c.y);
        d1[2 * stride] = fmaf(c1, z1.z, c.z);
        d1[3 * stride] = fmaf(c1, z1.w, c.w);
      }
    }
    return;
  }
  // general ranks / unaligned C: one element per iteration
  for (int i = tid; i < ncols * RT; i += EPI_THREADS) {
    const int s = i / RT, j = i % RT;
    float v0 = 0.f, v1 = 0.f;
    if (s < valid_cols && j < r) {
      const int64_t e = (int64_t)(col0 + s) * r + j;
      const float c = Cg ? Cg[e] : 0.f;
      const uint64_t grp = (uint64_t)(e >> 2);
      const int w = (int)(e & 3);
      const float z0 = z0_on ? z_select(z_normals4(seed, layer_id, q0, grp), w) : 0.f;
      const float z1 = z1_on ? (z1_same ? z0 : z_select(z_normals4(seed, layer_id, q1, grp), w)) : 0.f;
      v0 = fmaf(c0, z0, c);
      v1 = fmaf(c1, z1, c);
    }
    tb0[j * stride + s] = v0;
    if (tb1) tb1[j * stride + s] = v1;
  }
}

// The same tables from precomputed transposed Z (Zq0 / Zq1: a query's [r][d_out]
// table, Zq1 may equal Zq0): tb[j * stride + s] = c Z[j][col0 + s].  One thread
// per 4 consecutive columns of one rank: coalesced 16-byte loads (d_out % 8 == 0).
template <int RT>
__device__ __forceinline__ void build_tables_z(float* tb0, float* tb1, int stride, const float* __restrict__ Zq0,
                                               const float* __restrict__ Zq1, float c0, float c1, int col0,
                                               int ncols, int d_out, int r, int tid) {
  const int per_row = ncols / 4;
  for (int it = tid; it < RT * per_row; it += EPI_THREADS) {
    const int j = it / per_row, s = 4 * (it - j * per_row);
    const int col = col0 + s;
    float4 v0 = make_float4(0.f, 0.f, 0.f, 0.f), v1 = v0;
    if (j < r && col < d_out) {
      const float4 z0 = *reinterpret_cast<const float4*>(Zq0 + (int64_t)j * d_out + col);
      v0 = make_float4(c0 * z0.x, c0 * z0.y, c0 * z0.z, c0 * z0.w);
      if (tb1) {
        const float4 z1 = Zq1 == Zq0 ? z0 : *reinterpret_cast<const float4*>(Zq1 + (int64_t)j * d_out + col);
        v1 = make_float4(c1 * z1.x, c1 * z1.y, c1 * z1.z, c1 * z1.w);
      }
    }
    *reinterpret_cast<float4*>(tb0 + j * stride + s) = v0;
    if (tb1) *reinterpret_cast<float4*>(tb1 + j * stride + s) = v1;
  }
}

// d = a * b + c on two fp32 lanes at once (one packed FMA; each lane rounds
// like fmaf).
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
      "mov.b64 ra, {%2, %3};\n\t"
      "mov.b64 rb, {%4, %5};\n\t"
      "mov.b64 rc, {%6, %7};\n\t"
      "fma.rn.f32x2 rd, ra, rb, rc;\n\t"
      "mov.b64 {%0, %1}, rd;\n\t}"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}

// Low-rank sums of CW consecutive table columns for one token row:
//   s[i] = sum_j tb[j * stride + c + i] p[j]     (j ascending).
template <int RT, int CW>
__device__ __forceinline__ void lowrank_t(const float* tb, int stride, int c, const float* p, float* s) {
  float2 acc[CW / 2];
#pragma unroll
  for (int i = 0; i < CW / 2; ++i) acc[i] = make_float2(0.f, 0.f);
  asm volatile("" ::: "memory");     // keep the table loads of one call together (register pressure)
#pragma unroll
  for (int j = 0; j < RT; ++j) {
    const float4* t4 = reinterpret_cast<const float4*>(tb + j * stride + c);
    const float2 pj = make_float2(p[j], p[j]);
#pragma unroll
    for (int q = 0; q < CW / 4; ++q) {
      const float4 v = t4[q];
      acc[2 * q] = ffma2(make_float2(v.x, v.y), pj, acc[2 * q]);
      acc[2 * q + 1] = ffma2(make_float2(v.z, v.w), pj, acc[2 * q + 1]);
    }
  }
#pragma unroll
  for (int i = 0; i < CW / 2; ++i) { s[2 * i] = acc[i].x; s[2 * i + 1] = acc[i].y; }
}

__device__ __forceinline__ float silu_fast(float x) { return __fdividef(x, 1.0f + __expf(-x)); }

__device__ __forceinline__ uint32_t pack2(float a, float b, __nv_bfloat16*) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ uint32_t pack2(float a, float b, __half*) {
  __half2 h = __floats2half2_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Store CW (8 or 16) consecutive outputs from registers (16-byte vectors when
// all are valid and the destination is 16-byte aligned).
template <typename TO, int CW>
__device__ __forceinline__ void storeN(TO* dst, const float* v, int n_valid, bool vec_ok = true) {
  if (n_valid >= CW && vec_ok) {
    if constexpr (sizeof(TO) == 4) {
      float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
      for (int i = 0; i < CW / 4; ++i) d4[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    } else {
      uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
      for (int i = 0; i < CW / 8; ++i)
        d4[i] = make_uint4(pack2(v[8 * i], v[8 * i + 1], (TO*)nullptr), pack2(v[8 * i + 2], v[8 * i + 3], (TO*)nullptr),
                           pack2(v[8 * i + 4], v[8 * i + 5], (TO*)nullptr),
                           pack2(v[8 * i + 6], v[8 * i + 7], (TO*)nullptr));
    }
  } else {
#pragma unroll
    for (int i = 0; i < CW; ++i)
      if (i < n_valid) dst[i] = from_f32<TO>(v[i]);
  }
}

template <int CW>
__device__ __forceinline__ void tmem_ldN(uint32_t taddr, float* v) {
  if constexpr (CW == 16) tc::tmem_ld16(taddr, v);
  else tc::tmem_ld8(taddr, v);
}

// ---- INT4 dequantisation into a 128-byte-swizzled bf16 B tile ----
// 8 nibbles (elements k..k+7, low nibble first) scaled by s -> 8 bf16 (16 bytes).
__device__ __forceinline__ uint4 dequant8(uint32_t w, __nv_bfloat162 s2) {
  const uint32_t x = w ^ 0x88888888u;                 // nibble q -> q + 8 in [0, 15]
  const __nv_bfloat162 c136 = __floats2bfloat162_rn(136.0f, 136.0f);
  uint32_t out[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const uint32_t lo = (x >> (8 * i)) & 0xFu, hi = (x >> (8 * i + 4)) & 0xFu;
    uint32_t v = 0x43004300u | lo | (hi << 16);       // bf16 pair (128 + q + 8)
    __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&v);
    h = __hmul2(__hsub2(h, c136), s2);                // q exactly, then q * s rounded to bf16
    out[i] = *reinterpret_cast<uint32_t*>(&h);
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

// Row `row` (0..255) of the B tile of K-block kb: source row, packed bytes and scale.
struct DqRow {
  uint4 q0, q1;       // 32 packed bytes = 64 elements
  __half s;
  bool valid;
};

template <int MODE>
__device__ __forceinline__ DqRow dq_load(const Params& prm, int n_blk, int row, int kb) {
  DqRow d;
  const uint8_t* Wq = prm.Wq;
  const __half* Ws = prm.Ws;
  int n;
  if (MODE == MODE_GATED) {
    n = n_blk * (BN / 2) + (row & (BN / 2 - 1));
    if (row >= BN / 2) { Wq = prm.Wq2; Ws = prm.Ws2; }
  } else {
    n = n_blk * BN + row;
  }
  d.valid = n < prm.d_out;
  if (d.valid) {
    const uint4* src = reinterpret_cast<const uint4*>(Wq + (int64_t)n * (prm.d_in / 2) + kb * (BK / 2));
    d.q0 = __ldg(src);
    d.q1 = __ldg(src + 1);
    d.s = Ws[(int64_t)n * (prm.d_in / 128) + (kb * BK) / 128];
  } else {
    d.q0 = d.q1 = make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);   // q = 0
    d.s = __float2half_rn(0.f);
  }
  return d;
}

__device__ __forceinline__ void dq_store(uint8_t* btile, int row, const DqRow& d) {
  const __nv_bfloat16 sb = __float2bfloat16_rn(__half2float(d.s));
  const __nv_bfloat162 s2 = __halves2bfloat162(sb, sb);
  uint8_t* rowp = btile + row * 128;
  const uint32_t w[8] = {d.q0.x, d.q0.y, d.q0.z, d.q0.w, d.q1.x, d.q1.y, d.q1.z, d.q1.w};
#pragma unroll
  for (int c = 0; c < 8; ++c)
    *reinterpret_cast<uint4*>(rowp + ((c ^ (row & 7)) << 4)) = dequant8(w[c], s2);
}

// The epilogue's wait for a finished accumulator, taken by one thread and
// shared through a named barrier so that all epilogue threads leave (or
// continue) together even if the wait gives up.
template <typename SS>
__device__ __forceinline__ bool epi_wait_full(SS* ss, int buf, uint32_t parity, volatile int* abort_flag,
                                              int* status, int etid) {
  if (etid == 0) ss->epi_ok = tc::mbar_wait(tc::smem_u32(&ss->tmem_full[buf]), parity, abort_flag, status) ? 1 : 0;
  tc::named_bar_sync(2, EPI_THREADS);
  tc::tc_fence_after();
  const bool ok = *reinterpret_cast<volatile int*>(&ss->epi_ok) != 0;
  tc::named_bar_sync(2, EPI_THREADS);   // everyone has read epi_ok before thread 0 may rewrite it
  return ok;
}

template <int RT>
__device__ __forceinline__ void load_p(float* p, const float* __restrict__ P, int64_t m, int r, bool row_ok,
                                       bool vec_ok) {
  if (row_ok && r == RT && vec_ok) {
    const float4* src = reinterpret_cast<const float4*>(P + m * r);
#pragma unroll
    for (int q = 0; q < RT / 4; ++q) {
      const float4 v = src[q];
      p[4 * q] = v.x; p[4 * q + 1] = v.y; p[4 * q + 2] = v.z; p[4 * q + 3] = v.w;
    }
  } else {
#pragma unroll
    for (int j = 0; j < RT; ++j) p[j] = (row_ok && j < r) ? P[m * r + j] : 0.f;
  }
}

// Pair / gated epilogue of one accumulator tile for this CTA's 128 rows
// [row0, row0 + 128) (row m of thread (quad, lane)).  Column chunk by column
// chunk, and two evaluation blocks per pass, it builds the tables of the
// low-rank terms the MMA did not add (C + c_b Z_b, or c_b Z_b when C p came
// from the tensor cores), waits for the accumulator (first pass), adds them,
// applies the activation or the SiLU gate and stores.  Stacked rows use the
// block they belong to; shared rows are written once per block, and a pass
// over the two signs of one query (coefficients +c, -c) builds one Z table and
// forms acc +- c Z p.  With the whole term on the tensor cores it only converts
// and stores.  Returns false when the wait gave up.
template <typename TO, int RT, int MODE, int CW, typename SS>
__device__ __forceinline__ bool epi_pair_tile(const Params& prm, SS* ss, float* tbl, int etid, int half,
                                              int64_t row0, int64_t m, bool row_ok, int n_blk, int bn, int buf,
                                              uint32_t acc_phase, uint32_t t_row, volatile int* abort_flag) {
  constexpr bool GATED = MODE == MODE_GATED;
  constexpr int SLOTS = GATED ? gated_slots(RT) : pair_slots(RT);   // table columns per chunk
  constexpr int STRIDE = SLOTS + TPAD;
  constexpr int TSZ = RT * STRIDE;                         // floats per table
  static_assert((GATED ? 4 : 2) * TSZ <= TBL_FLOATS, "epilogue tables exceed their shared-memory region");
  const int r = prm.r;
  const int64_t T = prm.T;
  TO* Y = static_cast<TO*>(prm.Y);
  const int ncol_tile = GATED ? BN / 2 : bn;               // output columns of this tile
  if (prm.aug_mode == LOWRANK_ALL_ON_TC) {
    // stacked rows, the whole low-rank term in the accumulator
    if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
    const int cbeg = half * (ncol_tile / 2);
    for (int c0 = cbeg; c0 < cbeg + ncol_tile / 2; c0 += CW) {
      const int n = n_blk * ncol_tile + c0;
      if (n >= prm.d_out) break;
      const int nv = min(CW, prm.d_out - n);
      if (GATED) {
        float g[CW], u[CW], h[CW];
        tmem_ldN<CW>(t_row + (uint32_t)c0, g);
        tmem_ldN<CW>(t_row + (uint32_t)(BN / 2 + c0), u);
#pragma unroll
        for (int i = 0; i < CW; ++i) h[i] = silu_fast(g[i]) * u[i];
        if (row_ok) storeN<TO, CW>(Y + m * prm.d_out + n, h, nv);
      } else {
        float acc[CW];
        tmem_ldN<CW>(t_row + (uint32_t)c0, acc);
#pragma unroll
        for (int i = 0; i < CW; ++i) acc[i] = apply_act(acc[i], prm.act);
        if (row_ok) storeN<TO, CW>(Y + m * prm.d_out + n, acc, nv);
      }
    }
    return true;
  }
  const bool c_in_acc = prm.aug_mode == LOWRANK_C_ON_TC;
  float p[RT], p2[RT];
  const bool vec = prm.vec_ok != 0;
  load_p<RT>(p, prm.P, m, r, row_ok, vec);
  if (GATED) load_p<RT>(p2, prm.P2, m, r, row_ok, vec);
  // evaluation blocks this CTA's rows touch
  int b_first = 0, b_last = prm.nb - 1;
  if (!prm.shared) {
    const int64_t last_row = min(row0 + BM, prm.rows) - 1;
    b_first = (int)(row0 / T);
    b_last = (int)(last_row / T);
  }
  if (b_last < b_first)    // no valid row in this CTA's part of the tile: only release the accumulator
    return epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid);
  const int my_b = (!prm.shared && row_ok) ? (int)(m / T) : -1;
  const float* Cg = c_in_acc ? nullptr : prm.C;
  const float* Cg2 = c_in_acc ? nullptr : prm.C2;
  bool waited = false;
  for (int s0 = 0; s0 < ncol_tile; s0 += SLOTS) {
    const int cwid = min(SLOTS, ncol_tile - s0);          // a multiple of 32
    const int col0 = n_blk * ncol_tile + s0;
    for (int bp = b_first; bp <= b_last; bp += 2) {
      const bool two = bp + 1 <= b_last;
      const int b1 = two ? bp + 1 : bp;
      // the two signs of one query on a shared input: one table Z, outputs acc +- c Z p
      const bool mirror = c_in_acc && prm.shared && two && prm.qry[b1] == prm.qry[bp] &&
                          prm.coef[b1] == -prm.coef[bp] && prm.coef[bp] != 0.f;
      // a block needs a table unless its term is already in the accumulator (C p there, c_b = 0)
      const bool need0 = !c_in_acc || prm.coef[bp] != 0.f;
      const bool need1 = two && !mirror && (!c_in_acc || prm.coef[b1] != 0.f);
      const float tc0 = mirror ? 1.f : prm.coef[bp];
      tc::named_bar_sync(1, EPI_THREADS);                 // previous pass's readers are done
      if (need0 || need1) {
        // table slot 0 holds block bp (or block b1 alone when bp needs none)
        float* t0 = tbl;
        float* t1 = (need0 && need1) ? tbl + TSZ : nullptr;
        const float c0v = need0 ? tc0 : prm.coef[b1];
        if (c_in_acc) {
          // c_b Z_b from the transposed Z tables
          const int z0 = need0 ? prm.zq[bp] : prm.zq[b1];
          const int z1 = prm.zq[b1] >= 0 ? prm.zq[b1] : z0;
          build_tables_z<RT>(t0, t1, STRIDE, prm.Zt + z0 * prm.zt_qstride, prm.Zt + z1 * prm.zt_qstride, c0v,
                             prm.coef[b1], col0, cwid, prm.d_out, r, etid);
          if (GATED)
            build_tables_z<RT>(t0 + 2 * TSZ, t1 ? t1 + 2 * TSZ : nullptr, STRIDE, prm.Zt2 + z0 * prm.zt_qstride,
                               prm.Zt2 + z1 * prm.zt_qstride, c0v, prm.coef[b1], col0, cwid, prm.d_out, r, etid);
        } else {
          const uint64_t q0v = need0 ? prm.qry[bp] : prm.qry[b1];
          build_tables<RT>(t0, t1, STRIDE, Cg, prm.layer_id, col0, cwid, prm.d_out, r, prm.seed, c0v, q0v,
                           prm.coef[b1], prm.qry[b1], etid, vec);
          if (GATED)
            build_tables<RT>(t0 + 2 * TSZ, t1 ? t1 + 2 * TSZ : nullptr, STRIDE, Cg2, prm.layer_id2, col0, cwid,
                             prm.d_out, r, prm.seed, c0v, q0v, prm.coef[b1], prm.qry[b1], etid, vec);
        }
      }
      tc::named_bar_sync(1, EPI_THREADS);
      if (!waited) {
        if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
        waited = true;
      }
      // table index of block bp + t (-1: no term to add)
      const int tix0 = need0 ? 0 : -1;
      const int tix1 = need1 ? (need0 ? 1 : 0) : -1;
      const int sel = my_b - bp;                          // stacked: my block in this pass
      const bool active = prm.shared ? row_ok : (sel == 0 || (sel == 1 && two));
      if (!prm.shared && !__any_sync(0xffffffffu, active)) continue;   // no row of this warp in the pass
      const int nt = prm.shared ? (two ? 2 : 1) : 1;
      const int cbeg = s0 + half * (cwid / 2);
      for (int c0 = cbeg; c0 < cbeg + cwid / 2; c0 += CW) {
        const int n = n_blk * ncol_tile + c0;
        if (n >= prm.d_out) break;                        // uniform: same columns for the whole warp
        const int nv = min(CW, prm.d_out - n);
        if (GATED) {
          float g[CW], u[CW];
          tmem_ldN<CW>(t_row + (uint32_t)c0, g);
          tmem_ldN<CW>(t_row + (uint32_t)(BN / 2 + c0), u);
          if (active) {
            if (mirror) {
              float sg[CW], su[CW];
              lowrank_t<RT, CW>(tbl, STRIDE, c0 - s0, p, sg);
              lowrank_t<RT, CW>(tbl + 2 * TSZ, STRIDE, c0 - s0, p2, su);
              const float cz = prm.coef[bp];
#pragma unroll
              for (int i = 0; i < CW; ++i) {       // in place: sg <- h(+c), su <- h(-c)
                const float hp = silu_fast(fmaf(cz, sg[i], g[i])) * fmaf(cz, su[i], u[i]);
                const float hm = silu_fast(fmaf(-cz, sg[i], g[i])) * fmaf(-cz, su[i], u[i]);
                sg[i] = hp;
                su[i] = hm;
              }
              storeN<TO, CW>(Y + ((int64_t)bp * T + m) * prm.d_out + n, sg, nv);
              storeN<TO, CW>(Y + ((int64_t)b1 * T + m) * prm.d_out + n, su, nv);
            } else {
#pragma unroll 1
              for (int t = 0; t < nt; ++t) {
                const int tix = (prm.shared ? t : sel) == 0 ? tix0 : tix1;
                float hg[CW], hu[CW];
                if (tix >= 0) {
                  lowrank_t<RT, CW>(tbl + tix * TSZ, STRIDE, c0 - s0, p, hg);
#pragma unroll
                  for (int i = 0; i < CW; ++i) hg[i] += g[i];
                  lowrank_t<RT, CW>(tbl + (2 + tix) * TSZ, STRIDE, c0 - s0, p2, hu);
#pragma unroll
                  for (int i = 0; i < CW; ++i) hu[i] = silu_fast(hg[i]) * (hu[i] + u[i]);
                } else {
#pragma unroll
                  for (int i = 0; i < CW; ++i) hu[i] = silu_fast(g[i]) * u[i];
                }
                const int64_t row = prm.shared ? (int64_t)(bp + t) * T + m : m;
                storeN<TO, CW>(Y + row * prm.d_out + n, hu, nv);
              }
            }
          }
        } else {
          float acc[CW];
          tmem_ldN<CW>(t_row + (uint32_t)c0, acc);
          if (active) {
            if (mirror) {
              float sl[CW], y[CW];
              lowrank_t<RT, CW>(tbl, STRIDE, c0 - s0, p, sl);
              const float cz = prm.coef[bp];
#pragma unroll
              for (int i = 0; i < CW; ++i) y[i] = apply_act(fmaf(cz, sl[i], acc[i]), prm.act);
              storeN<TO, CW>(Y + ((int64_t)bp * T + m) * prm.d_out + n, y, nv);
#pragma unroll
              for (int i = 0; i < CW; ++i) y[i] = apply_act(fmaf(-cz, sl[i], acc[i]), prm.act);
              storeN<TO, CW>(Y + ((int64_t)b1 * T + m) * prm.d_out + n, y, nv);
            } else {
#pragma unroll 1
              for (int t = 0; t < nt; ++t) {
                const int tix = (prm.shared ? t : sel) == 0 ? tix0 : tix1;
                float sl[CW], y[CW];
                if (tix >= 0) {
                  lowrank_t<RT, CW>(tbl + tix * TSZ, STRIDE, c0 - s0, p, sl);
                } else {
#pragma unroll
                  for (int i = 0; i < CW; ++i) sl[i] = 0.f;
                }
#pragma unroll
                for (int i = 0; i < CW; ++i) y[i] = apply_act(acc[i] + sl[i], prm.act);
                const int64_t row = prm.shared ? (int64_t)(bp + t) * T + m : m;
                storeN<TO, CW>(Y + row * prm.d_out + n, y, nv);
              }
            }
          }
        }
      }
    }
  }
  return true;
}

template <typename TO, int RT, int MODE, int AB_BF16, bool W4>
__global__ void __launch_bounds__(num_threads(W4), 1)
pair_tc_kernel(const __grid_constant__ TmaSet tm, const Params prm) {
  // epilogue chunk width (columns per tcgen05.ld): 8 where the registers are scarce (INT4's 14 warps,
  // the gated pair's two accumulators and two projections)
  constexpr int CW = (W4 || MODE == MODE_GATED) ? 8 : 16;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  float* tbl = reinterpret_cast<float*>(smem + STAGES * STAGE_BYTES);
  SharedState* ss = reinterpret_cast<SharedState*>(tbl + TBL_FLOATS);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  volatile int* abort_flag = &ss->abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      // full: the producer's expect_tx arrival, plus one arrival per dequantising thread (INT4)
      tc::mbar_init(tc::smem_u32(&ss->full[s]), W4 ? 1 + DQ_THREADS : 1);
      tc::mbar_init(tc::smem_u32(&ss->empty[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(tc::smem_u32(&ss->tmem_full[b]), 1);
      tc::mbar_init(tc::smem_u32(&ss->tmem_empty[b]), EPI_THREADS);
    }
    tc::mbar_init(tc::smem_u32(&ss->drain), 1);
    ss->abort_flag = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm.a);
    if (!W4) tc::prefetch_tmap(&tm.b);
    if (!W4 && MODE == MODE_GATED) tc::prefetch_tmap(&tm.b2);
    if (prm.aug_kb > 0) {
      tc::prefetch_tmap(&tm.aa);
      tc::prefetch_tmap(&tm.ba);
      if (MODE == MODE_GATED) tc::prefetch_tmap(&tm.ba2);
    }
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(&ss->tmem_base), TMEM_COLS);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem_base = ss->tmem_base;
  pdl_wait();                             // the previous kernel's outputs (X, P, operand tables) are visible
  pdl_trigger();

  const int num_m = prm.num_m, num_n = prm.num_n, num_k = prm.num_k;
  const int total_k = num_k + (W4 ? 0 : prm.aug_kb);   // main K-blocks, then the low-rank ones
  const int bn = MODE == MODE_GATED ? BN : prm.bn;  // this launch's N-tile width

  if (warp == 0) {
    // ---------------- TMA producer ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      uint32_t issued_mask = 0, issued_parity = 0;   // per stage: a load in flight, and its full-phase parity
      bool ok = true;
      for (int tile = blockIdx.x; tile < prm.num_tiles && ok; tile += gridDim.x) {
        int m_blk, n_blk;
        tile_coords(tile, num_m, num_n, m_blk, n_blk);
        for (int kb = 0; kb < total_k; ++kb) {
          if (!tc::mbar_wait(tc::smem_u32(&ss->empty[stage]), phase ^ 1u, abort_flag, prm.status)) { ok = false; break; }
          const uint32_t full = tc::smem_u32(&ss->full[stage]);
          tc::mbar_arrive_expect_tx(full, W4 ? A_BYTES : (MODE == MODE_GATED ? STAGE_BYTES : A_BYTES + bn * BK * 2));
          const uint32_t sa = tc::smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_BYTES;
          const bool aug = kb >= num_k;
          int kx = kb * BK, kxb = kb * BK, yb = 0;
          if (aug) aug_coords(prm, (int64_t)m_blk * BM, BM, kb - num_k, kx, kxb, yb);
          tc::tma_load_2d(sa, aug ? &tm.aa : &tm.a, kx, m_blk * BM, full);
          if (W4) {
            // B arrives from the dequantising warps
          } else if (MODE == MODE_GATED) {
            tc::tma_load_2d(sb, aug ? &tm.ba : &tm.b, kxb, yb + n_blk * (BN / 2), full);
            tc::tma_load_2d(sb + B_BYTES / 2, aug ? &tm.ba2 : &tm.b2, kxb, yb + n_blk * (BN / 2), full);
          } else {
            tc::tma_load_2d(sb, aug ? &tm.ba : &tm.b, kxb, yb + n_blk * bn, full);
          }
          issued_mask |= 1u << stage;
          issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        // wind down: wait (bounded) for our own copies still in flight
        for (int s = 0; s < STAGES; ++s)
          if (issued_mask & (1u << s))
            tc::mbar_wait_drain(tc::smem_u32(&ss->full[s]), (issued_parity >> s) & 1u, 100000000ull);
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer ----------------
    if (lane == 0) {
      const uint32_t IDESC = tc::idesc_f16(BM, bn, AB_BF16);
      const uint32_t IDESC_AUG = tc::idesc_f16(BM, bn, 1);   // low-rank K-blocks are bf16
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int local = 0;
      bool issued_any = false;
      for (int tile = blockIdx.x; tile < prm.num_tiles && ok; tile += gridDim.x, ++local) {
        const int buf = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!tc::mbar_wait(tc::smem_u32(&ss->tmem_empty[buf]), acc_phase ^ 1u, abort_flag, prm.status)) { ok = false; break; }
        tc::tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
        for (int kb = 0; kb < total_k; ++kb) {
          if (!tc::mbar_wait(tc::smem_u32(&ss->full[stage]), phase, abort_flag, prm.status)) { ok = false; break; }
          tc::tc_fence_after();
          const uint32_t sa = tc::smem_u32(smem + stage * STAGE_BYTES);
          const uint32_t sb = sa + A_BYTES;
          const uint32_t idesc = kb < num_k ? IDESC : IDESC_AUG;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k) {
            const uint64_t ad = tc::sdesc_k_sw128(sa + k * 32);
            const uint64_t bd = tc::sdesc_k_sw128(sb + k * 32);
            tc::mma_f16(d_tmem, ad, bd, idesc, (kb | k) != 0 ? 1u : 0u);
          }
          tc::mma_commit(tc::smem_u32(&ss->empty[stage]));   // frees the stage when these MMAs finish
          issued_any = true;
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        tc::mma_commit(tc::smem_u32(&ss->tmem_full[buf]));   // accumulator ready for the epilogue
      }
      if (issued_any) {
        // all MMAs issued by this thread complete before TMEM is released
        tc::mma_commit(tc::smem_u32(&ss->drain));
        tc::mbar_wait_drain(tc::smem_u32(&ss->drain), 0, 100000000ull);
      }
    }
  } else if (W4 && warp < 2 + DQ_THREADS / 32) {
    // ---------------- INT4 dequantisation (warps 2..5) ----------------
    const int dtid = threadIdx.x - 64;             // 0..127: rows 2*dtid and 2*dtid + 1 of each B tile
    int stage = 0;
    uint32_t phase = 0;
    bool ok = true;
    bool have = false;
    DqRow cur0, cur1;
    // walk the same (tile, K-block) sequence as the producer, one K-block of loads ahead
    int tile = blockIdx.x, kb = 0;
    if (tile < prm.num_tiles) {
      int m_blk, n_blk;
      tile_coords(tile, num_m, num_n, m_blk, n_blk);
      cur0 = dq_load<MODE>(prm, n_blk, 2 * dtid, 0);
      cur1 = dq_load<MODE>(prm, n_blk, 2 * dtid + 1, 0);
      have = true;
    }
    while (have && ok) {
      // next K-block's loads first
      int nt = tile, nkb = kb + 1;
      if (nkb == num_k) { nkb = 0; nt += gridDim.x; }
      DqRow nxt0, nxt1;
      const bool more = nt < prm.num_tiles;
      if (more) {
        int m_blk, n_blk;
        tile_coords(nt, num_m, num_n, m_blk, n_blk);
        nxt0 = dq_load<MODE>(prm, n_blk, 2 * dtid, nkb);
        nxt1 = dq_load<MODE>(prm, n_blk, 2 * dtid + 1, nkb);
      }
      if (!tc::mbar_wait(tc::smem_u32(&ss->empty[stage]), phase ^ 1u, abort_flag, prm.status)) { ok = false; break; }
      uint8_t* btile = smem + stage * STAGE_BYTES + A_BYTES;
      dq_store(btile, 2 * dtid, cur0);
      dq_store(btile, 2 * dtid + 1, cur1);
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");   // generic writes -> tensor-core reads
      tc::mbar_arrive(tc::smem_u32(&ss->full[stage]));
      if (++stage == STAGES) { stage = 0; phase ^= 1u; }
      tile = nt; kb = nkb; cur0 = nxt0; cur1 = nxt1; have = more;
    }
  } else {
    // ---------------- epilogue (8 warps) ----------------
    const int etid = threadIdx.x - epi_base(W4);    // 0..255
    const int half = etid >> 7;                     // which half of the tile's columns
    const int quad = warp & 3;                      // TMEM lane quadrant this warp may access
    const int row_in_tile = quad * 32 + lane;
    const int r = prm.r;
    int local = 0;
    for (int tile = blockIdx.x; tile < prm.num_tiles; tile += gridDim.x, ++local) {
      int m_blk, n_blk;
      tile_coords(tile, num_m, num_n, m_blk, n_blk);
      const int buf = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      const int64_t m = (int64_t)m_blk * BM + row_in_tile;
      const bool row_ok = m < prm.rows;
      const uint32_t t_row = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * BN);

      if (MODE == MODE_PLAIN) {
        if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) break;
        float* D = static_cast<float*>(prm.Y);
        for (int c0 = half * (bn / 2); c0 < (half + 1) * (bn / 2); c0 += CW) {
          float v[CW];
          tmem_ldN<CW>(t_row + (uint32_t)c0, v);
          const int n = n_blk * bn + c0;
          if (row_ok && n < prm.d_out) {
            storeN<float, CW>(D + m * prm.ldy + n, v, min(CW, prm.d_out - n), prm.vec_ok != 0);
          }
        }
        tc::tc_fence_before();
        tc::mbar_arrive(tc::smem_u32(&ss->tmem_empty[buf]));
        continue;
      }

      const bool ok = epi_pair_tile<TO, RT, MODE, CW>(prm, ss, tbl, etid, half, (int64_t)m_blk * BM, m, row_ok,
                                                      n_blk, bn, buf,
                                                      acc_phase, t_row, abort_flag);
      if (!ok) break;
      tc::tc_fence_before();
      tc::mbar_arrive(tc::smem_u32(&ss->tmem_empty[buf]));
    }
  }

  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem_base, TMEM_COLS);
  }
}

}  // namespace pairtc
}  // namespace zoact
