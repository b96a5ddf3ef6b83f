// Pair forward on CTA pairs (tcgen05 cta_group::2): the same computation as
// pair_tc_kernel (Section 3, the perturbed forward pass stacked over both
// signs), with 256-row tiles split across the two SMs of a cluster.
//
// Each CTA loads its 128 rows of X and half of the tile's W rows (bn / 2) into
// its own shared memory; the leader CTA issues tcgen05.mma.cta_group::2
// 256 x bn x 16, which reads the operands of both CTAs and accumulates rows
// 0..127 in the leader's TMEM and rows 128..255 in the peer's.  Per SM this
// moves half the W bytes of the one-CTA kernel for the same FLOPs, so the ring
// holds 6 stages of 32 KB.  Barriers: each producer arrives (with its byte
// count) on the leader's stage barrier and its TMA completes there; the
// leader's commits are multicast to both CTAs' stage-free and
// accumulator-ready barriers; each CTA's epilogue signals the leader's
// accumulator-free barrier once all of its threads have read the tile.
// Gated mode: the leader's half of B is W_gate, the peer's W_up, so the
// accumulator columns are [gate | up] as in the one-CTA kernel.
//
// INT4 weights (W4, stacked rows with the whole low-rank term on the MMA; opt-in,
// ZOACT_INT4=kernel): W comes as packed nibbles and never as bf16 in HBM.  Per
// K-block each CTA's producer brings its 128 rows of packed bytes (4 KB) and
// their fp16 scales (a box of 8 groups, 2 KB) by TMA into the stage's B slot,
// completing on a CTA-local barrier (raw).  Eight more warps per CTA (576
// threads) dequantise in batches of DQ_BATCH stages: they read every packed
// half-row, synchronise, overwrite the slots with the 128-byte-swizzled bf16 B
// half -- every weight q * s formed in fp32 (exact) and rounded once to bf16,
// the value an expansion of W to bf16 holds -- fence the async proxy, and one
// thread arrives on the leader's stage barriers: the batch's first with
// cluster-scope release, the others relaxed (the MMA issuer, which waits with
// cluster-scope acquire, takes the stages in order).  The leader's stage
// barrier counts two dequantising arrivals besides the two producers' (whose
// TMA on it brings only X).
// Measured on the Llama-3-8B gate/up shapes (8192 stacked rows): one release per
// stage made a gated call 3.3x slower than expanding W first (a cluster-scope
// release took ~0.5 us); batches of three and eight warps bring it to 1.8x
// (2.09 vs 1.14 ms).  A separate ring that fetched the packed blocks ahead of
// their stages, with two groups taking alternate batches, measured 2.17 ms;
// with no dequantisation at all (only its waits, barriers and arrivals) that
// structure still took 1.47 ms.  The expansion therefore stays the default.
#pragma once
#include "pair_tc_kernel.cuh"

namespace zoact {
namespace pairtc {

constexpr int STAGES2 = 6;
constexpr int B_HALF_BYTES = (BN / 2) * BK * 2;
constexpr int STAGE2_BYTES = A_BYTES + B_HALF_BYTES;
constexpr int SMEM2_BYTES = 1024 + STAGES2 * STAGE2_BYTES + TBL_FLOATS * 4 + 256;
constexpr int BM2 = 2 * BM;
// Staged output (whole low-rank term on the MMA: no tables): each epilogue
// warpgroup owns one 16 KB buffer in the table region for 128 rows x 128 bytes.
constexpr int STG_BYTES = 16384;
static_assert(2 * STG_BYTES <= TBL_FLOATS * 4, "staging buffers exceed the table region");
// Staged output of the two signs on a shared input: the Z tables (gate, up) fill the
// region's first MIRROR_STG_OFF bytes and each warpgroup stages 16 columns of both
// signs (2 x 128 rows x 32 bytes) above them.
constexpr int MIRROR_STG_OFF = 17408;
constexpr int MIRROR_STG_BYTES = 8192;
static_assert(MIRROR_STG_OFF % 1024 == 0 && MIRROR_STG_OFF + 2 * MIRROR_STG_BYTES <= TBL_FLOATS * 4,
              "mirror staging buffers exceed the table region");


struct SharedState2 {
  uint64_t full[STAGES2];
  uint64_t empty[STAGES2];
  uint64_t tmem_full[2];
  uint64_t tmem_empty[2];
  uint64_t drain;
  uint64_t tload[2];      // fused loss: target chunk landed in a warpgroup's staging buffer
  uint32_t tmem_base;
  int abort_flag;
  int epi_ok;
  int sk_last;            // split tail: this CTA's piece was the tile's last to finish
  int dq_ok;              // INT4: the dequantising group's stage waits succeeded
  uint64_t raw[STAGES2];  // INT4: the stage's packed weights and scales landed (CTA-local TMA)
};
static_assert(sizeof(SharedState2) <= 256, "barrier block outgrew its shared-memory slot");
static_assert(SMEM2_BYTES <= 232448, "dynamic shared memory above the 227 KB a CTA may use");

namespace tc2 {

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to(uint32_t saddr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
  return r;
}
// Arrivals on a barrier of (possibly) the other CTA, with the default (CTA-scope
// release) semantics: a cluster-scope release here would order the arrival
// after this thread's outstanding bulk copies and serialise the copy ring.
__device__ __forceinline__ void arrive_expect_tx_cluster(uint32_t bar_cluster, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cluster.b64 _, [%0], %1;" ::"r"(bar_cluster), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void arrive_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// An arrival with cluster-scope release: shared-memory writes this CTA made before it (and fenced for the
// async proxy) are visible to a cluster-scope acquire of the completed phase in the other CTA.
__device__ __forceinline__ void arrive_release_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// An arrival without ordering: only for a phase whose data an earlier release arrival (to a barrier the
// consumer acquires first) already covers.
__device__ __forceinline__ void arrive_relaxed_cluster(uint32_t bar_cluster) {
  asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// TMA tile load into this CTA's shared memory whose completion is signalled on
// a barrier of the leader CTA of the pair.
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* map, int32_t x, int32_t y,
                                                 uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
      "[%4];" ::"r"(dst),
      "l"(map), "r"(x), "r"(y), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ void tmem_alloc2(uint32_t dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
               : "memory");
}
__device__ __forceinline__ void tmem_relinquish2() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc2(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void mma2_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}
// Arrive on the barrier at this offset in both CTAs of the pair once the
// issuing thread's MMAs have completed.
__device__ __forceinline__ void commit2_both(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
      "h"((uint16_t)3)
      : "memory");
}
__device__ __forceinline__ void commit2_own(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

}  // namespace tc2

// Byte offset of 16-byte granule g of row r in a 128-byte-swizzled staging box
// (the layout a SWIZZLE_128B tensor map reads: granule index XOR row mod 8).
__device__ __forceinline__ uint32_t sw128_off(int r, int g) {
  return (uint32_t)(r * 128 + ((g ^ (r & 7)) << 4));
}

template <typename TO>
__device__ __forceinline__ uint4 pack8_16(const float* v) {
  return make_uint4(pack2(v[0], v[1], (TO*)nullptr), pack2(v[2], v[3], (TO*)nullptr), pack2(v[4], v[5], (TO*)nullptr),
                    pack2(v[6], v[7], (TO*)nullptr));
}

// Write PW values of staging row rl, starting at column p of the chunk, as
// 16-byte granules: 128-byte swizzled rows (full chunks) or unswizzled rows of
// 16 columns (narrow chunks).
template <typename TO, int PW>
__device__ __forceinline__ void stage_granules(uint32_t sbuf, int rl, int p, const float* v, bool full) {
  constexpr int EB = (int)sizeof(TO);
  constexpr int GE = 16 / EB;       // values per granule
#pragma unroll
  for (int q = 0; q < PW / GE; ++q) {
    const int gi = p / GE + q;
    const uint32_t off = full ? sw128_off(rl, gi) : (uint32_t)(rl * 16 * EB + gi * 16);
    if constexpr (EB == 2)
      tc::st_shared_v4(sbuf + off, pack8_16<TO>(v + 8 * q));
    else
      tc::st_shared_v4(sbuf + off, make_uint4(__float_as_uint(v[4 * q]), __float_as_uint(v[4 * q + 1]),
                                              __float_as_uint(v[4 * q + 2]), __float_as_uint(v[4 * q + 3])));
  }
}

// Epilogue of one accumulator tile whose whole low-rank term is in the
// accumulator, written through shared memory: this warpgroup's columns go in
// chunks of 128 bytes per row (then 16-column chunks for the remainder) into
// its staging buffer, and one thread stores each chunk with a bulk tensor store
// of 128 rows (rows and columns outside Y are dropped by the store).  Returns
// false when the accumulator wait gave up.  `pending`: the issuing thread has
// bulk stores in flight.
template <typename TO, int MODE>
__device__ __forceinline__ bool epi_all_staged(const Params& prm, const TmaSet& tm, SharedState2* ss, uint8_t* stg,
                                               int etid, int half, int rl, int64_t row0, int n_blk, int bn, int buf,
                                               uint32_t acc_phase, uint32_t t_row, volatile int* abort_flag,
                                               bool& pending) {
  constexpr bool GATED = MODE == MODE_GATED;
  constexpr int EB = (int)sizeof(TO);
  constexpr int CC = 128 / EB;      // columns of a full chunk (one swizzled 128-byte row each)
  constexpr int NC = 16;            // columns of a narrow chunk (unswizzled rows of 16 * EB bytes)
  if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
  const int ncol_tile = GATED ? BN / 2 : bn;
  const int wcols = ncol_tile / 2;  // this warpgroup's columns, a multiple of 16 (of 64 with row scales)
  const int cb = half * wcols;
  const bool issuer = (etid & 127) == 0;
  const uint32_t sbuf = tc::smem_u32(stg + half * STG_BYTES);
  const int64_t row = row0 + rl;
  const bool row_ok = row < prm.rows;
  // row scales: the input row's 1/s (uniform test), and this row's running sum of squares of the stored
  // outputs of the current 64-column part
  const bool scaled = prm.in_scale != nullptr;
  const float rs = scaled && row_ok ? __ldg(prm.in_scale + row) : 1.f;
  const bool sums = prm.out_sumsq != nullptr;
  float ssq = 0.f;
  int part = -1;
  for (int c = 0; c < wcols;) {
    const int n = n_blk * ncol_tile + cb + c;
    if (n >= prm.d_out) break;                      // uniform over the warpgroup
    const bool full = wcols - c >= CC;
    const int cw = full ? CC : NC;
    if (sums && (n >> 6) != part) {                 // a new 64-column part (parts never straddle chunks)
      if (part >= 0 && row_ok) prm.out_sumsq[(int64_t)part * prm.rows + row] = ssq;
      part = n >> 6;
      ssq = 0.f;
    }
    if (issuer && pending) tc::bulk_wait_read0();   // the buffer's previous store has read it
    tc::named_bar_sync(4 + half, 128);
    if (full) {
      // 32 columns per TMEM load: few tcgen05.ld / wait pairs beside the MMAs
#pragma unroll 1
      for (int p = 0; p < CC; p += 32) {
        float v[32];
        if (GATED) {
          float u[32];
          tc::tmem_ld32(t_row + (uint32_t)(cb + c + p), v);
          tc::tmem_ld32(t_row + (uint32_t)(BN / 2 + cb + c + p), u);
          if (scaled) {
#pragma unroll
            for (int i = 0; i < 32; ++i) { v[i] *= rs; u[i] *= rs; }
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = silu_fast(v[i]) * u[i];
        } else {
          tc::tmem_ld32(t_row + (uint32_t)(cb + c + p), v);
          if (scaled) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= rs;
          }
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = apply_act(v[i], prm.act);
        }
        if (sums) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float y = to_f32<TO>(from_f32<TO>(v[i]));   // the value Y stores
            if (n + p + i < prm.d_out) ssq = fmaf(y, y, ssq);
          }
        }
        stage_granules<TO, 32>(sbuf, rl, p, v, true);
      }
    } else {
      float v[16];
      if (GATED) {
        float u[16];
        tc::tmem_ld16(t_row + (uint32_t)(cb + c), v);
        tc::tmem_ld16(t_row + (uint32_t)(BN / 2 + cb + c), u);
        if (scaled) {
#pragma unroll
          for (int i = 0; i < 16; ++i) { v[i] *= rs; u[i] *= rs; }
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = silu_fast(v[i]) * u[i];
      } else {
        tc::tmem_ld16(t_row + (uint32_t)(cb + c), v);
        if (scaled) {
#pragma unroll
          for (int i = 0; i < 16; ++i) v[i] *= rs;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = apply_act(v[i], prm.act);
      }
      if (sums) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float y = to_f32<TO>(from_f32<TO>(v[i]));
          if (n + i < prm.d_out) ssq = fmaf(y, y, ssq);
        }
      }
      stage_granules<TO, 16>(sbuf, rl, 0, v, false);
    }
    tc::fence_proxy_async_smem();                   // the staging writes, before the bulk store reads them
    tc::named_bar_sync(4 + half, 128);
    if (issuer) {
      tc::tma_store_2d(full ? &tm.y : &tm.y16, n, (int)row0, sbuf);
      tc::bulk_commit();
      pending = true;
    }
    c += cw;
  }
  if (sums && part >= 0 && row_ok) prm.out_sumsq[(int64_t)part * prm.rows + row] = ssq;
  return true;
}

// Epilogue of the two signs of one query on a shared input (C p in the
// accumulator, c_1 = -c_0, 16-bit outputs), staged: per column pass the Z
// tables of gate (and up) are built at tbl (and tbl + TSZ), then each warpgroup
// forms acc +- c_0 Z p for 16 columns of its 128 rows, writes both signs into
// its staging buffer and one thread stores them with bulk tensor stores through
// tm.y (rows [0, T) of Y) and tm.y16 (rows [T, 2T)), which drop rows past T and
// columns past d_out.  Returns false when the accumulator wait gave up.
template <typename TO, int RT, int MODE>
__device__ __forceinline__ bool epi_mirror_staged(const Params& prm, const TmaSet& tm, SharedState2* ss, float* tbl,
                                                  int etid, int half, int rl, int64_t row0, int64_t m, bool row_ok,
                                                  int n_blk, int bn, int buf, uint32_t acc_phase, uint32_t t_row,
                                                  volatile int* abort_flag, bool& pending) {
  constexpr bool GATED = MODE == MODE_GATED;
  constexpr int SLOTS = GATED ? gated_slots(RT) : pair_slots(RT);
  constexpr int STRIDE = SLOTS + TPAD;
  constexpr int TSZ = RT * STRIDE;
  static_assert((GATED ? 2 : 1) * TSZ * 4 <= MIRROR_STG_OFF, "mirror tables overlap the staging buffers");
  static_assert(sizeof(TO) == 2, "staged mirror output is 16-bit");
  const int r = prm.r;
  float p[RT], p2[RT];
  const bool vec = prm.vec_ok != 0;
  load_p<RT>(p, prm.P, m, r, row_ok, vec);
  if (GATED) load_p<RT>(p2, prm.P2, m, r, row_ok, vec);
  const int ncol_tile = GATED ? BN / 2 : bn;
  const float cz = prm.coef[0];
  const int zq = prm.zq[0];
  const bool issuer = (etid & 127) == 0;
  const uint32_t sp = tc::smem_u32(tbl) + MIRROR_STG_OFF + half * MIRROR_STG_BYTES;   // + sign; - sign at +4096
  bool waited = false;
  for (int s0 = 0; s0 < ncol_tile; s0 += SLOTS) {
    const int cwid = min(SLOTS, ncol_tile - s0);            // a multiple of 32
    const int col0 = n_blk * ncol_tile + s0;
    tc::named_bar_sync(1, EPI_THREADS);                     // previous pass's readers are done
    build_tables_z<RT>(tbl, nullptr, STRIDE, prm.Zt + zq * prm.zt_qstride, prm.Zt + zq * prm.zt_qstride, 1.f, 0.f,
                       col0, cwid, prm.d_out, r, etid);
    if (GATED)
      build_tables_z<RT>(tbl + TSZ, nullptr, STRIDE, prm.Zt2 + zq * prm.zt_qstride, prm.Zt2 + zq * prm.zt_qstride,
                         1.f, 0.f, col0, cwid, prm.d_out, r, etid);
    tc::named_bar_sync(1, EPI_THREADS);
    if (!waited) {
      if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
      waited = true;
    }
    const int cbeg = s0 + half * (cwid / 2);
    for (int c0 = cbeg; c0 < cbeg + cwid / 2; c0 += 16) {
      const int n = n_blk * ncol_tile + c0;
      if (n >= prm.d_out) break;                            // uniform over the warpgroup
      if (issuer && pending) tc::bulk_wait_read0();         // the buffers' previous stores have read them
      tc::named_bar_sync(4 + half, 128);
#pragma unroll
      for (int k8 = 0; k8 < 16; k8 += 8) {
        float hp[8], hm[8];
        if (GATED) {
          float g[8], u[8], sg[8], su[8];
          tc::tmem_ld8(t_row + (uint32_t)(c0 + k8), g);
          tc::tmem_ld8(t_row + (uint32_t)(BN / 2 + c0 + k8), u);
          lowrank_t<RT, 8>(tbl, STRIDE, c0 + k8 - s0, p, sg);
          lowrank_t<RT, 8>(tbl + TSZ, STRIDE, c0 + k8 - s0, p2, su);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            hp[i] = silu_fast(fmaf(cz, sg[i], g[i])) * fmaf(cz, su[i], u[i]);
            hm[i] = silu_fast(fmaf(-cz, sg[i], g[i])) * fmaf(-cz, su[i], u[i]);
          }
        } else {
          float a[8], sl[8];
          tc::tmem_ld8(t_row + (uint32_t)(c0 + k8), a);
          lowrank_t<RT, 8>(tbl, STRIDE, c0 + k8 - s0, p, sl);
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            hp[i] = apply_act(fmaf(cz, sl[i], a[i]), prm.act);
            hm[i] = apply_act(fmaf(-cz, sl[i], a[i]), prm.act);
          }
        }
        tc::st_shared_v4(sp + (uint32_t)(rl * 32 + (k8 >> 3) * 16), pack8_16<TO>(hp));
        tc::st_shared_v4(sp + 4096u + (uint32_t)(rl * 32 + (k8 >> 3) * 16), pack8_16<TO>(hm));
      }
      tc::fence_proxy_async_smem();
      tc::named_bar_sync(4 + half, 128);
      if (issuer) {
        tc::tma_store_2d(&tm.y, n, (int)row0, sp);
        tc::tma_store_2d(&tm.y16, n, (int)row0, sp + 4096u);
        tc::bulk_commit();
        pending = true;
      }
    }
  }
  return true;
}

// Column order of a 16-column table chunk for four-row epilogue threads: thread t
// (q = t % 4) uses chunk columns 2q, 2q+1, 8+2q, 9+2q, stored contiguously at 4q.
__device__ __forceinline__ int perm16(int c) { return 4 * ((c & 7) >> 1) + ((c >> 3) << 1) + (c & 1); }

// Z table of one query over columns [col0, col0 + ncols) in 16-column chunks
// permuted by perm16: tb[j * stride + (s & ~15) + perm16(s & 15)] = c Z[j][col0 + s],
// zero where col0 + s >= d_out or j >= r.  One thread per 4 consecutive columns.
template <int RT>
__device__ __forceinline__ void build_tables_z16(float* tb, int stride, const float* __restrict__ Zq, float c, int col0,
                                                 int ncols, int d_out, int r, int tid) {
  const int per_row = ncols / 4;
  for (int it = tid; it < RT * per_row; it += EPI_THREADS) {
    const int j = it / per_row, s = 4 * (it - j * per_row);
    const int col = col0 + s;
    float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    if (j < r && col < d_out) z = *reinterpret_cast<const float4*>(Zq + (int64_t)j * d_out + col);
    float* row = tb + j * stride + (s & ~15);
    const int cc = s & 15;                      // columns cc, cc+1 and cc+2, cc+3 land as two pairs
    *reinterpret_cast<float2*>(row + perm16(cc)) = make_float2(c * z.x, c * z.y);
    *reinterpret_cast<float2*>(row + perm16(cc + 2)) = make_float2(c * z.z, c * z.w);
  }
}

// The staged two-sign epilogue with four rows per thread (rank tile <= 16; a gated
// launch whose gate and up share one projection P).  TMEM is read with 16x256b
// loads, so each thread holds rows t/4 + 8k (k = 0..3) of its warp's 32 and four
// columns of each 16-column chunk; one 16-byte shared read of the permuted Z table
// then feeds 16 FMAs (4 rows x 4 columns) instead of 4, a quarter of the table
// reads of the row-per-thread form.  Outputs are staged as in epi_mirror_staged.
template <typename TO, int RT, int MODE>
__device__ __forceinline__ bool epi_mirror4_staged(const Params& prm, const TmaSet& tm, SharedState2* ss, float* tbl,
                                                   int etid, int half, int quad, int lane, int64_t row0, int n_blk,
                                                   int bn, int buf, uint32_t acc_phase, uint32_t t_q,
                                                   volatile int* abort_flag, bool& pending) {
  constexpr bool GATED = MODE == MODE_GATED;
  constexpr int SLOTS = GATED ? gated_slots(RT) : pair_slots(RT);
  constexpr int STRIDE = SLOTS + TPAD;
  constexpr int TSZ = RT * STRIDE;
  static_assert(RT <= 16, "four rows of projections per thread");
  static_assert((GATED ? 2 : 1) * TSZ * 4 <= MIRROR_STG_OFF, "mirror tables overlap the staging buffers");
  static_assert(SLOTS % 32 == 0 && STRIDE % 4 == 0, "16-column chunks of 16-byte aligned table rows");
  static_assert(sizeof(TO) == 2, "staged mirror output is 16-bit");
  const int r = prm.r;
  const int q = lane & 3, rq = lane >> 2;
  const bool vec = prm.vec_ok != 0;
  float p[4][RT];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int64_t m = row0 + quad * 32 + rq + 8 * k;
    load_p<RT>(p[k], prm.P, m, r, m < prm.rows, vec);
  }
  const int ncol_tile = GATED ? BN / 2 : bn;
  const float cz = prm.coef[0];
  const int zq = prm.zq[0];
  const bool issuer = (etid & 127) == 0;
  const uint32_t sp = tc::smem_u32(tbl) + MIRROR_STG_OFF + half * MIRROR_STG_BYTES;   // + sign; - sign at +4096
  bool waited = false;
  for (int s0 = 0; s0 < ncol_tile; s0 += SLOTS) {
    const int cwid = min(SLOTS, ncol_tile - s0);            // a multiple of 32
    const int col0 = n_blk * ncol_tile + s0;
    tc::named_bar_sync(1, EPI_THREADS);                     // previous pass's readers are done
    build_tables_z16<RT>(tbl, STRIDE, prm.Zt + zq * prm.zt_qstride, 1.f, col0, cwid, prm.d_out, r, etid);
    if (GATED)
      build_tables_z16<RT>(tbl + TSZ, STRIDE, prm.Zt2 + zq * prm.zt_qstride, 1.f, col0, cwid, prm.d_out, r, etid);
    tc::named_bar_sync(1, EPI_THREADS);
    if (!waited) {
      if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
      waited = true;
    }
    const int cbeg = s0 + half * (cwid / 2);
    for (int c0 = cbeg; c0 < cbeg + cwid / 2; c0 += 16) {
      const int n = n_blk * ncol_tile + c0;
      if (n >= prm.d_out) break;                            // uniform over the warpgroup
      float g[16], u[16];
      tc::tmem_ld_rows4(t_q + (uint32_t)c0, g);
      if (GATED) tc::tmem_ld_rows4(t_q + (uint32_t)(BN / 2 + c0), u);
      float2 zg[4][2], zu[4][2];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        zg[k][0] = zg[k][1] = zu[k][0] = zu[k][1] = make_float2(0.f, 0.f);
      }
      const float* tg = tbl + (c0 - s0) + 4 * q;
#pragma unroll
      for (int j = 0; j < RT; ++j) {
        const float4 a = *reinterpret_cast<const float4*>(tg + j * STRIDE);
        float4 b = a;
        if (GATED) b = *reinterpret_cast<const float4*>(tg + TSZ + j * STRIDE);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
          const float2 pj = make_float2(p[k][j], p[k][j]);
          zg[k][0] = ffma2(make_float2(a.x, a.y), pj, zg[k][0]);
          zg[k][1] = ffma2(make_float2(a.z, a.w), pj, zg[k][1]);
          if (GATED) {
            zu[k][0] = ffma2(make_float2(b.x, b.y), pj, zu[k][0]);
            zu[k][1] = ffma2(make_float2(b.z, b.w), pj, zu[k][1]);
          }
        }
      }
      if (issuer && pending) tc::bulk_wait_read0();         // the buffers' previous stores have read them
      tc::named_bar_sync(4 + half, 128);
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        const float zgk[4] = {zg[k][0].x, zg[k][0].y, zg[k][1].x, zg[k][1].y};
        const float zuk[4] = {zu[k][0].x, zu[k][0].y, zu[k][1].x, zu[k][1].y};
        float hp[4], hm[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float gv = g[4 * k + i];
          if (GATED) {
            const float uv = u[4 * k + i];
            hp[i] = silu_fast(fmaf(cz, zgk[i], gv)) * fmaf(cz, zuk[i], uv);
            hm[i] = silu_fast(fmaf(-cz, zgk[i], gv)) * fmaf(-cz, zuk[i], uv);
          } else {
            hp[i] = apply_act(fmaf(cz, zgk[i], gv), prm.act);
            hm[i] = apply_act(fmaf(-cz, zgk[i], gv), prm.act);
          }
        }
        // row quad*32 + rq + 8k of the staging rows (32 bytes each): columns 2q, 2q+1 and 8+2q, 9+2q
        const uint32_t ro = (uint32_t)((quad * 32 + rq + 8 * k) * 32 + 4 * q);
        tc::st_shared_b32(sp + ro, pack2(hp[0], hp[1], (TO*)nullptr));
        tc::st_shared_b32(sp + ro + 16u, pack2(hp[2], hp[3], (TO*)nullptr));
        tc::st_shared_b32(sp + 4096u + ro, pack2(hm[0], hm[1], (TO*)nullptr));
        tc::st_shared_b32(sp + 4096u + ro + 16u, pack2(hm[2], hm[3], (TO*)nullptr));
      }
      tc::fence_proxy_async_smem();
      tc::named_bar_sync(4 + half, 128);
      if (issuer) {
        tc::tma_store_2d(&tm.y, n, (int)row0, sp);
        tc::tma_store_2d(&tm.y16, n, (int)row0, sp + 4096u);
        tc::bulk_commit();
        pending = true;
      }
    }
  }
  return true;
}

// Column width of one table pass of the staged q-query epilogue: four permuted tables
// (two blocks x gate, up) of RT x (MULTI4_SLOTS + TPAD) floats below the staging buffers.
constexpr int MULTI4_SLOTS = 64;

// The staged epilogue of several evaluation blocks on a shared input (C p in the
// accumulator; the one-sided q-query estimator, or any blocks that are not the two
// signs of one query), four rows per thread as in epi_mirror4_staged.  Blocks go in
// pairs: per column pass the permuted tables c_b Z_b of both (gate at tbl + t TSZ,
// up at tbl + (2 + t) TSZ; none for c_b = 0) are built, then each warpgroup forms
// acc + c_b Z_b p for 16 columns of its 128 rows, one block after the other, stages
// both blocks' outputs and one thread stores them through tm.y, a 3-D map over
// the blocks' [T, d_out] slabs that drops rows past T and columns past d_out.
template <typename TO, int RT, int MODE>
__device__ __forceinline__ bool epi_multi4_staged(const Params& prm, const TmaSet& tm, SharedState2* ss, float* tbl,
                                                  int etid, int half, int quad, int lane, int64_t row0, int n_blk,
                                                  int bn, int buf, uint32_t acc_phase, uint32_t t_q,
                                                  volatile int* abort_flag, bool& pending) {
  constexpr bool GATED = MODE == MODE_GATED;
  constexpr int SLOTS = MULTI4_SLOTS;
  constexpr int STRIDE = SLOTS + TPAD;
  constexpr int TSZ = RT * STRIDE;
  static_assert(RT <= 16, "four rows of projections per thread");
  static_assert((GATED ? 4 : 2) * TSZ * 4 <= MIRROR_STG_OFF, "q-query tables overlap the staging buffers");
  static_assert(sizeof(TO) == 2, "staged q-query output is 16-bit");
  const int r = prm.r;
  const int q = lane & 3, rq = lane >> 2;
  const bool vec = prm.vec_ok != 0;
  float p[4][RT];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const int64_t m = row0 + quad * 32 + rq + 8 * k;
    load_p<RT>(p[k], prm.P, m, r, m < prm.rows, vec);
  }
  const int ncol_tile = GATED ? BN / 2 : bn;
  const bool issuer = (etid & 127) == 0;
  const uint32_t sp = tc::smem_u32(tbl) + MIRROR_STG_OFF + half * MIRROR_STG_BYTES;   // block slot t at +4096 t
  bool waited = false;
  for (int s0 = 0; s0 < ncol_tile; s0 += SLOTS) {
    const int cwid = min(SLOTS, ncol_tile - s0);            // a multiple of 32
    const int col0 = n_blk * ncol_tile + s0;
    for (int bp = 0; bp < prm.nb; bp += 2) {
      const int nblk = min(2, prm.nb - bp);
      tc::named_bar_sync(1, EPI_THREADS);                   // previous pass's readers are done
      for (int t = 0; t < nblk; ++t) {
        const int b = bp + t;
        if (prm.coef[b] == 0.f) continue;                   // its term is already in the accumulator
        build_tables_z16<RT>(tbl + t * TSZ, STRIDE, prm.Zt + prm.zq[b] * prm.zt_qstride, prm.coef[b], col0, cwid,
                             prm.d_out, r, etid);
        if (GATED)
          build_tables_z16<RT>(tbl + (2 + t) * TSZ, STRIDE, prm.Zt2 + prm.zq[b] * prm.zt_qstride, prm.coef[b], col0,
                               cwid, prm.d_out, r, etid);
      }
      tc::named_bar_sync(1, EPI_THREADS);
      if (!waited) {
        if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
        waited = true;
      }
      const int cbeg = s0 + half * (cwid / 2);
      for (int c0 = cbeg; c0 < cbeg + cwid / 2; c0 += 16) {
        const int n = n_blk * ncol_tile + c0;
        if (n >= prm.d_out) break;                          // uniform over the warpgroup
        float g[16], u[16];
        tc::tmem_ld_rows4(t_q + (uint32_t)c0, g);
        if (GATED) tc::tmem_ld_rows4(t_q + (uint32_t)(BN / 2 + c0), u);
        if (issuer && pending) tc::bulk_wait_read0();       // the buffers' previous stores have read them
        tc::named_bar_sync(4 + half, 128);
#pragma unroll 1
        for (int t = 0; t < nblk; ++t) {
          float2 zg[4][2], zu[4][2];
#pragma unroll
          for (int k = 0; k < 4; ++k) zg[k][0] = zg[k][1] = zu[k][0] = zu[k][1] = make_float2(0.f, 0.f);
          if (prm.coef[bp + t] != 0.f) {
            const float* tg = tbl + t * TSZ + (c0 - s0) + 4 * q;
            const float* tu = tbl + (2 + t) * TSZ + (c0 - s0) + 4 * q;
#pragma unroll
            for (int j = 0; j < RT; ++j) {
              const float4 a = *reinterpret_cast<const float4*>(tg + j * STRIDE);
              float4 bv = a;
              if (GATED) bv = *reinterpret_cast<const float4*>(tu + j * STRIDE);
#pragma unroll
              for (int k = 0; k < 4; ++k) {
                const float2 pj = make_float2(p[k][j], p[k][j]);
                zg[k][0] = ffma2(make_float2(a.x, a.y), pj, zg[k][0]);
                zg[k][1] = ffma2(make_float2(a.z, a.w), pj, zg[k][1]);
                if (GATED) {
                  zu[k][0] = ffma2(make_float2(bv.x, bv.y), pj, zu[k][0]);
                  zu[k][1] = ffma2(make_float2(bv.z, bv.w), pj, zu[k][1]);
                }
              }
            }
          }
          const uint32_t sb = sp + 4096u * (uint32_t)t;
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float zgk[4] = {zg[k][0].x, zg[k][0].y, zg[k][1].x, zg[k][1].y};
            const float zuk[4] = {zu[k][0].x, zu[k][0].y, zu[k][1].x, zu[k][1].y};
            float h[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              if (GATED)
                h[i] = silu_fast(g[4 * k + i] + zgk[i]) * (u[4 * k + i] + zuk[i]);
              else
                h[i] = apply_act(g[4 * k + i] + zgk[i], prm.act);
            }
            const uint32_t ro = (uint32_t)((quad * 32 + rq + 8 * k) * 32 + 4 * q);
            tc::st_shared_b32(sb + ro, pack2(h[0], h[1], (TO*)nullptr));
            tc::st_shared_b32(sb + ro + 16u, pack2(h[2], h[3], (TO*)nullptr));
          }
        }
        tc::fence_proxy_async_smem();
        tc::named_bar_sync(4 + half, 128);
        if (issuer) {
          for (int t = 0; t < nblk; ++t) tc::tma_store_3d(&tm.y, n, (int)row0, bp + t, sp + 4096u * (uint32_t)t);
          tc::bulk_commit();
          pending = true;
        }
      }
    }
  }
  return true;
}

// Compensated fp32 sum of squares: d^2 = p + e exactly (p = fp32(d d), e = fma(d, d, -p));
// the p go into a Neumaier sum (the rounding error of every add carried in c) and the
// tiny e into a plain sum, so S = s + c + e keeps about twice fp32 precision without
// fp64 adds -- enough that the difference of the two signs' sums is still accurate.
struct CompSum {
  float s = 0.f, c = 0.f, e = 0.f;
  __device__ __forceinline__ void add_sq(float d) {
    const float p = d * d;
    e += fmaf(d, d, -p);
    const float t = s + p;
    c += fabsf(s) >= p ? (s - t) + p : (p - t) + s;
    s = t;
  }
  __device__ __forceinline__ double value() const { return (double)s + (double)c + (double)e; }
};

// 8 16-bit values of a 16-byte granule.
template <typename TO>
__device__ __forceinline__ void unpack8_16(uint4 g, float* v) {
  const uint32_t w[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    TO lo, hi;
    const uint16_t a = (uint16_t)(w[i] & 0xFFFFu), b = (uint16_t)(w[i] >> 16);
    memcpy(&lo, &a, 2);
    memcpy(&hi, &b, 2);
    v[2 * i] = to_f32<TO>(lo);
    v[2 * i + 1] = to_f32<TO>(hi);
  }
}

// Loss-pair epilogue of one accumulator tile (STAGE_LOSS: stacked rows, the whole
// low-rank term in the accumulator, T a multiple of 256 so that this CTA's 128 rows
// all belong to one sign).  Y is not written: for each 128-byte chunk of this
// warpgroup's columns one thread loads the target's matching [128 x chunk] box into
// the warpgroup's staging buffer (tm.y, 128-byte swizzled; tm.y16 for 16-column
// remainders), and every thread adds (round(y) - t)^2 of its row -- y rounded to
// Y's 16-bit type as zoact_loss_pair would read it -- to the compensated sum of
// squares of the row's sign.  Columns past d_out are skipped (their accumulator columns hold the
// other block's low-rank term).  Returns false when the accumulator wait gave up.
template <typename TO>
__device__ __forceinline__ bool epi_loss_staged(const Params& prm, const TmaSet& tm, SharedState2* ss, uint8_t* stg,
                                                int etid, int half, int rl, int64_t row0, int n_blk, int bn, int buf,
                                                uint32_t acc_phase, uint32_t t_row, volatile int* abort_flag,
                                                uint32_t& tphase, CompSum* acc) {
  constexpr int EB = (int)sizeof(TO);
  constexpr int CC = 128 / EB;      // columns of a full chunk
  constexpr int NC = 16;            // columns of a narrow chunk
  static_assert(EB == 2, "fused loss of 16-bit outputs");
  if (!epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid)) return false;
  const int wcols = bn / 2;
  const int cb = half * wcols;
  const int sgn = row0 >= prm.T ? 1 : 0;
  const int64_t trow0 = row0 - (sgn ? prm.T : 0);
  const bool issuer = (etid & 127) == 0;
  const uint32_t sbuf = tc::smem_u32(stg + half * STG_BYTES);
  const uint32_t tbar = tc::smem_u32(&ss->tload[half]);
  CompSum& S = acc[sgn];
  for (int c = 0; c < wcols;) {
    const int n = n_blk * bn + cb + c;
    if (n >= prm.d_out) break;                      // uniform over the warpgroup
    const bool full = wcols - c >= CC;
    const int cw = full ? CC : NC;
    if (prm.has_target) {
      tc::named_bar_sync(4 + half, 128);            // the previous chunk's readers of the buffer are done
      if (issuer) {
        tc::mbar_arrive_expect_tx(tbar, (uint32_t)(BM * cw * EB));
        tc::tma_load_2d(sbuf, full ? &tm.y : &tm.y16, n, (int)trow0, tbar);
        // bounded: on expiry the abort flag is set and the launch writes no loss, but the warpgroup stays
        // on one path (no thread leaves a named barrier short)
        tc::mbar_wait(tbar, tphase, abort_flag, prm.status);
      }
      tphase ^= 1u;
      tc::named_bar_sync(4 + half, 128);            // the chunk has landed
    }
    for (int p = 0; p < cw; p += 16) {
      float v[16];
      tc::tmem_ld16(t_row + (uint32_t)(cb + c + p), v);
#pragma unroll
      for (int g = 0; g < 2; ++g) {
        float t8[8];
        if (prm.has_target) {
          const int gi = (p >> 3) + g;
          unpack8_16<TO>(tc::ld_shared_v4(sbuf + (full ? sw128_off(rl, gi) : (uint32_t)(rl * NC * EB + gi * 16))),
                         t8);
        } else {
#pragma unroll
          for (int i = 0; i < 8; ++i) t8[i] = 0.f;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const float y = to_f32<TO>(from_f32<TO>(apply_act(v[8 * g + i], prm.act)));
          if (n + p + 8 * g + i < prm.d_out) S.add_sq(y - t8[i]);   // y - t is exact in fp32
        }
      }
    }
    c += cw;
  }
  return true;
}

// The end of a fused-loss launch: the epilogue threads' sums (two signs) are added
// in a fixed order into this CTA's partial; the last CTA to finish (atomic ticket)
// adds all partials in CTA order and writes {L+, L-, D, a}, D = L+ - L- and
// a = D / (2 eps), then resets the ticket.  red: 2 x EPI_THREADS doubles of shared memory.
__device__ __forceinline__ void loss_finish(const Params& prm, const CompSum* acc, double* red, int etid) {
  red[2 * etid] = acc[0].value();
  red[2 * etid + 1] = acc[1].value();
  tc::named_bar_sync(3, EPI_THREADS);
  if (etid >= 32) return;
  // warp 0 of the epilogue: lane l adds threads l, l + 32, ...; then a fixed butterfly
  double s0 = 0.0, s1 = 0.0;
  for (int i = etid; i < EPI_THREADS; i += 32) { s0 += red[2 * i]; s1 += red[2 * i + 1]; }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s0 += __shfl_xor_sync(0xffffffffu, s0, o);
    s1 += __shfl_xor_sync(0xffffffffu, s1, o);
  }
  unsigned int last = 0;
  if (etid == 0) {
    prm.loss_part[2 * blockIdx.x] = s0;
    prm.loss_part[2 * blockIdx.x + 1] = s1;
    __threadfence();
    last = atomicAdd(prm.loss_ticket, 1u) == gridDim.x - 1 ? 1u : 0u;
  }
  last = __shfl_sync(0xffffffffu, last, 0);
  if (!last) return;
  __threadfence();
  double a0 = 0.0, a1 = 0.0;
  for (unsigned int b = etid; b < gridDim.x; b += 32) {
    a0 += __ldcg(prm.loss_part + 2 * b);
    a1 += __ldcg(prm.loss_part + 2 * b + 1);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    a0 += __shfl_xor_sync(0xffffffffu, a0, o);
    a1 += __shfl_xor_sync(0xffffffffu, a1, o);
  }
  if (etid == 0) {
    const double inv = 1.0 / ((double)prm.T * (double)prm.d_out);
    const double Lp = a0 * inv, Lm = a1 * inv, D = (a0 - a1) * inv;
    const double a = D / (2.0 * (double)prm.loss_eps);
    prm.loss_out[0] = Lp;
    prm.loss_out[1] = Lm;
    prm.loss_out[2] = D;
    prm.loss_out[3] = a;
    if (!isfinite(Lp) || !isfinite(Lm) || !isfinite(a)) record_error(prm.status, ZOACT_ERR_NONFINITE);
    *prm.loss_ticket = 0u;
  }
}

// SMODE (StageMode): STAGE_ALL -- the launch has the whole low-rank term on the
// MMA (aug_mode LOWRANK_ALL_ON_TC) and Y's store maps in tm.y / tm.y16, the
// table region holds the output staging buffers; STAGE_MIRROR -- the two signs
// of one query on a shared input (aug_mode LOWRANK_C_ON_TC, two blocks), the
// region holds the Z tables and two smaller buffers.  A launch that does not
// match its SMODE records ZOACT_ERR_INVALID_ARG and exits before touching
// shared memory.
// One unit of a pair's work: K-blocks [kb0, kb1) of a tile.  Whole tiles have
// npieces = 1; a piece of a split tail tile is piece `piece` (in K order) of
// `npieces` and keeps its partial accumulator in slot `slot`.
struct WorkUnit {
  int tile, kb0, kb1, piece, npieces, slot;
};

// The i-th unit of cluster c: whole tiles c, c + n, ... below sk_first (all tiles
// without a split tail), then at most one tail piece: pair c = j * sk_tiles + t
// takes K range j of tail tile t, so the pieces running side by side cover the
// same K range of neighbouring tiles and share operand panels in L2 as a wave of
// whole tiles does.  False past the last unit.  The producer, the MMA issuer and
// the epilogue walk the same sequence.
__device__ __forceinline__ bool next_unit(const Params& prm, int c, int n, int K, int i, WorkUnit& u) {
  const int lim = prm.sk_tiles > 0 ? prm.sk_first : prm.num_tiles;
  const int whole = c < lim ? (lim - c + n - 1) / n : 0;
  if (i < whole) {
    u.tile = c + i * n; u.kb0 = 0; u.kb1 = K; u.piece = 0; u.npieces = 1; u.slot = -1;
    return true;
  }
  if (prm.sk_tiles == 0 || i != whole || c >= prm.sk_tiles * prm.sk_split) return false;
  const int j = c / prm.sk_tiles, t = c - j * prm.sk_tiles;
  u.tile = prm.sk_first + t;
  u.kb0 = (int)((int64_t)j * K / prm.sk_split);
  u.kb1 = (int)((int64_t)(j + 1) * K / prm.sk_split);
  u.piece = j; u.npieces = prm.sk_split; u.slot = c;
  return true;
}

// A tail piece: the accumulator holds only this piece's K-blocks.  Every piece
// stores its fp32 partial (this CTA's 128 rows x bn columns) in its slot and
// takes a ticket of the tile; the piece that arrives last adds all pieces'
// partials in K order -- its own from TMEM -- and writes the sum back to TMEM,
// where the epilogue finds the whole accumulator.  No CTA waits for another, and
// the fixed order makes the sum independent of which piece ends last.  Returns
// whether this piece was the last.  Slot layout: element (row, col) at float4
// (col / 4) * BM + row, so a warp's 32 rows are 512 contiguous bytes.
__device__ __forceinline__ bool sk_fixup(const Params& prm, SharedState2* ss, const WorkUnit& u, int etid, int half,
                                         int row, uint32_t t_row, int bn, uint32_t rank) {
  constexpr size_t SLOT_F4 = (size_t)BM * BN / 4;
  const int wcols = bn / 2, cb = half * wcols;
  float4* own = reinterpret_cast<float4*>(prm.sk_part) + (size_t)(2 * u.slot + (int)rank) * SLOT_F4;
  for (int p = 0; p < wcols; p += 16) {
    float v[16];
    tc::tmem_ld16(t_row + (uint32_t)(cb + p), v);
#pragma unroll
    for (int q = 0; q < 4; ++q)
      __stcg(own + (size_t)((cb + p) / 4 + q) * BM + row,
             make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
  }
  __threadfence();
  tc::named_bar_sync(3, EPI_THREADS);
  const int t = u.tile - prm.sk_first;
  if (etid == 0) {
    unsigned int* tk = prm.sk_ticket + 2 * t + (int)rank;
    const bool last = atomicAdd(tk, 1u) == (unsigned int)(u.npieces - 1);
    if (last) atomicExch(tk, 0u);                   // every piece has arrived: zero for the next launch
    ss->sk_last = last ? 1 : 0;
  }
  tc::named_bar_sync(3, EPI_THREADS);
  const bool last = *reinterpret_cast<volatile int*>(&ss->sk_last) != 0;
  if (!last) return false;
  __threadfence();
  // piece j of tail tile t is pair j * sk_tiles + t's; each 16-column chunk adds the pieces in K order, the
  // four loads of one piece in flight together (few registers beside the epilogue's)
  const float4* base = reinterpret_cast<const float4*>(prm.sk_part) + (size_t)rank * SLOT_F4;
  for (int p = 0; p < wcols; p += 16) {
    float sum[16];
    tc::tmem_ld16(t_row + (uint32_t)(cb + p), sum);     // this piece's own partial, used at its place below
    float mine[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) mine[e] = sum[e];
#pragma unroll 1
    for (int j = 0; j < u.npieces; ++j) {
      float v[16];
      if (j == u.piece) {
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = mine[e];
      } else {
        const float4* src = base + (size_t)(2 * (j * prm.sk_tiles + t)) * SLOT_F4 + (size_t)((cb + p) / 4) * BM + row;
        float4 x[4];
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) x[qq] = __ldcg(src + (size_t)qq * BM);
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          v[4 * qq] = x[qq].x; v[4 * qq + 1] = x[qq].y; v[4 * qq + 2] = x[qq].z; v[4 * qq + 3] = x[qq].w;
        }
      }
#pragma unroll
      for (int e = 0; e < 16; ++e) sum[e] = j == 0 ? v[e] : sum[e] + v[e];
    }
    tc::tmem_st16(t_row + (uint32_t)(cb + p), sum);
  }
  tc::tmem_wait_st();
  return true;
}

// ---- INT4 dequantisation on CTA pairs ----
constexpr int DQ_BAR = 7;                   // named barrier of the dequantising group
constexpr int DQ2_THREADS = 256;            // dequantising warps of an INT4 CTA-pair launch (half a row each)
constexpr int DQ_BATCH = 3;                 // stages per cluster-scope release (STAGES2 is a multiple)
static_assert(STAGES2 % DQ_BATCH == 0, "release batches must tile the ring");
__host__ __device__ constexpr int num_threads2(bool w4) { return 64 + EPI_THREADS + (w4 ? DQ2_THREADS : 0); }
__host__ __device__ constexpr int epi_base2(bool w4) { return 64 + (w4 ? DQ2_THREADS : 0); }
constexpr uint32_t W4_PACKED_BYTES = 4096;  // 128 rows x 32 packed bytes (64 weights) of one K-block
constexpr uint32_t W4_SCALE_BYTES = 2048;   // 128 rows x 8 fp16 scale groups (the box holding this K-block's)

// Eight INT4 elements of one word (element j in bits 4j..4j+3, 4-bit two's complement) times the scale s,
// in K order as 8 bf16 (one 16-byte granule).  With v = q + 8 (the nibble XOR 8), a byte permute puts the
// byte of elements (2b, 2b+1) into bits 8..15 under the exponent of 2^15; masking leaves the fp32 values
// 32768 + v_lo and 32768 + 16 v_hi exactly.  One packed FMA then gives (32768 + v_lo) s - 32776 s = q_lo s
// and (32768 + 16 v_hi)(s / 16) - 2056 s = q_hi s exactly -- every product and offset has at most 24
// significant bits -- and the conversion rounds both to bf16 once.
__device__ __forceinline__ uint4 dequant8_exact(uint32_t w, float s, float off_lo, float s16, float off_hi) {
  const uint32_t x = w ^ 0x88888888u;
  uint32_t out[4];
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const uint32_t r = __byte_perm(x, 0x47000000u, 0x7504u | ((uint32_t)b << 4));   // 0x47 00 byte_b 00
    const float2 q = ffma2(make_float2(__uint_as_float(r & 0xFF000F00u), __uint_as_float(r & 0xFF00F000u)),
                           make_float2(s, s16), make_float2(off_lo, off_hi));
    const __nv_bfloat162 h = __floats2bfloat162_rn(q.x, q.y);
    out[b] = *reinterpret_cast<const uint32_t*>(&h);
  }
  return make_uint4(out[0], out[1], out[2], out[3]);
}

// Half `hf` (granules 4 hf .. 4 hf + 3) of row `row` of the stage's 128-byte-swizzled B half, from 16
// packed bytes and the row's scale.
__device__ __forceinline__ void dq2_store_half(uint32_t btile, int row, int hf, uint4 q, float s) {
  const float off_lo = -32776.0f * s, s16 = 0.0625f * s, off_hi = -2056.0f * s;
  const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
  for (int c = 0; c < 4; ++c)
    tc::st_shared_v4(btile + sw128_off(row, 4 * hf + c), dequant8_exact(w[c], s, off_lo, s16, off_hi));
}

template <typename TO, int RT, int MODE, int AB_BF16, int SMODE = STAGE_NONE, bool W4 = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(num_threads2(W4), 1)
pair_tc2_kernel(const __grid_constant__ TmaSet tm, const Params prm) {
  static_assert(!W4 || (SMODE == STAGE_ALL && AB_BF16 == 1 && MODE != MODE_PLAIN),
                "INT4 CTA pairs: stacked rows with the whole low-rank term on the MMA, bf16 operands");
  constexpr int CW = MODE == MODE_GATED ? 8 : 16;   // epilogue chunk width (gated: two accumulators)
  const bool mismatch =
      (SMODE == STAGE_ALL && (prm.aug_mode != LOWRANK_ALL_ON_TC || prm.y_staged != STAGE_ALL)) ||
      ((SMODE == STAGE_MIRROR || SMODE == STAGE_MIRROR4) &&
       (prm.aug_mode != LOWRANK_C_ON_TC || prm.y_staged != SMODE || !prm.shared || prm.nb != 2)) ||
      (SMODE == STAGE_MULTI4 && (prm.aug_mode != LOWRANK_C_ON_TC || prm.y_staged != SMODE || !prm.shared ||
                                 prm.nb < 2)) ||
      ((SMODE == STAGE_MIRROR4 || SMODE == STAGE_MULTI4) && MODE == MODE_GATED && prm.P2 != prm.P) ||
      (SMODE == STAGE_LOSS && (MODE != MODE_PAIR || prm.aug_mode != LOWRANK_ALL_ON_TC || prm.y_staged != SMODE ||
                               prm.shared || prm.nb != 2 || prm.T % BM2 != 0));
  if (mismatch) {                                   // uniform: both CTAs of a pair leave
    pdl_wait();
    if (threadIdx.x == 0 && blockIdx.x == 0) record_error(prm.status, ZOACT_ERR_INVALID_ARG);
    return;
  }
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  float* tbl = reinterpret_cast<float*>(smem + STAGES2 * STAGE2_BYTES);
  SharedState2* ss = reinterpret_cast<SharedState2*>(tbl + TBL_FLOATS);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = tc2::cluster_rank();
  const bool leader = rank == 0;
  volatile int* abort_flag = &ss->abort_flag;

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES2; ++s) {
      // one producer arrival from each CTA (leader's copy is used), and with INT4 one from each CTA's
      // dequantising group
      tc::mbar_init(tc::smem_u32(&ss->full[s]), W4 ? 4 : 2);
      tc::mbar_init(tc::smem_u32(&ss->empty[s]), 1);
    }
    for (int b = 0; b < 2; ++b) {
      tc::mbar_init(tc::smem_u32(&ss->tmem_full[b]), 1);
      tc::mbar_init(tc::smem_u32(&ss->tmem_empty[b]), 2);   // one arrival per CTA (leader's copy is used)
    }
    if (W4)
      for (int st = 0; st < STAGES2; ++st) tc::mbar_init(tc::smem_u32(&ss->raw[st]), 1);
    tc::mbar_init(tc::smem_u32(&ss->drain), 1);
    tc::mbar_init(tc::smem_u32(&ss->tload[0]), 1);
    tc::mbar_init(tc::smem_u32(&ss->tload[1]), 1);
    ss->abort_flag = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tm.a);
    tc::prefetch_tmap(&tm.b);
    if (MODE == MODE_GATED) tc::prefetch_tmap(&tm.b2);
    if (W4) {
      tc::prefetch_tmap(&tm.s);
      if (MODE == MODE_GATED) tc::prefetch_tmap(&tm.s2);
    }
    if (prm.aug_kb > 0) {
      tc::prefetch_tmap(&tm.aa);
      tc::prefetch_tmap(&tm.ba);
      if (MODE == MODE_GATED) tc::prefetch_tmap(&tm.ba2);
    }
  }
  if (warp == 1) {
    tc2::tmem_alloc2(tc::smem_u32(&ss->tmem_base), TMEM_COLS);
    tc2::tmem_relinquish2();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc2::cluster_sync();                    // both CTAs' barriers exist before any remote arrival
  tc::tc_fence_after();
  const uint32_t tmem_base = ss->tmem_base;
  pdl_wait();                             // the previous kernel's outputs (X, P, operand tables) are visible
  pdl_trigger();

  const int num_m = prm.num_m, num_n = prm.num_n, num_k = prm.num_k;
  const int total_k = num_k + prm.aug_kb;   // main K-blocks, then the low-rank ones
  const int bn = MODE == MODE_GATED ? BN : prm.bn;
  const int bh = bn / 2;                  // W rows per CTA
  const uint32_t stage_tx = A_BYTES + bh * BK * 2;
  const int cluster_id = blockIdx.x >> 1, n_clusters = gridDim.x >> 1;

  if (warp == 0) {
    // ---------------- TMA producer (both CTAs) ----------------
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      WorkUnit u;
      for (int i = 0; ok && next_unit(prm, cluster_id, n_clusters, total_k, i, u); ++i) {
        int m_blk, n_blk;
        tile_coords(u.tile, num_m, num_n, m_blk, n_blk, prm.group_m);
        for (int kb = u.kb0; kb < u.kb1; ++kb) {
          if (!tc::mbar_wait(tc::smem_u32(&ss->empty[stage]), phase ^ 1u, abort_flag, prm.status)) { ok = false; break; }
          const uint32_t full_leader = tc2::map_to(tc::smem_u32(&ss->full[stage]), 0);
          const bool aug = kb >= num_k;
          // INT4: W's K-blocks come from the dequantising warps, only X (and the low-rank blocks) by TMA
          tc2::arrive_expect_tx_cluster(full_leader, (W4 && !aug) ? (uint32_t)A_BYTES : stage_tx);
          const uint32_t sa = tc::smem_u32(smem + stage * STAGE2_BYTES);
          const uint32_t sb = sa + A_BYTES;
          int kx = kb * BK, kxb = kb * BK, yb = 0;
          if (aug) aug_coords(prm, (int64_t)m_blk * BM2, BM2, kb - num_k, kx, kxb, yb);
          tc2::tma_load_2d_pair(sa, aug ? &tm.aa : &tm.a, kx, m_blk * BM2 + (int)rank * BM, full_leader);
          if (W4 && !aug) {
            // this CTA's packed rows and their scales into the B slot, for the dequantising warps
            const uint32_t raw = tc::smem_u32(&ss->raw[stage]);
            const bool up = MODE == MODE_GATED && !leader;
            const int y0 = MODE == MODE_GATED ? n_blk * (BN / 2) : n_blk * bn + (int)rank * bh;
            tc::mbar_arrive_expect_tx(raw, W4_PACKED_BYTES + W4_SCALE_BYTES);
            tc::tma_load_2d(sb, up ? &tm.b2 : &tm.b, kb * (BK / 2), y0, raw);
            tc::tma_load_2d(sb + W4_PACKED_BYTES, up ? &tm.s2 : &tm.s, ((kb * BK) / 128) & ~7, y0, raw);
          } else if (MODE == MODE_GATED)
            tc2::tma_load_2d_pair(sb, aug ? (leader ? &tm.ba : &tm.ba2) : (leader ? &tm.b : &tm.b2), kxb,
                                  yb + n_blk * (BN / 2), full_leader);
          else
            tc2::tma_load_2d_pair(sb, aug ? &tm.ba : &tm.b, kxb, yb + n_blk * bn + (int)rank * bh, full_leader);
          if (++stage == STAGES2) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        // our copies complete on the leader's barriers; give them time to land before the CTA winds down
        const uint64_t t0 = tc::global_timer_ns();
        while (tc::global_timer_ns() - t0 < 2000000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ---------------- MMA issuer (leader CTA) ----------------
    if (lane == 0 && leader) {
      const uint32_t idesc_main = tc::idesc_f16(BM2, bn, AB_BF16);
      const uint32_t idesc_aug = tc::idesc_f16(BM2, bn, 1);   // low-rank K-blocks are bf16
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      int local = 0;
      bool issued_any = false;
      WorkUnit u;
      for (int i = 0; ok && next_unit(prm, cluster_id, n_clusters, total_k, i, u); ++i, ++local) {
        const int buf = local & 1;
        const uint32_t acc_phase = (local >> 1) & 1;
        if (!tc::mbar_wait(tc::smem_u32(&ss->tmem_empty[buf]), acc_phase ^ 1u, abort_flag, prm.status)) { ok = false; break; }
        tc::tc_fence_after();
        const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
        for (int kb = u.kb0; kb < u.kb1; ++kb) {
          // INT4: the stage also carries the dequantising groups' cluster-scope release arrivals
          const bool got = W4 ? tc::mbar_wait_cl(tc::smem_u32(&ss->full[stage]), phase, abort_flag, prm.status)
                              : tc::mbar_wait(tc::smem_u32(&ss->full[stage]), phase, abort_flag, prm.status);
          if (!got) { ok = false; break; }
          tc::tc_fence_after();
          const uint32_t sa = tc::smem_u32(smem + stage * STAGE2_BYTES);
          const uint32_t sb = sa + A_BYTES;
          const uint32_t idesc = kb < num_k ? idesc_main : idesc_aug;
#pragma unroll
          for (int k = 0; k < BK / 16; ++k)
            tc2::mma2_f16(d_tmem, tc::sdesc_k_sw128(sa + k * 32), tc::sdesc_k_sw128(sb + k * 32), idesc,
                          (kb != u.kb0 || k != 0) ? 1u : 0u);
          tc2::commit2_both(tc::smem_u32(&ss->empty[stage]));    // frees the stage in both CTAs
          issued_any = true;
          if (++stage == STAGES2) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        tc2::commit2_both(tc::smem_u32(&ss->tmem_full[buf]));   // accumulator ready in both CTAs
      }
      if (issued_any) {
        tc2::commit2_own(tc::smem_u32(&ss->drain));
        tc::mbar_wait_drain(tc::smem_u32(&ss->drain), 0, 100000000ull);
      }
    }
  } else if (W4 && warp < 2 + DQ2_THREADS / 32) {
    // ---------------- INT4 dequantisation (warps 2..9, both CTAs) ----------------
    // Batches of DQ_BATCH stages: one thread waits for all of them (packed block landed, or the stage free
    // for a low-rank block the producer loads itself), the group reads every packed half-row, then
    // overwrites the slots with bf16, fences the async proxy, and one thread arrives on the leader's
    // stage barriers: the first with cluster-scope release (it orders the whole batch's writes), the
    // others relaxed -- the MMA issuer acquires the first before it looks at the others.
    const int dt = threadIdx.x - 64;
    const int row = dt >> 1, hf = dt & 1;           // this thread's half of one of the CTA's 128 W rows
    int stage = 0;
    uint32_t phase = 0;
    uint32_t raw_par = 0;                           // per stage: parity of its next raw phase (W blocks only)
    int i = 0, kb = 0;
    WorkUnit u;
    bool live = next_unit(prm, cluster_id, n_clusters, total_k, 0, u);
    if (live) kb = u.kb0;
    while (live) {
      int bst[DQ_BATCH], bkb[DQ_BATCH];
      bool bmain[DQ_BATCH];
      uint32_t bpar[DQ_BATCH], bphase[DQ_BATCH];
      int nb = 0;
#pragma unroll
      for (int b = 0; b < DQ_BATCH; ++b) {
        if (live) {
          bst[b] = stage; bkb[b] = kb; bmain[b] = kb < num_k;
          bpar[b] = (raw_par >> stage) & 1u; bphase[b] = phase;
          if (bmain[b]) raw_par ^= 1u << stage;
          if (++stage == STAGES2) { stage = 0; phase ^= 1u; }
          if (++kb >= u.kb1) {
            ++i;
            live = next_unit(prm, cluster_id, n_clusters, total_k, i, u);
            if (live) kb = u.kb0;
          }
          nb = b + 1;
        }
      }
      if (dt == 0) {
        bool ok = true;
        for (int b = 0; b < nb && ok; ++b)
          ok = bmain[b] ? tc::mbar_wait(tc::smem_u32(&ss->raw[bst[b]]), bpar[b], abort_flag, prm.status)
                        : tc::mbar_wait(tc::smem_u32(&ss->empty[bst[b]]), bphase[b] ^ 1u, abort_flag, prm.status);
        ss->dq_ok = ok ? 1 : 0;
      }
      tc::named_bar_sync(DQ_BAR, DQ2_THREADS);
      if (*reinterpret_cast<volatile int*>(&ss->dq_ok) == 0) break;
      uint4 q[DQ_BATCH];
      float sc[DQ_BATCH];
#pragma unroll
      for (int b = 0; b < DQ_BATCH; ++b) {
        if (b < nb && bmain[b]) {
          const uint32_t sb = tc::smem_u32(smem + bst[b] * STAGE2_BYTES + A_BYTES);
          q[b] = tc::ld_shared_v4(sb + (uint32_t)row * 32u + (uint32_t)hf * 16u);
          const int g = (bkb[b] * BK) / 128;                      // the scale group of this K-block
          const uint32_t sw = tc::ld_shared_b32(sb + W4_PACKED_BYTES + (uint32_t)row * 16u + (uint32_t)(g & 6) * 2u);
          const uint16_t sh = (uint16_t)((g & 1) ? (sw >> 16) : (sw & 0xFFFFu));
          __half hs;
          memcpy(&hs, &sh, 2);
          sc[b] = __half2float(hs);
        }
      }
      tc::named_bar_sync(DQ_BAR, DQ2_THREADS);     // every packed row is read: overwrite the slots
#pragma unroll
      for (int b = 0; b < DQ_BATCH; ++b)
        if (b < nb && bmain[b]) dq2_store_half(tc::smem_u32(smem + bst[b] * STAGE2_BYTES + A_BYTES), row, hf, q[b], sc[b]);
      tc::fence_proxy_async_smem();                 // generic writes -> the tensor cores' reads
      tc::named_bar_sync(DQ_BAR, DQ2_THREADS);     // the batch's half-tiles are written
      if (dt == 0) {
        tc2::arrive_release_cluster(tc2::map_to(tc::smem_u32(&ss->full[bst[0]]), 0));
        for (int b = 1; b < nb; ++b) tc2::arrive_relaxed_cluster(tc2::map_to(tc::smem_u32(&ss->full[bst[b]]), 0));
      }
    }
  } else {
    // ---------------- epilogue (warps 2..9, both CTAs; INT4: warps 10..17) ----------------
    const int etid = threadIdx.x - epi_base2(W4);
    const int half = etid >> 7;
    const int quad = warp & 3;
    const int row_in_tile = quad * 32 + lane;
    const uint32_t tmem_empty_leader0 = tc2::map_to(tc::smem_u32(&ss->tmem_empty[0]), 0);
    const uint32_t tmem_empty_leader1 = tc2::map_to(tc::smem_u32(&ss->tmem_empty[1]), 0);
    int local = 0;
    bool pending = false;                   // staged output: this thread has bulk stores in flight
    uint32_t tphase = 0;                    // fused loss: parity of this warpgroup's next target load
    CompSum lacc[2];                        // fused loss: running sums of the + and - rows
    bool aborted = false;
    WorkUnit u;
    for (int i = 0; next_unit(prm, cluster_id, n_clusters, total_k, i, u); ++i, ++local) {
      int m_blk, n_blk;
      tile_coords(u.tile, num_m, num_n, m_blk, n_blk, prm.group_m);
      const int buf = local & 1;
      const uint32_t acc_phase = (local >> 1) & 1;
      const int64_t row0 = (int64_t)m_blk * BM2 + (int64_t)rank * BM;
      const int64_t m = row0 + row_in_tile;
      const bool row_ok = m < prm.rows;
      const uint32_t t_row = tmem_base + ((uint32_t)(quad * 32) << 16) + (uint32_t)(buf * BN);
      bool ok = true;
      bool epi = true;
      if (u.npieces > 1) {
        // a tail piece: only the last one to finish runs the epilogue, on the summed accumulator
        ok = epi_wait_full(ss, buf, acc_phase, abort_flag, prm.status, etid);
        if (ok) {
          epi = sk_fixup(prm, ss, u, etid, half, row_in_tile, t_row, bn, rank);
          tc::tc_fence_before();
          tc::named_bar_sync(3, EPI_THREADS);       // the summed accumulator is in TMEM for every warp
          tc::tc_fence_after();
        }
      }
      if (!ok || !epi) {
      } else if constexpr (SMODE == STAGE_ALL)
        ok = epi_all_staged<TO, MODE>(prm, tm, ss, reinterpret_cast<uint8_t*>(tbl), etid, half, row_in_tile, row0,
                                      n_blk, bn, buf, acc_phase, t_row, abort_flag, pending);
      else if constexpr (SMODE == STAGE_MIRROR)
        ok = epi_mirror_staged<TO, RT, MODE>(prm, tm, ss, tbl, etid, half, row_in_tile, row0, m, row_ok, n_blk, bn,
                                             buf, acc_phase, t_row, abort_flag, pending);
      else if constexpr (SMODE == STAGE_MIRROR4)
        ok = epi_mirror4_staged<TO, RT, MODE>(prm, tm, ss, tbl, etid, half, quad, lane, row0, n_blk, bn, buf,
                                              acc_phase, t_row, abort_flag, pending);
      else if constexpr (SMODE == STAGE_MULTI4)
        ok = epi_multi4_staged<TO, RT, MODE>(prm, tm, ss, tbl, etid, half, quad, lane, row0, n_blk, bn, buf,
                                             acc_phase, t_row, abort_flag, pending);
      else if constexpr (SMODE == STAGE_LOSS)
        ok = epi_loss_staged<TO>(prm, tm, ss, reinterpret_cast<uint8_t*>(tbl), etid, half, row_in_tile, row0, n_blk,
                                 bn, buf, acc_phase, t_row, abort_flag, tphase, lacc);
      else
        ok = epi_pair_tile<TO, RT, MODE, CW>(prm, ss, tbl, etid, half, row0, m, row_ok, n_blk, bn, buf, acc_phase,
                                             t_row, abort_flag);
      if (!ok) { aborted = true; break; }
      tc::tc_fence_before();
      tc::named_bar_sync(3, EPI_THREADS);        // every epilogue thread of this CTA has read the tile
      if (etid == 0) tc2::arrive_cluster(buf ? tmem_empty_leader1 : tmem_empty_leader0);
    }
    if (pending) tc::bulk_wait0();           // the stores have read the staging buffers and completed
    if constexpr (SMODE == STAGE_LOSS) {
      // every epilogue thread gets here (the accumulator wait gives up uniformly); an aborted CTA adds no
      // partial, so the ticket stays short and the launch reports ZOACT_ERR_TIMEOUT with no loss written
      tc::named_bar_sync(3, EPI_THREADS);
      if (etid == 0) ss->epi_ok = (*abort_flag || aborted) ? 0 : 1;   // one reading, shared by all
      tc::named_bar_sync(3, EPI_THREADS);
      if (*reinterpret_cast<volatile int*>(&ss->epi_ok) != 0) {
        loss_finish(prm, lacc, reinterpret_cast<double*>(tbl), etid);
      } else if ((etid & 127) == 0) {               // give a target load still in flight time to land
        const uint64_t t0 = tc::global_timer_ns();
        while (tc::global_timer_ns() - t0 < 2000000ull) {
        }
      }
    }
  }

  tc::tc_fence_before();
  __syncthreads();
  tc2::cluster_sync();                    // the peer's MMAs and copies are done before TMEM and smem go away
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc2::tmem_dealloc2(tmem_base, TMEM_COLS);
  }
}

}  // namespace pairtc
}  // namespace zoact
