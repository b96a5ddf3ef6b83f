// Low-rank projection P = X U on the tensor cores (Section 3: the factor X V_r
// of the perturbed forward pass), for 16-bit X.
//
// The projection is HBM-bound on X (r is 1..32), so it must stream X at full
// bandwidth; CUDA-core FMAs cannot keep up at r = 16.  X is bf16/fp16 and
// exact in the MMA; U (fp32) is split into three 16-bit terms
// U = U0 + U1 + U2 (each the rounding of what is left), which keeps the
// product at fp32 accuracy.  The three terms are stacked as the rows of one
// K-major operand Ut [NB, d_in] (NB = 3 * RT padded to a multiple of 16), so a
// single tcgen05.mma 128 x NB x 16 per K-step produces all three partial
// products into TMEM; the epilogue adds them.
//
// Grid: (row blocks of 128, K-splits).  Per CTA: warp 0 streams X tiles
// (128 x 64) and Ut tiles (NB x 64) through a 4-stage TMA ring (two CTAs per
// SM; the grid is one wave of them), warp 1 issues
// the MMAs, then all four warps read the accumulator (one row per thread) and
// write the split's partial [rows, r] (or P itself without split).
#include "internal.h"
#include "tc_common.cuh"

namespace zoact {
namespace {

constexpr int PBM = 128, PBK = 64, PSTAGES = 4;
constexpr int P_A_BYTES = PBM * PBK * 2;

template <int NB>
__host__ __device__ constexpr int p_stage_bytes() { return P_A_BYTES + NB * PBK * 2; }
template <int NB>
__host__ __device__ constexpr int p_smem_bytes() { return 1024 + PSTAGES * p_stage_bytes<NB>() + 256; }

struct ProjShared {
  uint64_t full[PSTAGES];
  uint64_t empty[PSTAGES];
  uint64_t done;
  uint32_t tmem_base;
  int abort_flag;
  int ok;
};

// Ut: groups of RT ranks (one group for r <= 32; groups of 64 above), each NB rows:
// [0, RT) = U0^T, [RT, 2RT) = U1^T, [2RT, 3RT) = U2^T of the group's ranks, rest zero.
template <typename T16>
__global__ void split_u_kernel(const float* __restrict__ U, T16* __restrict__ Ut, int d_in, int r, int RT, int NB,
                               int groups) {
  const int64_t n = (int64_t)groups * NB * d_in;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int row_all = (int)(i / d_in);
    const int k = (int)(i % d_in);
    const int g = row_all / NB, row = row_all % NB;
    const int term = row / RT, j = g * RT + row % RT;
    float v = 0.f;
    if (term < 3 && j < r) {
      float rest = U[(int64_t)k * r + j];
      for (int t = 0; t <= term; ++t) {
        const float h = to_f32<T16>(from_f32<T16>(rest));
        if (t == term) v = h;
        rest -= h;
      }
    }
    Ut[i] = from_f32<T16>(v);
  }
}

template <int NB, int RT, int AB_BF16>
__global__ void __launch_bounds__(128, 1)
proj_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmU, float* __restrict__ out,
               int64_t rows, int r, int ld_out, int kb_per_split, int num_kb, int* status) {
  constexpr int STAGE = p_stage_bytes<NB>();
  constexpr uint32_t TCOLS = NB <= 32 ? 32 : (NB <= 64 ? 64 : (NB <= 128 ? 128 : 256));
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
  ProjShared* ss = reinterpret_cast<ProjShared*>(smem + PSTAGES * STAGE);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  volatile int* abort_flag = &ss->abort_flag;
  const int kb0 = blockIdx.y * kb_per_split;
  const int kb1 = min(num_kb, kb0 + kb_per_split);
  const int m0 = blockIdx.x * PBM;

  if (threadIdx.x == 0) {
    for (int s = 0; s < PSTAGES; ++s) {
      tc::mbar_init(tc::smem_u32(&ss->full[s]), 1);
      tc::mbar_init(tc::smem_u32(&ss->empty[s]), 1);
    }
    tc::mbar_init(tc::smem_u32(&ss->done), 1);
    ss->abort_flag = 0;
    tc::fence_mbar_init();
    tc::prefetch_tmap(&tmX);
    tc::prefetch_tmap(&tmU);
  }
  if (warp == 1) {
    tc::tmem_alloc(tc::smem_u32(&ss->tmem_base), TCOLS);
    tc::tmem_relinquish();
  }
  tc::tc_fence_before();
  __syncthreads();
  tc::tc_fence_after();
  const uint32_t tmem = ss->tmem_base;
  pdl_wait();                             // X (the previous kernel's output) is visible
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // ---- TMA producer ----
    uint32_t issued_mask = 0, issued_parity = 0;
    int stage = 0;
    uint32_t phase = 0;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (!tc::mbar_wait(tc::smem_u32(&ss->empty[stage]), phase ^ 1u, abort_flag, status)) break;
      const uint32_t full = tc::smem_u32(&ss->full[stage]);
      tc::mbar_arrive_expect_tx(full, STAGE);
      const uint32_t sa = tc::smem_u32(smem + stage * STAGE);
      tc::tma_load_2d(sa, &tmX, kb * PBK, m0, full);
      tc::tma_load_2d(sa + P_A_BYTES, &tmU, kb * PBK, 0, full);
      issued_mask |= 1u << stage;
      issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
      if (++stage == PSTAGES) { stage = 0; phase ^= 1u; }
    }
    if (*abort_flag)
      for (int s = 0; s < PSTAGES; ++s)
        if (issued_mask & (1u << s))
          tc::mbar_wait_drain(tc::smem_u32(&ss->full[s]), (issued_parity >> s) & 1u, 100000000ull);
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer ----
    constexpr uint32_t IDESC = tc::idesc_f16(PBM, NB, AB_BF16);
    int stage = 0;
    uint32_t phase = 0;
    bool any = false;
    for (int kb = kb0; kb < kb1; ++kb) {
      if (!tc::mbar_wait(tc::smem_u32(&ss->full[stage]), phase, abort_flag, status)) break;
      tc::tc_fence_after();
      const uint32_t sa = tc::smem_u32(smem + stage * STAGE);
      const uint32_t sb = sa + P_A_BYTES;
#pragma unroll
      for (int k = 0; k < PBK / 16; ++k)
        tc::mma_f16(tmem, tc::sdesc_k_sw128(sa + k * 32), tc::sdesc_k_sw128(sb + k * 32), IDESC,
                    (kb != kb0 || k != 0) ? 1u : 0u);
      tc::mma_commit(tc::smem_u32(&ss->empty[stage]));
      any = true;
      if (++stage == PSTAGES) { stage = 0; phase ^= 1u; }
    }
    if (any) {
      tc::mma_commit(tc::smem_u32(&ss->done));
    } else {
      tc::mbar_arrive(tc::smem_u32(&ss->done));   // empty K-range: nothing to wait for
    }
  }
  __syncwarp();

  // ---- epilogue: all four warps, one row per thread ----
  if (threadIdx.x == 0)
    ss->ok = tc::mbar_wait(tc::smem_u32(&ss->done), 0, abort_flag, status) ? 1 : 0;
  __syncthreads();
  tc::tc_fence_after();
  const bool ok = *reinterpret_cast<volatile int*>(&ss->ok) != 0 && kb1 > kb0;
  const int64_t m = m0 + threadIdx.x;
  // r valid ranks of this launch; split partials are [splits][rows][r], direct output rows have stride ld_out
  float* dst = out + (int64_t)blockIdx.y * rows * ld_out + m * ld_out;
  const uint32_t lane_base = tmem + ((uint32_t)(warp * 32) << 16);
  if constexpr (RT <= 8) {
    float acc[NB];
    if (ok) {
#pragma unroll
      for (int c = 0; c < NB; c += 16) tc::tmem_ld16(lane_base + (uint32_t)c, acc + c);
    } else {
#pragma unroll
      for (int c = 0; c < NB; ++c) acc[c] = 0.f;
    }
    if (m < rows) {
#pragma unroll
      for (int j = 0; j < RT; ++j)
        if (j < r) dst[j] = (acc[j] + acc[RT + j]) + acc[2 * RT + j];
    }
  } else {
    // 16 ranks at a time: their three terms are columns j, RT + j, 2 RT + j
#pragma unroll 1
    for (int jc = 0; jc < RT; jc += 16) {
      float t0[16], t1[16], t2[16];
      if (ok) {
        tc::tmem_ld16(lane_base + (uint32_t)jc, t0);
        tc::tmem_ld16(lane_base + (uint32_t)(RT + jc), t1);
        tc::tmem_ld16(lane_base + (uint32_t)(2 * RT + jc), t2);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) { t0[i] = 0.f; t1[i] = 0.f; t2[i] = 0.f; }
      }
      if (m < rows) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
          if (jc + i < r) dst[jc + i] = (t0[i] + t1[i]) + t2[i];
      }
    }
  }
  tc::tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc::tc_fence_after();
    tc::tmem_dealloc(tmem, TCOLS);
  }
}

// P[t, j0 + j] = sum over splits of part[split][t][j] (split order), j < rg; P rows have stride ldp.
__global__ void splitk_sum_kernel(const float* __restrict__ part, float* __restrict__ P, int64_t n, int splits, int rg,
                                  int ldp, int j0) {
  pdl_wait();
  pdl_trigger();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    float s = 0.f;
    for (int k = 0; k < splits; ++k) s += part[(int64_t)k * n + i];
    const int64_t t = i / rg;
    P[t * ldp + j0 + (i - t * rg)] = s;
  }
}

template <int NB, int RT, int AB>
int launch_one(Ctx* ctx, const CUtensorMap& mx, const CUtensorMap& mu, float* out, int64_t rows, int r, int ld_out,
               int kbps, int num_kb, dim3 grid) {
  auto kern = proj_tc_kernel<NB, RT, AB>;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, p_smem_bytes<NB>()));
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, grid, dim3(128), p_smem_bytes<NB>(), mx, mu, out, rows, r, ld_out, kbps,
                            num_kb, ctx->d_status));
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

template <int AB>
int dispatch(Ctx* ctx, int rt, const CUtensorMap& mx, const CUtensorMap& mu, float* out, int64_t rows, int r,
             int ld_out, int kbps, int num_kb, dim3 grid) {
  switch (rt) {
    case 4: return launch_one<16, 4, AB>(ctx, mx, mu, out, rows, r, ld_out, kbps, num_kb, grid);
    case 8: return launch_one<32, 8, AB>(ctx, mx, mu, out, rows, r, ld_out, kbps, num_kb, grid);
    case 16: return launch_one<48, 16, AB>(ctx, mx, mu, out, rows, r, ld_out, kbps, num_kb, grid);
    case 32: return launch_one<96, 32, AB>(ctx, mx, mu, out, rows, r, ld_out, kbps, num_kb, grid);
    default: return launch_one<192, 64, AB>(ctx, mx, mu, out, rows, r, ld_out, kbps, num_kb, grid);
  }
}

// ranks per group of the split basis (one group up to 32 ranks, groups of 64 above) and rows per group
int proj_rt(int r) { return r <= 4 ? 4 : r <= 8 ? 8 : r <= 16 ? 16 : r <= 32 ? 32 : 64; }
int proj_nb(int rt) { return rt == 4 ? 16 : rt == 8 ? 32 : rt == 16 ? 48 : rt == 32 ? 96 : 192; }

}  // namespace

int basis_tc_rows(int r) {
  const int rt = proj_rt(r);
  return proj_nb(rt) * ((r + rt - 1) / rt);
}

int launch_basis_prepare(Ctx* ctx, const float* U, int d_in, int r, int xdtype, void* Ut) {
  const int rt = proj_rt(r);
  const int nb = proj_nb(rt);
  const int groups = (r + rt - 1) / rt;
  const int64_t n = (int64_t)groups * nb * d_in;
  int64_t blocks = (n + 255) / 256;
  if (blocks > 8LL * ctx->sm_count) blocks = 8LL * ctx->sm_count;
  if (xdtype == ZOACT_DT_BF16)
    split_u_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, ctx->stream>>>(U, static_cast<__nv_bfloat16*>(Ut), d_in,
                                                                             r, rt, nb, groups);
  else
    split_u_kernel<__half><<<(unsigned)blocks, 256, 0, ctx->stream>>>(U, static_cast<__half*>(Ut), d_in, r, rt, nb,
                                                                      groups);
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

int launch_lowrank_proj_tc(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U, int r,
                           float* P) {
  if (rows <= 0) return ZOACT_OK;
  // Ut: the split basis, [nb, d_in] 16-bit, rebuilt on every call (U is small)
  void* Ut = scratch(ctx, SLOT_UT, (size_t)basis_tc_rows(r) * d_in * 2);
  if (!Ut) return ZOACT_ERR_NOMEM;
  const int st = launch_basis_prepare(ctx, U, d_in, r, xdtype, Ut);
  if (st) return st;
  return launch_lowrank_proj_tc_prepared(ctx, X, xdtype, rows, d_in, Ut, r, P);
}

int launch_lowrank_proj_tc_prepared(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const void* Ut,
                                    int r, float* P) {
  if (rows <= 0) return ZOACT_OK;
  const int rt = proj_rt(r);
  const int nb = proj_nb(rt);
  const int groups = (r + rt - 1) / rt;
  CUtensorMap mx;
  int st = encode_tmap_2d_16bit(&mx, X, xdtype, rows, d_in, PBM);
  if (st) return st;
  const int num_kb = (d_in + PBK - 1) / PBK;
  const int64_t row_blocks = (rows + PBM - 1) / PBM;
  // K-splits so the grid is one wave of two CTAs per SM, at least 2 K-blocks per split
  int splits = (int)((2LL * ctx->sm_count) / row_blocks);
  if (splits > num_kb / 2) splits = num_kb / 2;
  if (splits < 1) splits = 1;
  const int kbps = (num_kb + splits - 1) / splits;
  splits = (num_kb + kbps - 1) / kbps;
  // one launch per group of ranks (X is re-read per group; a single group up to r = 32)
  for (int g = 0; g < groups; ++g) {
    const int j0 = g * rt, rg = r - j0 < rt ? r - j0 : rt;
    CUtensorMap mu;
    st = encode_tmap_2d_16bit(&mu, static_cast<const uint8_t*>(Ut) + (size_t)g * nb * d_in * 2, xdtype, nb, d_in, nb);
    if (st) return st;
    float* out = P + j0;
    int ld_out = r;
    if (splits > 1) {
      out = static_cast<float*>(scratch(ctx, SLOT_SPLITK, (size_t)splits * rows * rg * sizeof(float)));
      if (!out) return ZOACT_ERR_NOMEM;
      ld_out = rg;
    }
    const dim3 grid((unsigned)row_blocks, (unsigned)splits);
    st = xdtype == ZOACT_DT_BF16 ? dispatch<1>(ctx, rt, mx, mu, out, rows, rg, ld_out, kbps, num_kb, grid)
                                 : dispatch<0>(ctx, rt, mx, mu, out, rows, rg, ld_out, kbps, num_kb, grid);
    if (st) return st;
    if (splits > 1) {
      const int64_t n = rows * rg;
      int64_t blocks = (n + 255) / 256;
      if (blocks > 4LL * ctx->sm_count) blocks = 4LL * ctx->sm_count;
      ZOACT_CUDA_TRY(launch_pdl(ctx, splitk_sum_kernel, dim3((unsigned)blocks), dim3(256), 0, out, P, n, splits, rg,
                                r, j0));
      ++ctx->n_launch;
      ZOACT_CHECK_LAUNCH();
    }
  }
  return ZOACT_OK;
}

}  // namespace zoact
