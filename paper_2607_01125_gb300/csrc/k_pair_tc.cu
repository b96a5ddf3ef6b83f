// Host side of the tensor-core pair forward: tensor-map encoding, argument
// checks and dispatch to the per-dtype instantiations of pair_tc_kernel.
#include <cstdlib>
#include <cstring>
#include <mutex>

#include "pair_tc_kernel.cuh"

namespace zoact {

namespace pairtc {
int dispatch_bf16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p);
int dispatch_fp16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p);
int dispatch_w4(Ctx* ctx, int mode, int rt, int ydtype, const CUtensorMap& a, const Params& p);
int dispatch2_bf16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p);
int dispatch2_fp16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p);
int dispatch2_w4(Ctx* ctx, int mode, int ydtype, const TmaSet& tm, const Params& p);
}  // namespace pairtc

namespace {

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

int rank_template(int r) { return r <= 4 ? 4 : r <= 8 ? 8 : r <= 16 ? 16 : 32; }

// N-tile width of the one-CTA kernel for a rows x n output on sm_count persistent
// CTAs: the width whose tiles fill the last wave best (useful outputs / (waves *
// SMs * tile size)); ties go to the wider tile, which reuses each A tile for more
// columns.  Widths below 192 measured slower per FLOP than this model predicts, so
// they are not tried.  (CTA pairs always take 256: see launch_pair_tc.)
int choose_bn(int64_t rows, int64_t n, int sm_count, int bm = pairtc::BM) {
  static const int cand[] = {256, 224, 192};
  const int64_t num_m = (rows + bm - 1) / bm;
  int best = 256;
  double best_eff = -1.0;
  for (int bn : cand) {
    const int64_t tiles = num_m * ((n + bn - 1) / bn);
    const int64_t waves = (tiles + sm_count - 1) / sm_count;
    const double eff = (double)rows * (double)n / ((double)waves * sm_count * bm * bn);
    if (eff > best_eff * 1.01) {
      best_eff = eff;
      best = bn;
    }
  }
  return best;
}

}  // namespace

int encode_tmap_2d_16bit(CUtensorMap* map, const void* base, int dtype, int64_t rows, int64_t cols, int box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return ZOACT_ERR_CUDA;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  const CUtensorMapDataType dt =
      dtype == ZOACT_DT_FP16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const CUresult res = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? ZOACT_OK : ZOACT_ERR_INVALID_ARG;
}

// Unswizzled boxes of 8- or 16-bit integers (INT4 packed weights, fp16 scales read as raw bits).
int encode_tmap_2d_int(CUtensorMap* map, const void* base, int elem_bytes, int64_t rows, int64_t cols, int box_cols,
                       int box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return ZOACT_ERR_CUDA;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * elem_bytes};
  const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  const CUtensorMapDataType dt = elem_bytes == 1 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16;
  const CUresult res = fn(map, dt, 2, const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? ZOACT_OK : ZOACT_ERR_INVALID_ARG;
}

int encode_tmap_store(CUtensorMap* map, void* base, int ydtype, int64_t rows, int64_t cols, int box_cols,
                      int box_rows, bool swizzle128) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return ZOACT_ERR_CUDA;
  const size_t es = dtype_size(ydtype);
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * es};
  const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1u, 1u};
  const CUtensorMapDataType dt = ydtype == ZOACT_DT_FP32   ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                 : ydtype == ZOACT_DT_FP16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                                           : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const CUresult res = fn(map, dt, 2, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          swizzle128 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
                          CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? ZOACT_OK : ZOACT_ERR_INVALID_ARG;
}

int encode_tmap_store3(CUtensorMap* map, void* base, int ydtype, int64_t nb, int64_t rows, int64_t cols,
                       int box_cols, int box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return ZOACT_ERR_CUDA;
  const size_t es = dtype_size(ydtype);
  const cuuint64_t dims[3] = {(cuuint64_t)cols, (cuuint64_t)rows, (cuuint64_t)nb};
  const cuuint64_t strides[2] = {(cuuint64_t)cols * es, (cuuint64_t)rows * cols * es};
  const cuuint32_t box[3] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows, 1u};
  const cuuint32_t estr[3] = {1u, 1u, 1u};
  const CUtensorMapDataType dt = ydtype == ZOACT_DT_FP32   ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                 : ydtype == ZOACT_DT_FP16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                                           : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
  const CUresult res = fn(map, dt, 3, base, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? ZOACT_OK : ZOACT_ERR_INVALID_ARG;
}

bool pair_rowscale_supported(const Ctx* ctx, int64_t rows, int shared, int xdtype, int wtype, int nb) {
  using namespace pairtc;
  if (!ctx->may_allocate || shared || rows < 2 * BM || nb < 1) return false;
  if (xdtype != ZOACT_DT_BF16 && xdtype != ZOACT_DT_FP16) return false;
  const char* sel = std::getenv("ZOACT_PAIR_KERNEL");
  const char* lsel = std::getenv("ZOACT_LOWRANK");
  if ((sel && std::strcmp(sel, "1cta") == 0) || (lsel && std::strcmp(lsel, "epilogue") == 0)) return false;
  if (wtype == ZOACT_DT_INT4_G128) {
    // INT4 reaches the CTA-pair kernel expanded to bf16 (from 1024 rows, or ZOACT_INT4=staged) or with
    // ZOACT_INT4=kernel; below 1024 rows the one-CTA kernel dequantises it
    const char* isel = std::getenv("ZOACT_INT4");
    return rows >= INT4_STAGED_MIN_ROWS || (isel && (std::strcmp(isel, "staged") == 0 || std::strcmp(isel, "kernel") == 0));
  }
  return true;
}

int launch_pair_tc(Ctx* ctx, const PairArgs& a) {
  using namespace pairtc;
  // ranks above 32 have no epilogue tables: the low-rank term must ride the MMA, which needs stacked rows
  const bool big_r = a.r > 32;
  if (big_r && !ctx->may_allocate) return ZOACT_ERR_UNSUPPORTED;
  if (big_r && a.shared) {
    // a shared input is copied once per evaluation block (and its projection with it), then run stacked
    const size_t x_bytes = (size_t)a.T * a.d_in * dtype_size(a.xdtype);
    const size_t p_bytes = (size_t)a.T * a.r * sizeof(float);
    const int np = a.W2 && a.P2 != a.P ? 2 : 1;
    uint8_t* buf = static_cast<uint8_t*>(scratch(ctx, SLOT_STACKED_X, a.nb * (x_bytes + np * p_bytes) + 1024));
    if (!buf) return ZOACT_ERR_NOMEM;
    uint8_t* xs = buf;
    float* ps = reinterpret_cast<float*>(buf + (a.nb * x_bytes + 255) / 256 * 256);
    float* ps2 = np == 2 ? ps + (size_t)a.nb * a.T * a.r : ps;
    for (int b = 0; b < a.nb; ++b) {
      ZOACT_CUDA_TRY(cudaMemcpyAsync(xs + b * x_bytes, a.X, x_bytes, cudaMemcpyDeviceToDevice, ctx->stream));
      ZOACT_CUDA_TRY(cudaMemcpyAsync(ps + (size_t)b * a.T * a.r, a.P, p_bytes, cudaMemcpyDeviceToDevice, ctx->stream));
      if (np == 2)
        ZOACT_CUDA_TRY(cudaMemcpyAsync(ps2 + (size_t)b * a.T * a.r, a.P2, p_bytes, cudaMemcpyDeviceToDevice,
                                       ctx->stream));
    }
    PairArgs b = a;
    b.X = xs;
    b.P = ps;
    b.P2 = a.W2 ? ps2 : nullptr;
    b.shared = 0;
    b.rows = (int64_t)a.nb * a.T;
    return launch_pair_tc(ctx, b);
  }
  // INT4 weights.  Below 1024 rows the one-CTA kernel dequantises in the kernel; from 1024 rows W is expanded
  // to bf16 once per call and the bf16 kernel runs (the default: measured faster, see pair_tc2_kernel.cuh).
  // ZOACT_INT4=kernel runs stacked rows from 256 on the CTA-pair kernel with its own dequantising warps
  // (bf16 or fp32 output, d_in a multiple of 1024); ZOACT_INT4=staged expands W at every row count.
  const char* sel = std::getenv("ZOACT_PAIR_KERNEL");
  const bool one_cta = sel && std::strcmp(sel, "1cta") == 0;
  const char* lsel = std::getenv("ZOACT_LOWRANK");
  const bool lr_epi = lsel && std::strcmp(lsel, "epilogue") == 0;
  const char* isel = std::getenv("ZOACT_INT4");
  const bool int4_staged = isel && std::strcmp(isel, "staged") == 0;   // expansion at any row count
  const bool int4_kernel = isel && std::strcmp(isel, "kernel") == 0;   // CTA-pair in-kernel dequantisation
  // (the scales' tensor map wants rows of a multiple of 16 bytes: d_in a multiple of 1024)
  auto al16 = [](const void* q) { return q == nullptr || ((uintptr_t)q & 15u) == 0; };
  const bool w4_two = a.wtype == ZOACT_DT_INT4_G128 && !big_r && ctx->may_allocate && !a.shared && !a.fuse_loss &&
                      a.rows >= 2 * BM && a.xdtype == ZOACT_DT_BF16 && a.d_in % 1024 == 0 &&
                      al16(a.w_scales) && al16(a.w_scales2) &&
                      (a.ydtype == ZOACT_DT_BF16 || a.ydtype == ZOACT_DT_FP32) && !one_cta && !lr_epi &&
                      int4_kernel;
  if (a.wtype == ZOACT_DT_INT4_G128 && !w4_two &&
      (a.rows >= INT4_STAGED_MIN_ROWS || big_r || (int4_staged && ctx->may_allocate))) {
    // staged INT4: expand W (and W2) to bf16 in context scratch, then the bf16 kernel (timed together)
    const size_t bytes = (size_t)a.d_out * a.d_in * 2;
    void* wb = scratch(ctx, SLOT_WDQ0, bytes);
    if (!wb) return ZOACT_ERR_NOMEM;
    int st = timing_begin(ctx);
    if (st) return st;
    st = launch_dequant_int4(ctx, a.W, a.w_scales, wb, a.d_out, a.d_in);
    if (st) return st;
    PairArgs b = a;
    b.W = wb;
    b.w_scales = nullptr;
    b.wtype = ZOACT_DT_BF16;
    if (a.W2) {
      void* wb2 = scratch(ctx, SLOT_WDQ1, bytes);
      if (!wb2) return ZOACT_ERR_NOMEM;
      st = launch_dequant_int4(ctx, a.W2, a.w_scales2, wb2, a.d_out, a.d_in);
      if (st) return st;
      b.W2 = wb2;
      b.w_scales2 = nullptr;
    }
    st = launch_pair_tc(ctx, b);
    if (st) return st;
    return timing_end(ctx);
  }
  if (a.xdtype != ZOACT_DT_BF16 && a.xdtype != ZOACT_DT_FP16) return ZOACT_ERR_UNSUPPORTED;
  const bool w4 = a.wtype == ZOACT_DT_INT4_G128;
  if (w4 ? a.xdtype != ZOACT_DT_BF16 : a.wtype != a.xdtype) return ZOACT_ERR_UNSUPPORTED;
  if (a.ydtype != a.xdtype && a.ydtype != ZOACT_DT_FP32) return ZOACT_ERR_UNSUPPORTED;
  const bool gated = a.W2 != nullptr;
  // epilogue-table rank template (set below: the smallest one when the tables go unused)
  int rt = rank_template(a.r);
  if (a.rows <= 0) return ZOACT_OK;
  TmaSet tm;
  int st = encode_tmap_2d_16bit(&tm.a, a.X, a.xdtype, a.rows, a.d_in, BM);
  if (st) return st;
  // CTA pairs (256-row tiles) once there are enough rows to fill them (INT4: where w4_two allows)
  const bool two = (w4 ? w4_two : a.rows >= 2 * BM && !one_cta);
  // CTA pairs: always 256-wide tiles.  A 256 x bn x 16 MMA measured the same time for bn = 192, 224 and 256, so
  // a tile costs the same at any of these widths and the widest needs the fewest waves (the Llama-3-8B MLP step:
  // 0.645 ms at 256 and at 224, 0.709 at 192; the OPT stack: 145.7 ms at 256, 149.1 at 224).
  const int bn = (gated || w4 || two) ? BN : choose_bn(a.rows, a.d_out, ctx->sm_count);
  const int b_box = gated ? BN / 2 : (two ? bn / 2 : bn);
  tm.s = tm.s2 = tm.a;
  if (w4 && two) {
    // packed rows and their scales by TMA, dequantised in shared memory by the kernel's own warps
    st = encode_tmap_2d_int(&tm.b, a.W, 1, a.d_out, a.d_in / 2, BK / 2, BM);
    if (st) return st;
    st = encode_tmap_2d_int(&tm.s, a.w_scales, 2, a.d_out, a.d_in / 128, 8, BM);
    if (st) return st;
    tm.b2 = tm.b;
    tm.s2 = tm.s;
    if (gated) {
      st = encode_tmap_2d_int(&tm.b2, a.W2, 1, a.d_out, a.d_in / 2, BK / 2, BM);
      if (st) return st;
      st = encode_tmap_2d_int(&tm.s2, a.w_scales2, 2, a.d_out, a.d_in / 128, 8, BM);
      if (st) return st;
    }
  } else if (w4) {
    tm.b = tm.b2 = tm.a;                 // W arrives through the dequantising warps, not TMA
  } else {
    st = encode_tmap_2d_16bit(&tm.b, a.W, a.wtype, a.d_out, a.d_in, b_box);
    if (st) return st;
    if (gated) {
      st = encode_tmap_2d_16bit(&tm.b2, a.W2, a.wtype, a.d_out, a.d_in, BN / 2);
      if (st) return st;
    } else {
      tm.b2 = tm.b;
    }
  }
  // low-rank term: on the tensor cores where the context may hold the split operands (INT4: on CTA pairs)
  int lmode = LOWRANK_EPILOGUE;
  const bool distinct = gated && a.P2 != a.P;
  int slots = 1;
  if ((!w4 || two) && ctx->may_allocate && (big_r || !lr_epi)) {
    // stacked rows: the whole term on the tensor cores -- one K slot when every tile lies in one evaluation
    // block, else S slots (block index mod S) with S the most blocks a tile can span; shared inputs keep
    // +-Z p in the epilogue (C p on the tensor cores)
    const int64_t tile_rows = two ? 2 * BM : BM;
    lmode = LOWRANK_C_ON_TC;
    if (!a.shared) {
      lmode = LOWRANK_ALL_ON_TC;
      if (a.T % tile_rows != 0) {
        const int64_t span = (tile_rows - 1) / a.T + 2;
        slots = (int)(span < a.nb ? span : a.nb);
      }
    }
  }
  if (big_r && lmode != LOWRANK_ALL_ON_TC) return ZOACT_ERR_UNSUPPORTED;
  // layers run as one: the kernel must read the low-rank term only from the operand tables, which take each
  // layer's coefficients and Philox stream (callers check pair_rowscale_supported before launching anything)
  if (a.nseg > 1 && (gated || a.fuse_loss || lmode != LOWRANK_ALL_ON_TC)) return ZOACT_ERR_UNSUPPORTED;
  if (lmode == LOWRANK_ALL_ON_TC) rt = 4;   // whole term on the tensor cores: no epilogue tables
  // the fused loss needs CTA pairs whose 128-row halves each lie in one sign block, whole term on the MMA
  if (a.fuse_loss && !(two && !gated && lmode == LOWRANK_ALL_ON_TC && a.nb == 2 && !a.shared &&
                       a.T % (2 * BM) == 0 && dtype_size(a.ydtype) == 2))
    return ZOACT_ERR_UNSUPPORTED;
  const int ka = aug_cols(a.r);
  const int ka_tot = distinct ? 2 * ka : ka;
  tm.aa = tm.a; tm.ba = tm.b; tm.ba2 = tm.b2;
  int64_t aug_block_rows = 0;
  // C on the tensor cores: the distinct queries of the perturbed blocks, each one transposed Z table
  uint64_t zq_list[ZOACT_MAX_EVAL_BLOCKS];
  int zq_of[ZOACT_MAX_EVAL_BLOCKS];
  int nzq = 0;
  for (int b = 0; b < a.nb; ++b) {
    zq_of[b] = -1;
    if (lmode != LOWRANK_C_ON_TC || a.coef[b] == 0.f) continue;
    for (int i = 0; i < nzq; ++i)
      if (zq_list[i] == a.qry[b]) zq_of[b] = i;
    if (zq_of[b] < 0) {
      zq_list[nzq] = a.qry[b];
      zq_of[b] = nzq++;
    }
  }
  float* zt = nullptr;
  float* zt2 = nullptr;
  if (lmode != LOWRANK_EPILOGUE) {
    const int64_t nbB = lmode == LOWRANK_ALL_ON_TC ? a.nb : 1;
    const size_t a_bytes = (size_t)a.rows * slots * ka_tot * 2;
    const size_t b_bytes = (size_t)nbB * a.d_out * ka_tot * 2;
    uint8_t* abuf = static_cast<uint8_t*>(scratch(ctx, SLOT_AUG_A, a_bytes));
    uint8_t* bbuf = static_cast<uint8_t*>(scratch(ctx, SLOT_AUG_B, (gated ? 2 : 1) * b_bytes));
    if (!abuf || !bbuf) return ZOACT_ERR_NOMEM;
    uint8_t* bbuf2 = gated ? bbuf + b_bytes : nullptr;
    if (nzq > 0) {
      const size_t z_floats = (size_t)nzq * a.r * a.d_out;
      zt = static_cast<float*>(scratch(ctx, SLOT_AUG_Z, (gated ? 2 : 1) * z_floats * sizeof(float)));
      if (!zt) return ZOACT_ERR_NOMEM;
      zt2 = gated ? zt + z_floats : nullptr;
    }
    st = launch_aug_prep(ctx, a, lmode, ka, distinct ? 1 : 0, slots, abuf, bbuf, bbuf2, zt, zt2, zq_list, nzq);
    if (st) return st;
    st = encode_tmap_2d_16bit(&tm.aa, abuf, ZOACT_DT_BF16, a.rows, (int64_t)slots * ka_tot, BM);
    if (st) return st;
    st = encode_tmap_2d_16bit(&tm.ba, bbuf, ZOACT_DT_BF16, nbB * a.d_out, ka_tot, b_box);
    if (st) return st;
    if (gated) {
      st = encode_tmap_2d_16bit(&tm.ba2, bbuf2, ZOACT_DT_BF16, nbB * a.d_out, ka_tot, b_box);
      if (st) return st;
    } else {
      tm.ba2 = tm.ba;
    }
    aug_block_rows = a.d_out;
  }
  Params p{};
  p.P = a.P; p.C = a.C; p.P2 = a.P2; p.C2 = a.C2; p.Y = a.Y;
  p.rows = a.rows; p.T = a.T; p.d_in = a.d_in; p.d_out = a.d_out; p.r = a.r;
  p.shared = a.shared; p.act = a.act; p.seed = a.seed;
  p.nb = a.nb;
  for (int b = 0; b < ZOACT_MAX_EVAL_BLOCKS; ++b) {
    p.coef[b] = b < a.nb ? a.coef[b] : 0.f;
    p.qry[b] = b < a.nb ? a.qry[b] : 0;
  }
  p.layer_id = a.layer_id; p.layer_id2 = a.layer_id2;
  p.num_m = (int)((a.rows + BM - 1) / BM);
  p.bn = bn;
  p.num_n = gated ? (a.d_out + BN / 2 - 1) / (BN / 2) : (a.d_out + bn - 1) / bn;
  p.num_k = (a.d_in + BK - 1) / BK;
  if (two) p.num_m = (int)((a.rows + 2 * BM - 1) / (2 * BM));
  p.num_tiles = p.num_m * p.num_n;
  p.ldy = a.d_out;
  p.aug_mode = lmode;
  if (two) {
    // CTA pairs: M-groups as large as keep the group's X rows within ~48 MB of L2 (at least GROUP_M): each W
    // panel is then read once per group -- with d_in = 4096 and 32 M-tiles, twice instead of four times
    const double x_group = 2.0 * BM * (double)a.d_in * (double)dtype_size(a.xdtype);
    int gm = GROUP_M;
    while (2 * gm <= p.num_m && 2 * gm * x_group <= 48e6) gm *= 2;
    const char* gsel = std::getenv("ZOACT_GROUP_M");   // comparisons
    if (gsel && std::atoi(gsel) > 0) gm = std::atoi(gsel);
    p.group_m = gm;
  }
  // CTA pairs write Y through staged bulk stores when the whole term is on the MMA, and for the two signs
  // of one query on a shared input with 16-bit outputs (one store map per sign: rows [0, T) and [T, 2T))
  tm.y = tm.y16 = tm.a;
  p.y_staged = STAGE_NONE;
  const int es = (int)dtype_size(a.ydtype);
  if (a.fuse_loss) {
    // no output: the target comes through tm.y / tm.y16 into the staging buffers
    p.y_staged = STAGE_LOSS;
    p.has_target = a.target ? 1 : 0;
    p.loss_eps = a.loss_eps;
    p.loss_out = a.loss_out;
    p.loss_ticket = ctx->d_tickets + 4;
    p.loss_part = static_cast<double*>(scratch(ctx, SLOT_PARTIALS, (size_t)ctx->sm_count * 2 * sizeof(double)));
    if (!p.loss_part) return ZOACT_ERR_NOMEM;
    if (a.target) {
      void* t0 = const_cast<void*>(a.target);
      st = encode_tmap_store(&tm.y, t0, a.ydtype, a.T, a.d_out, 128 / es, BM, true);
      if (st) return st;
      st = encode_tmap_store(&tm.y16, t0, a.ydtype, a.T, a.d_out, 16, BM, false);
      if (st) return st;
    }
  } else if (two && lmode == LOWRANK_ALL_ON_TC && rt == 4) {
    st = encode_tmap_store(&tm.y, a.Y, a.ydtype, a.rows, a.d_out, 128 / es, BM, true);
    if (st) return st;
    st = encode_tmap_store(&tm.y16, a.Y, a.ydtype, a.rows, a.d_out, 16, BM, false);
    if (st) return st;
    p.y_staged = STAGE_ALL;
  } else if (two && lmode == LOWRANK_C_ON_TC && a.shared && a.nb == 2 && es == 2 && a.qry[0] == a.qry[1] &&
             a.coef[1] == -a.coef[0] && a.coef[0] != 0.f) {
    uint8_t* y0 = static_cast<uint8_t*>(a.Y);
    st = encode_tmap_store(&tm.y, y0, a.ydtype, a.T, a.d_out, 16, BM, false);
    if (st) return st;
    st = encode_tmap_store(&tm.y16, y0 + (size_t)a.T * a.d_out * es, a.ydtype, a.T, a.d_out, 16, BM, false);
    if (st) return st;
    // four rows per thread where the projections fit in registers (rank tile <= 16, one P for gate and up)
    p.y_staged = (rt <= 16 && (!gated || a.P2 == a.P)) ? STAGE_MIRROR4 : STAGE_MIRROR;
  } else if (two && lmode == LOWRANK_C_ON_TC && a.shared && a.nb >= 2 && es == 2 && rt <= 16 &&
             (!gated || a.P2 == a.P)) {
    // other evaluation blocks on a shared input (the one-sided q-query estimator): one 3-D store map
    st = encode_tmap_store3(&tm.y, a.Y, a.ydtype, a.nb, a.T, a.d_out, 16, BM);
    if (st) return st;
    tm.y16 = tm.y;
    p.y_staged = STAGE_MULTI4;
  }
  // row scales ride the staged epilogue of stacked rows only (pair_rowscale_supported screens the rest first)
  if ((a.in_scale || a.out_sumsq) && p.y_staged != STAGE_ALL) return ZOACT_ERR_UNSUPPORTED;
  p.in_scale = a.in_scale;
  p.out_sumsq = a.out_sumsq;
  p.aug_kb = lmode == LOWRANK_EPILOGUE ? 0 : slots * ka_tot / BK;
  p.aug_kb_slot = ka_tot / BK;
  p.aug_slots = slots;
  p.aug_block_rows = aug_block_rows;
  p.Zt = zt;
  p.Zt2 = zt2;
  p.zt_qstride = (int64_t)a.r * a.d_out;
  for (int b = 0; b < ZOACT_MAX_EVAL_BLOCKS; ++b) p.zq[b] = b < a.nb ? zq_of[b] : -1;
  // (al16: 16-byte alignment, defined above)
  p.vec_ok = al16(a.C) && al16(a.C2) && al16(a.P) && al16(a.P2);
  // Split tail: when the last wave of whole tiles would leave at least half of the pairs idle, each of its tiles
  // is cut into S = pairs / tail-tiles (<= 4) equal K ranges, one per pair, and the last piece of a tile to finish
  // adds the partials; the tail then takes 1/S of a tile's time.  ZOACT_SPLIT_TAIL=0 keeps whole tiles.
  const char* sksel = std::getenv("ZOACT_SPLIT_TAIL");
  if (two && ctx->may_allocate && !(sksel && sksel[0] == '0')) {
    const int pairs = ctx->sm_count / 2;
    const int rem = p.num_tiles % pairs;
    const int total_k = p.num_k + p.aug_kb;
    int split = rem > 0 ? pairs / rem : 0;
    if (split > 4) split = 4;
    if (split >= 2 && total_k / split >= 4) {
      p.sk_first = p.num_tiles - rem;
      p.sk_tiles = rem;
      p.sk_split = split;
      p.sk_part = static_cast<float*>(scratch(ctx, SLOT_SK_PART, (size_t)pairs * 2 * BM * BN * sizeof(float)));
      p.sk_ticket =
          static_cast<unsigned int*>(scratch_zeroed(ctx, SLOT_SK_TICKETS, (size_t)pairs * 2 * sizeof(unsigned)));
      if (!p.sk_part || !p.sk_ticket) return ZOACT_ERR_NOMEM;
    }
  }
  p.status = ctx->d_status;
  const int mode = gated ? MODE_GATED : MODE_PAIR;
  if (w4) {
    p.Wq = static_cast<const uint8_t*>(a.W);
    p.Ws = static_cast<const __half*>(a.w_scales);
    p.Wq2 = static_cast<const uint8_t*>(a.W2);
    p.Ws2 = static_cast<const __half*>(a.w_scales2);
    st = timing_begin(ctx);
    if (st) return st;
    st = two ? dispatch2_w4(ctx, mode, a.ydtype, tm, p) : dispatch_w4(ctx, mode, rt, a.ydtype, tm.a, p);
    if (st) return st;
    return timing_end(ctx);
  }
  st = timing_begin(ctx);
  if (st) return st;
  if (two)
    st = a.xdtype == ZOACT_DT_BF16 ? dispatch2_bf16(ctx, mode, rt, a.ydtype, tm, p)
                                   : dispatch2_fp16(ctx, mode, rt, a.ydtype, tm, p);
  else
    st = a.xdtype == ZOACT_DT_BF16 ? dispatch_bf16(ctx, mode, rt, a.ydtype, tm, p)
                                   : dispatch_fp16(ctx, mode, rt, a.ydtype, tm, p);
  if (st) return st;
  return timing_end(ctx);
}

int launch_gemm_tc_f32out(Ctx* ctx, const void* A, const void* B, int dtype, int M, int N, int K, float* D) {
  using namespace pairtc;
  if (M <= 0 || N <= 0) return ZOACT_OK;
  TmaSet tm;
  const int bn = choose_bn(M, N, ctx->sm_count);
  int st = encode_tmap_2d_16bit(&tm.a, A, dtype, M, K, BM);
  if (st) return st;
  st = encode_tmap_2d_16bit(&tm.b, B, dtype, N, K, bn);
  if (st) return st;
  tm.b2 = tm.ba = tm.ba2 = tm.y = tm.y16 = tm.b;
  tm.aa = tm.a;
  Params p{};
  p.Y = D;
  p.rows = M; p.T = M; p.d_in = K; p.d_out = N; p.r = 0;
  p.bn = bn;
  p.num_m = (M + BM - 1) / BM;
  p.num_n = (N + bn - 1) / bn;
  p.num_k = (K + BK - 1) / BK;
  p.num_tiles = p.num_m * p.num_n;
  p.ldy = N;
  p.vec_ok = (N % 4) == 0 && ((uintptr_t)D & 15u) == 0;
  p.status = ctx->d_status;
  return dtype == ZOACT_DT_BF16 ? dispatch_bf16(ctx, MODE_PLAIN, 4, ZOACT_DT_FP32, tm, p)
                                : dispatch_fp16(ctx, MODE_PLAIN, 4, ZOACT_DT_FP32, tm, p);
}

}  // namespace zoact
