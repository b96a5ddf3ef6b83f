// The C ABI of libzoact (declared in include/zoact.h): context, scratch,
// argument validation and dispatch to the kernels.  No compute happens on the
// host; every entry point only checks its arguments and enqueues kernels.
#include <cstdio>
#include <cstdlib>
#include <new>

#include "internal.h"

namespace zoact {

int cuda_fail(cudaError_t e, const char* what) {
  if (std::getenv("ZOACT_DEBUG")) std::fprintf(stderr, "libzoact: %s failed: %s\n", what, cudaGetErrorString(e));
  return e == cudaErrorMemoryAllocation ? ZOACT_ERR_NOMEM : ZOACT_ERR_CUDA;
}

void* scratch(Ctx* ctx, ScratchSlot slot, size_t bytes) {
  if (bytes == 0) bytes = 256;
  if (ctx->slot_bytes[slot] >= bytes) return ctx->slot_ptr[slot];
  if (!ctx->may_allocate) return nullptr;
  if (ctx->slot_ptr[slot]) {
    // queued kernels may still use the old buffer
    if (cudaStreamSynchronize(ctx->stream) != cudaSuccess) return nullptr;
    cudaFree(ctx->slot_ptr[slot]);
    ctx->slot_ptr[slot] = nullptr;
    ctx->slot_bytes[slot] = 0;
  }
  const size_t want = (bytes + 4095) / 4096 * 4096;
  void* p = nullptr;
  if (cudaMalloc(&p, want) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  ctx->slot_ptr[slot] = p;
  ctx->slot_bytes[slot] = want;
  return p;
}

void* scratch_zeroed(Ctx* ctx, ScratchSlot slot, size_t bytes) {
  const void* before = ctx->slot_ptr[slot];
  const size_t had = ctx->slot_bytes[slot];
  void* p = scratch(ctx, slot, bytes);
  if (p && (p != before || ctx->slot_bytes[slot] != had)) {
    if (cudaMemsetAsync(p, 0, ctx->slot_bytes[slot], ctx->stream) != cudaSuccess) {
      cudaGetLastError();
      return nullptr;
    }
  }
  return p;
}

constexpr int TIMING_PAIRS = 4096;

// The event pool is created when timing is switched on, so that no launch pays for it.
int timing_pool(Ctx* ctx) {
  if (ctx->tev) return ZOACT_OK;
  ctx->tev = new (std::nothrow) cudaEvent_t[2 * TIMING_PAIRS];
  if (!ctx->tev) return ZOACT_ERR_NOMEM;
  for (int i = 0; i < 2 * TIMING_PAIRS; ++i) {
    if (cudaEventCreate(&ctx->tev[i]) != cudaSuccess) {
      for (int j = 0; j < i; ++j) cudaEventDestroy(ctx->tev[j]);
      delete[] ctx->tev;
      ctx->tev = nullptr;
      return ZOACT_ERR_CUDA;
    }
  }
  ctx->tev_cap = TIMING_PAIRS;
  return ZOACT_OK;
}

// Nested begin / end pairs (a launch that runs another launcher inside it) time the outermost pair only.
int timing_begin(Ctx* ctx) {
  if (!ctx->timing || !ctx->tev) return ZOACT_OK;
  if (ctx->tev_depth++ > 0) return ZOACT_OK;
  if (ctx->tev_used >= ctx->tev_cap) {
    ++ctx->tev_dropped;
    return ZOACT_OK;
  }
  ZOACT_CUDA_TRY(cudaEventRecord(ctx->tev[2 * ctx->tev_used], ctx->stream));
  return ZOACT_OK;
}

int timing_end(Ctx* ctx) {
  if (!ctx->timing || !ctx->tev) return ZOACT_OK;
  if (ctx->tev_depth > 0 && --ctx->tev_depth > 0) return ZOACT_OK;
  if (ctx->tev_used >= ctx->tev_cap) return ZOACT_OK;
  ZOACT_CUDA_TRY(cudaEventRecord(ctx->tev[2 * ctx->tev_used + 1], ctx->stream));
  ++ctx->tev_used;
  return ZOACT_OK;
}

}  // namespace zoact

using namespace zoact;

namespace {

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

int set_device(zoact_ctx* ctx) {
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess) return ZOACT_ERR_CUDA;
  if (cur != ctx->device && cudaSetDevice(ctx->device) != cudaSuccess) return ZOACT_ERR_CUDA;
  return ZOACT_OK;
}

#define ZOACT_ENTER(ctx)                  \
  do {                                    \
    if (!(ctx)) return ZOACT_ERR_INVALID_ARG; \
    const int s_ = set_device(ctx);       \
    if (s_) return s_;                    \
  } while (0)

bool valid_act_dtype(int dt) { return dt == ZOACT_DT_FP32 || dt == ZOACT_DT_BF16 || dt == ZOACT_DT_FP16; }

int check_layer(const zoact_layer* L) {
  if (!L || !L->W || !L->U || !L->C) return ZOACT_ERR_INVALID_ARG;
  if (L->d_in <= 0 || L->d_out <= 0 || L->r <= 0) return ZOACT_ERR_INVALID_ARG;
  if (L->r > 256) return ZOACT_ERR_UNSUPPORTED;
  if ((int64_t)L->d_out * L->r >= (int64_t)1 << 34) return ZOACT_ERR_INVALID_ARG;
  if (L->wtype == ZOACT_DT_INT4_G128) {
    if (!L->w_scales || L->d_in % 128 != 0 || ((uintptr_t)L->W & 15u) != 0) return ZOACT_ERR_INVALID_ARG;
    return ZOACT_OK;
  }
  if (!valid_act_dtype(L->wtype)) return ZOACT_ERR_INVALID_ARG;
  return ZOACT_OK;
}

}  // namespace

extern "C" {

int zoact_create(zoact_ctx** out, int device, void* stream) {
  if (!out) return ZOACT_ERR_INVALID_ARG;
  *out = nullptr;
  int n = 0;
  if (cudaGetDeviceCount(&n) != cudaSuccess || device < 0 || device >= n) {
    cudaGetLastError();
    return ZOACT_ERR_INVALID_ARG;
  }
  zoact_ctx* ctx = new (std::nothrow) zoact_ctx();
  if (!ctx) return ZOACT_ERR_NOMEM;
  ctx->device = device;
  ctx->stream = static_cast<cudaStream_t>(stream);
  {
    // programmatic dependent launch of the step's kernels: on unless ZOACT_PDL=0
    const char* pdl = std::getenv("ZOACT_PDL");
    ctx->pdl = !(pdl && pdl[0] == '0');
  }
  int st = set_device(ctx);
  if (st) { delete ctx; return st; }
  if (cudaDeviceGetAttribute(&ctx->sm_count, cudaDevAttrMultiProcessorCount, device) != cudaSuccess) {
    delete ctx;
    return ZOACT_ERR_CUDA;
  }
  if (cudaMalloc(&ctx->d_status, 256) != cudaSuccess || cudaMalloc(&ctx->d_tickets, 256) != cudaSuccess ||
      cudaMemsetAsync(ctx->d_status, 0, 256, ctx->stream) != cudaSuccess ||
      cudaMemsetAsync(ctx->d_tickets, 0, 256, ctx->stream) != cudaSuccess ||
      cudaStreamSynchronize(ctx->stream) != cudaSuccess) {
    cudaGetLastError();
    if (ctx->d_status) cudaFree(ctx->d_status);
    if (ctx->d_tickets) cudaFree(ctx->d_tickets);
    delete ctx;
    return ZOACT_ERR_NOMEM;
  }
  *out = ctx;
  return ZOACT_OK;
}

int zoact_destroy(zoact_ctx* ctx) {
  if (!ctx) return ZOACT_OK;
  set_device(ctx);
  cudaStreamSynchronize(ctx->stream);
  for (int s = 0; s < SLOT_COUNT; ++s)
    if (ctx->slot_ptr[s]) cudaFree(ctx->slot_ptr[s]);
  cudaFree(ctx->d_status);
  cudaFree(ctx->d_tickets);
  if (ctx->tev) {
    for (int i = 0; i < 2 * ctx->tev_cap; ++i) cudaEventDestroy(ctx->tev[i]);
    delete[] ctx->tev;
  }
  delete ctx;
  return ZOACT_OK;
}

int zoact_set_stream(zoact_ctx* ctx, void* stream) {
  if (!ctx) return ZOACT_ERR_INVALID_ARG;
  ctx->stream = static_cast<cudaStream_t>(stream);
  return ZOACT_OK;
}

const char* zoact_status_string(int status) {
  switch (status) {
    case ZOACT_OK: return "ok";
    case ZOACT_ERR_INVALID_ARG: return "invalid argument";
    case ZOACT_ERR_UNSUPPORTED: return "unsupported by this build";
    case ZOACT_ERR_CUDA: return "CUDA runtime error";
    case ZOACT_ERR_NONFINITE: return "non-finite loss or estimator";
    case ZOACT_ERR_TIMEOUT: return "bounded device wait timed out";
    case ZOACT_ERR_NOMEM: return "out of device memory";
    case ZOACT_ERR_TOO_LARGE: return "request exceeds the fixed scratch of the no-allocation entry point";
    case ZOACT_ERR_REPLICA_MISMATCH: return "data-parallel replicas hold different coefficients";
    default: return "unknown status";
  }
}

int zoact_get_device_status(zoact_ctx* ctx, int* status, int reset) {
  ZOACT_ENTER(ctx);
  if (!status) return ZOACT_ERR_INVALID_ARG;
  ZOACT_CUDA_TRY(cudaStreamSynchronize(ctx->stream));
  int v = 0;
  ZOACT_CUDA_TRY(cudaMemcpy(&v, ctx->d_status, sizeof(int), cudaMemcpyDeviceToHost));
  *status = v;
  if (v == ZOACT_ERR_TIMEOUT) {
    // a launch that gave up may have left a grid-reduction or split-tail ticket part-counted: zero them all so
    // that the context's next launches count from zero again (the stream is idle here)
    ZOACT_CUDA_TRY(cudaMemsetAsync(ctx->d_tickets, 0, 256, ctx->stream));
    if (ctx->slot_ptr[SLOT_SK_TICKETS])
      ZOACT_CUDA_TRY(cudaMemsetAsync(ctx->slot_ptr[SLOT_SK_TICKETS], 0, ctx->slot_bytes[SLOT_SK_TICKETS], ctx->stream));
    ZOACT_CUDA_TRY(cudaStreamSynchronize(ctx->stream));
  }
  if (reset) {
    ZOACT_CUDA_TRY(cudaMemsetAsync(ctx->d_status, 0, sizeof(int), ctx->stream));
    ZOACT_CUDA_TRY(cudaStreamSynchronize(ctx->stream));
  }
  return ZOACT_OK;
}

namespace {
// Failure-detection test: leave every ticket of the context part-counted (as a
// launch that gave up can), then wait for a device flag that nothing sets, for
// at most wait_ns of %globaltimer, and record ZOACT_ERR_TIMEOUT as the library's
// bounded waits do.  One block; nothing traps or faults.
__global__ void timeout_probe_kernel(const volatile int* flag, int64_t wait_ns, int* status, unsigned int* t0,
                                     int n0, unsigned int* t1, int n1) {
  for (int i = threadIdx.x; i < n0; i += blockDim.x) t0[i] = 1u;
  for (int i = threadIdx.x; i < n1; i += blockDim.x) t1[i] = 1u;
  if (threadIdx.x != 0) return;
  uint64_t start, now;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(start));
  while (*flag == 0) {
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(now));
    if (now - start > (uint64_t)wait_ns) {
      record_error(status, ZOACT_ERR_TIMEOUT);
      return;
    }
  }
}
}  // namespace

int zoact_debug_timeout(zoact_ctx* ctx, int64_t wait_ns) {
  ZOACT_ENTER(ctx);
  if (wait_ns <= 0 || wait_ns > 1000000000LL) return ZOACT_ERR_INVALID_ARG;
  // the flag: a word of the status block past the status itself, zero since creation and never written
  const int* flag = ctx->d_status + 16;
  const int sk_words =
      ctx->slot_ptr[SLOT_SK_TICKETS] ? (int)(ctx->slot_bytes[SLOT_SK_TICKETS] / sizeof(unsigned)) : 0;
  timeout_probe_kernel<<<1, 128, 0, ctx->stream>>>(flag, wait_ns, ctx->d_status, ctx->d_tickets,
                                                   256 / (int)sizeof(unsigned),
                                                   static_cast<unsigned int*>(ctx->slot_ptr[SLOT_SK_TICKETS]), sk_words);
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

int zoact_kernel_timing(zoact_ctx* ctx, int enable) {
  ZOACT_ENTER(ctx);
  if (enable) {
    const int st = timing_pool(ctx);
    if (st != ZOACT_OK) return st;
  }
  ctx->timing = enable != 0;
  ctx->tev_used = 0;
  ctx->tev_dropped = 0;
  ctx->tev_depth = 0;
  return ZOACT_OK;
}

int zoact_kernel_time(zoact_ctx* ctx, double* ms_total, int64_t* launches) {
  ZOACT_ENTER(ctx);
  if (!ms_total || !launches) return ZOACT_ERR_INVALID_ARG;
  ZOACT_CUDA_TRY(cudaStreamSynchronize(ctx->stream));
  double total = 0.0;
  for (int i = 0; i < ctx->tev_used; ++i) {
    float ms = 0.f;
    ZOACT_CUDA_TRY(cudaEventElapsedTime(&ms, ctx->tev[2 * i], ctx->tev[2 * i + 1]));
    total += ms;
  }
  *ms_total = total;
  *launches = ctx->tev_used;
  ctx->tev_used = 0;
  ctx->tev_dropped = 0;
  ctx->tev_depth = 0;
  return ZOACT_OK;
}

int zoact_device_sm_count(zoact_ctx* ctx, int* sm_count) {
  if (!ctx || !sm_count) return ZOACT_ERR_INVALID_ARG;
  *sm_count = ctx->sm_count;
  return ZOACT_OK;
}

int zoact_get_launch_count(zoact_ctx* ctx, int64_t* count) {
  if (!ctx || !count) return ZOACT_ERR_INVALID_ARG;
  *count = ctx->n_launch;
  return ZOACT_OK;
}

int zoact_philox_normals(zoact_ctx* ctx, uint64_t seed, uint32_t layer_id, uint64_t query, int64_t n, float* z_out,
                         uint32_t* words_out) {
  ZOACT_ENTER(ctx);
  if (n < 0 || (n > 0 && !z_out)) return ZOACT_ERR_INVALID_ARG;
  if (n > ((int64_t)1 << 34)) return ZOACT_ERR_INVALID_ARG;
  return launch_philox_normals(ctx, seed, layer_id, query, n, z_out, words_out);
}

int zoact_lowrank_proj(zoact_ctx* ctx, const void* X, int xdtype, int64_t rows, int32_t d_in, const float* U,
                       int32_t r, float* P) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || d_in <= 0 || r <= 0 || !valid_act_dtype(xdtype)) return ZOACT_ERR_INVALID_ARG;
  if (r > 256) return ZOACT_ERR_UNSUPPORTED;
  if (rows == 0) return ZOACT_OK;
  if (!X || !U || !P || !aligned16(X)) return ZOACT_ERR_INVALID_ARG;
  if (d_in % (xdtype == ZOACT_DT_FP32 ? 4 : 8) != 0) return ZOACT_ERR_INVALID_ARG;
  return launch_lowrank_proj(ctx, X, xdtype, rows, d_in, U, r, P);
}

static int check_eval_blocks(const zoact_eval_blocks* b) {
  if (!b || b->n_blocks < 1 || b->n_blocks > ZOACT_MAX_EVAL_BLOCKS) return ZOACT_ERR_INVALID_ARG;
  for (int i = 0; i < b->n_blocks; ++i)
    if (!(b->coef[i] == b->coef[i]) || b->coef[i] > 3.0e38f || b->coef[i] < -3.0e38f) return ZOACT_ERR_INVALID_ARG;
  return ZOACT_OK;
}

static zoact_eval_blocks pair_blocks(float eps, uint64_t query) {
  zoact_eval_blocks b{};
  b.n_blocks = 2;
  b.coef[0] = eps;
  b.coef[1] = -eps;
  b.query[0] = b.query[1] = query;
  return b;
}

int64_t zoact_basis_prepared_bytes(int32_t d_in, int32_t r) {
  if (d_in <= 0 || r <= 0 || r > 256) return -1;
  return (int64_t)basis_tc_rows(r) * d_in * 2;
}

int zoact_basis_prepare(zoact_ctx* ctx, const float* U, int32_t d_in, int32_t r, int32_t xdtype, void* U_tc) {
  ZOACT_ENTER(ctx);
  if (!U || !U_tc || d_in <= 0 || r <= 0) return ZOACT_ERR_INVALID_ARG;
  if (r > 256) return ZOACT_ERR_UNSUPPORTED;
  if (xdtype != ZOACT_DT_BF16 && xdtype != ZOACT_DT_FP16) return ZOACT_ERR_INVALID_ARG;
  if (d_in % 8 != 0 || !aligned16(U_tc)) return ZOACT_ERR_INVALID_ARG;
  return launch_basis_prepare(ctx, U, d_in, r, xdtype, U_tc);
}

int zoact_lowrank_proj_prepared(zoact_ctx* ctx, const void* X, int xdtype, int64_t rows, int32_t d_in,
                                const void* U_tc, int32_t r, float* P) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || d_in <= 0 || r <= 0) return ZOACT_ERR_INVALID_ARG;
  if (r > 256) return ZOACT_ERR_UNSUPPORTED;
  if (xdtype != ZOACT_DT_BF16 && xdtype != ZOACT_DT_FP16) return ZOACT_ERR_INVALID_ARG;
  if (rows == 0) return ZOACT_OK;
  if (!X || !U_tc || !P || !aligned16(X) || !aligned16(U_tc) || d_in % 8 != 0) return ZOACT_ERR_INVALID_ARG;
  return launch_lowrank_proj_tc_prepared(ctx, X, xdtype, rows, d_in, U_tc, r, P);
}

// The loss pair fused into the last pair forward (zoact_pair_forward_loss).
struct FusedLoss {
  const void* target;
  double* out;
  float eps;
};

// Adapted linears run as one launch (zoact_pair_forward_group_rs): the columns, coefficients and Philox
// stream of each.
struct PairSegs {
  int n;
  int off[ZOACT_MAX_GROUP + 1];
  const float* C[ZOACT_MAX_GROUP];
  uint32_t lid[ZOACT_MAX_GROUP];
};

static int pair_common(zoact_ctx* ctx, const zoact_layer* L, const zoact_layer* L2, const void* X, int xdtype,
                       int64_t T, int input_shared, const float* P, const float* P2, const zoact_eval_blocks* blk,
                       uint64_t seed, int act, void* Y, int ydtype, const FusedLoss* fl = nullptr,
                       const zoact_rowscale* rs = nullptr, const PairSegs* segs = nullptr) {
  if (check_eval_blocks(blk)) return ZOACT_ERR_INVALID_ARG;
  int st = check_layer(L);
  if (st) return st;
  if (L2) {
    st = check_layer(L2);
    if (st) return st;
    if (L2->d_in != L->d_in || L2->d_out != L->d_out || L2->r != L->r || L2->wtype != L->wtype)
      return ZOACT_ERR_INVALID_ARG;
  }
  if (T < 0 || !valid_act_dtype(xdtype) || !valid_act_dtype(ydtype)) return ZOACT_ERR_INVALID_ARG;
  if (act < ZOACT_ACT_NONE || act > ZOACT_ACT_GELU) return ZOACT_ERR_INVALID_ARG;
  if (fl) {
    if (!fl->out || !(fl->eps > 0.0f) || (fl->target && !aligned16(fl->target))) return ZOACT_ERR_INVALID_ARG;
    if (input_shared || blk->n_blocks != 2 || T % 256 != 0 || xdtype == ZOACT_DT_FP32 ||
        (ydtype != ZOACT_DT_BF16 && ydtype != ZOACT_DT_FP16))
      return ZOACT_ERR_UNSUPPORTED;
  }
  if (T == 0) return ZOACT_OK;
  if (!X || (!Y && !fl)) return ZOACT_ERR_INVALID_ARG;
  if (L->wtype == ZOACT_DT_INT4_G128 ? xdtype != ZOACT_DT_BF16 : xdtype != L->wtype) return ZOACT_ERR_INVALID_ARG;
  if (!aligned16(X) || (Y && !aligned16(Y)) || !aligned16(L->W) || (L2 && !aligned16(L2->W)))
    return ZOACT_ERR_INVALID_ARG;
  if (L->d_in % (xdtype == ZOACT_DT_FP32 ? 4 : 8) != 0) return ZOACT_ERR_INVALID_ARG;
  if (L->d_out % 8 != 0) return ZOACT_ERR_INVALID_ARG;
  if (T > ((int64_t)1 << 40) / blk->n_blocks) return ZOACT_ERR_INVALID_ARG;
  const int64_t rows = input_shared ? T : blk->n_blocks * T;
  const bool rowscale = rs && (rs->in_scale || rs->out_sumsq);
  if (rowscale) {
    auto al4 = [](const void* q) { return ((uintptr_t)q & 3u) == 0; };
    if ((rs->in_scale && !al4(rs->in_scale)) || (rs->out_sumsq && !al4(rs->out_sumsq))) return ZOACT_ERR_INVALID_ARG;
    // before anything is launched: the kernels that apply row scales serve stacked rows from 256 on CTA pairs
    if (fl || !pair_rowscale_supported(ctx, rows, input_shared, xdtype, L->wtype, blk->n_blocks))
      return ZOACT_ERR_UNSUPPORTED;
  }
  // projection(s) U^T x, unless the caller passed them
  if (!P) {
    float* p = static_cast<float*>(scratch(ctx, SLOT_P0, (size_t)rows * L->r * sizeof(float)));
    if (!p) return ZOACT_ERR_NOMEM;
    st = launch_lowrank_proj(ctx, X, xdtype, rows, L->d_in, L->U, L->r, p);
    if (st) return st;
    P = p;
  }
  if (L2 && !P2 && L2->U == L->U && L2->r == L->r && L2->d_in == L->d_in) P2 = P;   // one basis: one projection
  if (L2 && !P2) {
    float* p = static_cast<float*>(scratch(ctx, SLOT_P1, (size_t)rows * L2->r * sizeof(float)));
    if (!p) return ZOACT_ERR_NOMEM;
    st = launch_lowrank_proj(ctx, X, xdtype, rows, L2->d_in, L2->U, L2->r, p);
    if (st) return st;
    P2 = p;
  }
  PairArgs a{};
  a.X = X; a.W = L->W; a.w_scales = L->w_scales; a.P = P; a.C = L->C; a.Y = Y;
  a.rows = rows; a.T = T; a.d_in = L->d_in; a.d_out = L->d_out; a.r = L->r;
  a.shared = input_shared ? 1 : 0; a.act = act;
  a.xdtype = xdtype; a.wtype = L->wtype; a.ydtype = ydtype;
  a.nb = blk->n_blocks;
  for (int b = 0; b < blk->n_blocks; ++b) { a.coef[b] = blk->coef[b]; a.qry[b] = blk->query[b]; }
  a.seed = seed; a.layer_id = L->layer_id;
  if (L2) { a.W2 = L2->W; a.w_scales2 = L2->w_scales; a.P2 = P2; a.C2 = L2->C; a.layer_id2 = L2->layer_id; }
  if (fl) { a.fuse_loss = 1; a.target = fl->target; a.loss_out = fl->out; a.loss_eps = fl->eps; }
  if (rowscale) { a.in_scale = rs->in_scale; a.out_sumsq = rs->out_sumsq; }
  if (segs && segs->n > 1) {
    a.nseg = segs->n;
    for (int g = 0; g <= segs->n; ++g) a.seg_off[g] = segs->off[g];
    for (int g = 0; g < segs->n; ++g) { a.seg_C[g] = segs->C[g]; a.seg_lid[g] = segs->lid[g]; }
  }
  if (xdtype == ZOACT_DT_FP32) return launch_pair_simt(ctx, a);
  return launch_pair_tc(ctx, a);
}

// Layers that read one input as one pair forward over their concatenated weights (include/zoact.h).
static int group_common(zoact_ctx* ctx, const zoact_layer* layers, int32_t n_layers, const void* X, int xdtype,
                        int64_t T, const float* P, const zoact_eval_blocks* blk, uint64_t seed, int act, void* Y,
                        int ydtype, const zoact_rowscale* rs) {
  if (!layers || n_layers < 1 || n_layers > ZOACT_MAX_GROUP) return ZOACT_ERR_INVALID_ARG;
  if (check_eval_blocks(blk)) return ZOACT_ERR_INVALID_ARG;
  const zoact_layer& L0 = layers[0];
  int st = check_layer(&L0);
  if (st) return st;
  const bool int4 = L0.wtype == ZOACT_DT_INT4_G128;
  const int64_t w_row = int4 ? L0.d_in / 2 : (int64_t)L0.d_in * (int64_t)dtype_size(L0.wtype);
  const int64_t s_row = int4 ? (int64_t)(L0.d_in / 128) * 2 : 0;
  PairSegs sg{};
  sg.n = n_layers;
  int64_t off = 0;
  for (int i = 0; i < n_layers; ++i) {
    const zoact_layer& Li = layers[i];
    st = check_layer(&Li);
    if (st) return st;
    if (Li.d_in != L0.d_in || Li.r != L0.r || Li.wtype != L0.wtype || Li.U != L0.U) return ZOACT_ERR_INVALID_ARG;
    // W rows (and INT4 scale rows) of layer i follow those of the layers before it
    if (static_cast<const char*>(Li.W) != static_cast<const char*>(L0.W) + off * w_row) return ZOACT_ERR_INVALID_ARG;
    if (int4 && static_cast<const char*>(Li.w_scales) != static_cast<const char*>(L0.w_scales) + off * s_row)
      return ZOACT_ERR_INVALID_ARG;
    sg.off[i] = (int)off;
    sg.C[i] = Li.C;
    sg.lid[i] = Li.layer_id;
    off += Li.d_out;
    if (off > 0x7fffffff) return ZOACT_ERR_INVALID_ARG;
  }
  sg.off[n_layers] = (int)off;
  zoact_layer Lc = L0;
  Lc.d_out = (int32_t)off;
  st = check_layer(&Lc);
  if (st) return st;
  if (T < 0 || T > ((int64_t)1 << 40) / blk->n_blocks) return ZOACT_ERR_INVALID_ARG;
  // one launch only where the kernel takes the whole low-rank term from the operand tables: decided before
  // anything (the projection included) is launched
  if (n_layers > 1 && T > 0 &&
      !pair_rowscale_supported(ctx, (int64_t)blk->n_blocks * T, 0, xdtype, L0.wtype, blk->n_blocks))
    return ZOACT_ERR_UNSUPPORTED;
  return pair_common(ctx, &Lc, nullptr, X, xdtype, T, 0, P, nullptr, blk, seed, act, Y, ydtype, nullptr, rs,
                     n_layers > 1 ? &sg : nullptr);
}

int zoact_pair_forward_loss(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                            const float* P, float eps, uint64_t seed, uint64_t query, int act, int ydtype,
                            const void* target, double* out) {
  ZOACT_ENTER(ctx);
  const zoact_eval_blocks b = pair_blocks(eps, query);
  const FusedLoss fl{target, out, eps};
  return pair_common(ctx, layer, nullptr, X, xdtype, T, 0, P, nullptr, &b, seed, act, nullptr, ydtype, &fl);
}

int zoact_pair_forward(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                       int input_shared, const float* P, float eps, uint64_t seed, uint64_t query, int act, void* Y,
                       int ydtype) {
  ZOACT_ENTER(ctx);
  const zoact_eval_blocks b = pair_blocks(eps, query);
  return pair_common(ctx, layer, nullptr, X, xdtype, T, input_shared, P, nullptr, &b, seed, act, Y, ydtype);
}

int zoact_multi_forward(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                        int input_shared, const float* P, const zoact_eval_blocks* blocks, uint64_t seed, int act,
                        void* Y, int ydtype) {
  ZOACT_ENTER(ctx);
  return pair_common(ctx, layer, nullptr, X, xdtype, T, input_shared, P, nullptr, blocks, seed, act, Y, ydtype);
}

int zoact_multi_forward_rs(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                           int input_shared, const float* P, const zoact_eval_blocks* blocks, uint64_t seed, int act,
                           void* Y, int ydtype, const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  return pair_common(ctx, layer, nullptr, X, xdtype, T, input_shared, P, nullptr, blocks, seed, act, Y, ydtype,
                     nullptr, rs);
}
int zoact_multi_forward_gated_rs(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up, const void* X,
                                 int xdtype, int64_t T, int input_shared, const float* P_gate, const float* P_up,
                                 const zoact_eval_blocks* blocks, uint64_t seed, void* H, int ydtype,
                                 const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  if (!gate || !up) return ZOACT_ERR_INVALID_ARG;
  if (xdtype == ZOACT_DT_FP32) return ZOACT_ERR_UNSUPPORTED;
  return pair_common(ctx, gate, up, X, xdtype, T, input_shared, P_gate, P_up, blocks, seed, ZOACT_ACT_NONE, H,
                     ydtype, nullptr, rs);
}
int zoact_multi_forward_gated(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up, const void* X,
                              int xdtype, int64_t T, int input_shared, const float* P_gate, const float* P_up,
                              const zoact_eval_blocks* blocks, uint64_t seed, void* H, int ydtype) {
  ZOACT_ENTER(ctx);
  if (!gate || !up) return ZOACT_ERR_INVALID_ARG;
  if (xdtype == ZOACT_DT_FP32) return ZOACT_ERR_UNSUPPORTED;
  return pair_common(ctx, gate, up, X, xdtype, T, input_shared, P_gate, P_up, blocks, seed, ZOACT_ACT_NONE, H,
                     ydtype);
}

int zoact_pair_forward_rs(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                          int input_shared, const float* P, float eps, uint64_t seed, uint64_t query, int act, void* Y,
                          int ydtype, const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  const zoact_eval_blocks b = pair_blocks(eps, query);
  return pair_common(ctx, layer, nullptr, X, xdtype, T, input_shared, P, nullptr, &b, seed, act, Y, ydtype, nullptr,
                     rs);
}

int zoact_pair_forward_gated_rs(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up, const void* X,
                                int xdtype, int64_t T, int input_shared, const float* P_gate, const float* P_up,
                                float eps, uint64_t seed, uint64_t query, void* H, int ydtype,
                                const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  if (!gate || !up) return ZOACT_ERR_INVALID_ARG;
  if (xdtype == ZOACT_DT_FP32) return ZOACT_ERR_UNSUPPORTED;
  const zoact_eval_blocks b = pair_blocks(eps, query);
  return pair_common(ctx, gate, up, X, xdtype, T, input_shared, P_gate, P_up, &b, seed, ZOACT_ACT_NONE, H, ydtype,
                     nullptr, rs);
}

int zoact_pair_forward_group_rs(zoact_ctx* ctx, const zoact_layer* layers, int32_t n_layers, const void* X,
                                int xdtype, int64_t T, const float* P, float eps, uint64_t seed, uint64_t query,
                                int act, void* Y, int ydtype, const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  const zoact_eval_blocks b = pair_blocks(eps, query);
  return group_common(ctx, layers, n_layers, X, xdtype, T, P, &b, seed, act, Y, ydtype, rs);
}

int zoact_multi_forward_group_rs(zoact_ctx* ctx, const zoact_layer* layers, int32_t n_layers, const void* X,
                                 int xdtype, int64_t T, const float* P, const zoact_eval_blocks* blocks,
                                 uint64_t seed, int act, void* Y, int ydtype, const zoact_rowscale* rs) {
  ZOACT_ENTER(ctx);
  return group_common(ctx, layers, n_layers, X, xdtype, T, P, blocks, seed, act, Y, ydtype, rs);
}

int zoact_rms_scale(zoact_ctx* ctx, const float* sumsq, int64_t rows, int32_t n, float eps, float* inv_scale) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || n <= 0 || !(eps >= 0.0f)) return ZOACT_ERR_INVALID_ARG;
  if (rows == 0) return ZOACT_OK;
  if (!sumsq || !inv_scale || ((uintptr_t)sumsq & 3u) || ((uintptr_t)inv_scale & 3u)) return ZOACT_ERR_INVALID_ARG;
  return launch_rms_scale(ctx, sumsq, rows, n, eps, inv_scale);
}

int zoact_pair_forward_gated(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up, const void* X,
                             int xdtype, int64_t T, int input_shared, const float* P_gate, const float* P_up,
                             float eps, uint64_t seed, uint64_t query, void* H, int ydtype) {
  ZOACT_ENTER(ctx);
  if (!gate || !up) return ZOACT_ERR_INVALID_ARG;
  if (xdtype == ZOACT_DT_FP32) return ZOACT_ERR_UNSUPPORTED;
  const zoact_eval_blocks b = pair_blocks(eps, query);
  return pair_common(ctx, gate, up, X, xdtype, T, input_shared, P_gate, P_up, &b, seed, ZOACT_ACT_NONE, H, ydtype);
}

int zoact_loss_pair(zoact_ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n, float eps,
                    double* out) {
  ZOACT_ENTER(ctx);
  if (!Y || !out || T <= 0 || n <= 0 || !valid_act_dtype(ydtype)) return ZOACT_ERR_INVALID_ARG;
  if (!(eps > 0.0f)) return ZOACT_ERR_INVALID_ARG;
  const int max_blocks = loss_pair_max_blocks(ctx);
  double* partials = static_cast<double*>(scratch(ctx, SLOT_PARTIALS, (size_t)max_blocks * 3 * sizeof(double)));
  if (!partials) return ZOACT_ERR_NOMEM;
  return launch_loss_pair(ctx, Y, ydtype, target, T, n, eps, out, partials, max_blocks);
}

int zoact_loss_multi(zoact_ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n,
                     int32_t n_blocks, float mu, double* out) {
  ZOACT_ENTER(ctx);
  if (!Y || !out || T <= 0 || n <= 0 || !valid_act_dtype(ydtype)) return ZOACT_ERR_INVALID_ARG;
  if (n_blocks < 2 || n_blocks > ZOACT_MAX_EVAL_BLOCKS || !(mu > 0.0f)) return ZOACT_ERR_INVALID_ARG;
  if (T * n > ((int64_t)1 << 40) / n_blocks) return ZOACT_ERR_INVALID_ARG;
  const int max_blocks = loss_pair_max_blocks(ctx);
  double* partials =
      static_cast<double*>(scratch(ctx, SLOT_PARTIALS, (size_t)max_blocks * 2 * n_blocks * sizeof(double)));
  if (!partials) return ZOACT_ERR_NOMEM;
  return launch_loss_multi(ctx, Y, ydtype, target, T, n, n_blocks, mu, out, partials, max_blocks);
}

static int check_blocks(const float* C, int64_t n_total, const zoact_coeff_block* blocks, int32_t n_blocks) {
  if (!C || n_total < 0 || n_blocks < 0 || (n_blocks > 0 && !blocks)) return ZOACT_ERR_INVALID_ARG;
  if (!aligned16(C)) return ZOACT_ERR_INVALID_ARG;
  int64_t prev_end = 0;
  for (int i = 0; i < n_blocks; ++i) {
    const zoact_coeff_block& b = blocks[i];
    if (b.offset < prev_end || b.offset % 4 != 0 || b.d_out <= 0 || b.r <= 0) return ZOACT_ERR_INVALID_ARG;
    const int64_t end = b.offset + (int64_t)b.d_out * b.r;
    if (end > n_total || (int64_t)b.d_out * b.r >= (int64_t)1 << 34) return ZOACT_ERR_INVALID_ARG;
    prev_end = end;
  }
  return ZOACT_OK;
}

int zoact_adam_step(zoact_ctx* ctx, float* C, float* m, float* v, int64_t n_total, const zoact_coeff_block* blocks,
                    int32_t n_blocks, const double* loss_out, float lr, float beta1, float beta2, float adam_eps,
                    int64_t step, uint64_t seed, uint64_t query) {
  ZOACT_ENTER(ctx);
  int st = check_blocks(C, n_total, blocks, n_blocks);
  if (st) return st;
  if (!m || !v || !loss_out || step < 1 || !aligned16(m) || !aligned16(v)) return ZOACT_ERR_INVALID_ARG;
  if (!(beta1 >= 0.f && beta1 < 1.f && beta2 >= 0.f && beta2 < 1.f)) return ZOACT_ERR_INVALID_ARG;
  return launch_adam(ctx, C, m, v, blocks, n_blocks, loss_out + 3, 1, &query, lr, beta1, beta2, adam_eps, step, seed,
                     0);
}

int zoact_adam_step_multi(zoact_ctx* ctx, float* C, float* m, float* v, int64_t n_total,
                          const zoact_coeff_block* blocks, int32_t n_blocks, const double* a, int32_t q,
                          const uint64_t* queries, float lr, float beta1, float beta2, float adam_eps, int64_t step,
                          uint64_t seed) {
  ZOACT_ENTER(ctx);
  int st = check_blocks(C, n_total, blocks, n_blocks);
  if (st) return st;
  if (!m || !v || !a || !queries || step < 1 || !aligned16(m) || !aligned16(v)) return ZOACT_ERR_INVALID_ARG;
  if (q < 1 || q > ZOACT_MAX_EVAL_BLOCKS - 1) return ZOACT_ERR_INVALID_ARG;
  if (!(beta1 >= 0.f && beta1 < 1.f && beta2 >= 0.f && beta2 < 1.f)) return ZOACT_ERR_INVALID_ARG;
  return launch_adam(ctx, C, m, v, blocks, n_blocks, a, q, queries, lr, beta1, beta2, adam_eps, step, seed, 0);
}

int zoact_sgd_step_multi(zoact_ctx* ctx, float* C, int64_t n_total, const zoact_coeff_block* blocks,
                         int32_t n_blocks, const double* a, int32_t q, const uint64_t* queries, float lr,
                         uint64_t seed) {
  ZOACT_ENTER(ctx);
  int st = check_blocks(C, n_total, blocks, n_blocks);
  if (st) return st;
  if (!a || !queries || q < 1 || q > ZOACT_MAX_EVAL_BLOCKS - 1) return ZOACT_ERR_INVALID_ARG;
  return launch_adam(ctx, C, nullptr, nullptr, blocks, n_blocks, a, q, queries, lr, 0.f, 0.f, 0.f, 1, seed, 1);
}

int zoact_sgd_step(zoact_ctx* ctx, float* C, int64_t n_total, const zoact_coeff_block* blocks, int32_t n_blocks,
                   const double* loss_out, float lr, uint64_t seed, uint64_t query) {
  ZOACT_ENTER(ctx);
  int st = check_blocks(C, n_total, blocks, n_blocks);
  if (st) return st;
  if (!loss_out) return ZOACT_ERR_INVALID_ARG;
  return launch_adam(ctx, C, nullptr, nullptr, blocks, n_blocks, loss_out + 3, 1, &query, lr, 0.f, 0.f, 0.f, 1, seed,
                     1);
}

int zoact_basis_init(zoact_ctx* ctx, const void* X_cal, int xdtype, int64_t n_tok, int32_t d_in, int32_t r,
                     int32_t oversample, int32_t n_iter, uint64_t seed, float* U_out, float* evals_out) {
  ZOACT_ENTER(ctx);
  if (!X_cal || !U_out || n_tok <= 0 || d_in <= 0 || r <= 0 || oversample < 0 || n_iter < 0 ||
      !valid_act_dtype(xdtype))
    return ZOACT_ERR_INVALID_ARG;
  if (r > d_in) return ZOACT_ERR_INVALID_ARG;
  if (xdtype != ZOACT_DT_FP32 && (d_in % 8 != 0 || !aligned16(X_cal))) return ZOACT_ERR_INVALID_ARG;
  if (n_tok > INT32_MAX) return ZOACT_ERR_UNSUPPORTED;
  return run_basis_init(ctx, X_cal, xdtype, n_tok, d_in, r, oversample, n_iter, seed, U_out, evals_out);
}

int zoact_subspace_overlap(zoact_ctx* ctx, const float* U_a, const float* U_b, int32_t d, int32_t r_a, int32_t r_b,
                           double* out) {
  ZOACT_ENTER(ctx);
  if (!U_a || !U_b || !out || d <= 0 || r_a <= 0 || r_b <= 0) return ZOACT_ERR_INVALID_ARG;
  if (r_a > 256 || r_b > 256) return ZOACT_ERR_UNSUPPORTED;
  return launch_subspace_overlap(ctx, U_a, U_b, d, r_a, r_b, out);
}

int zoact_gradient_energy(zoact_ctx* ctx, const float* U, int32_t d_in, int32_t r, const void* G, int gdtype, int64_t n,
                          double* out) {
  ZOACT_ENTER(ctx);
  if (!U || !G || !out || d_in <= 0 || r <= 0 || n <= 0 || !valid_act_dtype(gdtype)) return ZOACT_ERR_INVALID_ARG;
  if (r > 256) return ZOACT_ERR_UNSUPPORTED;
  return launch_gradient_energy(ctx, U, d_in, r, G, gdtype, n, out);
}

int zoact_rms_norm(zoact_ctx* ctx, const void* X, int dtype, int64_t rows, int32_t n, float eps, void* Y) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || n <= 0 || !valid_act_dtype(dtype)) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0 && (!X || !Y)) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0x7fffffff) return ZOACT_ERR_UNSUPPORTED;
  return launch_rms_norm(ctx, X, dtype, rows, n, eps, Y);
}

int zoact_mix_rms(zoact_ctx* ctx, const void* q, const void* k, const void* v, int dtype, int64_t rows, int32_t n,
                  int32_t n_rep, int32_t head_dim, float eps, void* Y) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || n <= 0 || n_rep <= 0 || head_dim <= 0 || !valid_act_dtype(dtype)) return ZOACT_ERR_INVALID_ARG;
  if (n % (n_rep * head_dim) != 0) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0 && (!q || !k || !v || !Y)) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0x7fffffff) return ZOACT_ERR_UNSUPPORTED;
  return launch_mix_rms(ctx, q, k, v, dtype, rows, n, n_rep, head_dim, eps, Y, n, n / n_rep);
}

int zoact_mix_rms_strided(zoact_ctx* ctx, const void* q, const void* k, const void* v, int dtype, int64_t rows,
                          int32_t n, int32_t n_rep, int32_t head_dim, int64_t ld_q, int64_t ld_kv, float eps,
                          void* Y) {
  ZOACT_ENTER(ctx);
  if (rows < 0 || n <= 0 || n_rep <= 0 || head_dim <= 0 || !valid_act_dtype(dtype)) return ZOACT_ERR_INVALID_ARG;
  if (n % (n_rep * head_dim) != 0 || ld_q < n || ld_kv < n / n_rep) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0 && (!q || !k || !v || !Y)) return ZOACT_ERR_INVALID_ARG;
  if (rows > 0x7fffffff) return ZOACT_ERR_UNSUPPORTED;
  return launch_mix_rms(ctx, q, k, v, dtype, rows, n, n_rep, head_dim, eps, Y, ld_q, ld_kv);
}

}  // extern "C"

int zoact_mean_over_ranks(zoact_ctx* ctx, double* v, int64_t n, int32_t world) {
  ZOACT_ENTER(ctx);
  if (n < 0 || world < 1 || (n > 0 && !v)) return ZOACT_ERR_INVALID_ARG;
  return launch_mean_over_ranks(ctx, v, n, world);
}

int zoact_arena_hash(zoact_ctx* ctx, const void* data, int64_t n_words, uint64_t* hash_out) {
  ZOACT_ENTER(ctx);
  if (!hash_out || n_words < 0 || n_words >= ((int64_t)1 << 32) || (n_words > 0 && !data)) return ZOACT_ERR_INVALID_ARG;
  if (((uintptr_t)hash_out & 7u) != 0) return ZOACT_ERR_INVALID_ARG;
  if (n_words >= 4 && ((uintptr_t)data & 15u) != 0) return ZOACT_ERR_INVALID_ARG;
  if (((uintptr_t)data & 3u) != 0) return ZOACT_ERR_INVALID_ARG;
  return launch_arena_hash(ctx, data, n_words, hash_out);
}
