// zoact_pair_forward_noalloc: the pair forward for callers that must not
// allocate device memory.
//
// Who needs it: code that runs where cudaMalloc is not allowed or not
// wanted -- inside a framework whose caching allocator owns all device memory
// and must not be bypassed, in a real-time loop that must never hit a
// synchronising allocation, or in a process with a hard memory budget.  The
// regular zoact_pair_forward keeps its projection U^T x in context scratch that
// zoact_create allocates and later calls may grow; this entry point needs no
// context at all.
//
// Its only scratch is the file-scope device array below (4 MiB plus a status
// slot), which every GPU that loads libzoact holds until the process exits.
// Limits beyond the regular entry point's: ranks up to 32 and 16-bit or fp32
// weights (INT4 is refused with ZOACT_ERR_UNSUPPORTED); the low-rank term is
// added from fp32 epilogue tables (the regular entry point can put it on the
// tensor cores), so the outputs agree with zoact_pair_forward within the pair
// forward's tolerance, not bit for bit.
// It stores P = X U ([rows, r] fp32) and, when room is left, the split-K
// partials of that projection.  A request with rows * r above
// ZOACT_NOALLOC_MAX_PROJ_FLOATS is rejected with ZOACT_ERR_TOO_LARGE before
// anything is launched.  All calls share the array and it keeps the last
// call's contents: the status slot is cleared at every call, and P and the
// partials are fully rewritten before they are read.  Calls that overlap on
// the GPU (other streams, other host threads) race on the array.
#include <cuda.h>

#include <mutex>

#include "internal.h"

namespace zoact {
namespace {

constexpr int64_t NOALLOC_FLOATS = ZOACT_NOALLOC_MAX_PROJ_FLOATS;
constexpr int NOALLOC_MAX_DEVICES = 64;

// [0, NOALLOC_FLOATS): projection and split-K partials; the slot after it: status word
static __device__ __align__(256) float g_noalloc_scratch[NOALLOC_FLOATS + 64];

std::mutex g_mu;
float* g_addr[NOALLOC_MAX_DEVICES] = {};
int g_sm_count[NOALLOC_MAX_DEVICES] = {};
unsigned long long g_ctx_id[NOALLOC_MAX_DEVICES] = {};

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

// The process-unique id of the current CUDA context (driver API, CUDA >= 12.0); 0 when there is none yet or
// the query is not available.  A device reset destroys the context, and the array lives in a module loaded
// into it: its address is only valid for the context it was looked up in.
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

// Device address of the array in the current context of device `dev`.  Looked up (with the device current)
// on the first call on the device, and again whenever the current context is not the one of the last lookup
// (after cudaDeviceReset, or when the caller binds another context), so a cached address is never used in a
// context it does not belong to.  Where the context id cannot be read, every call looks the address up.
int scratch_address(int dev, float** out, int* sm_count) {
  if (dev < 0 || dev >= NOALLOC_MAX_DEVICES) return ZOACT_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_mu);
  const unsigned long long id = current_context_id();
  if (!g_addr[dev] || id == 0 || id != g_ctx_id[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);   // creates the context if needed
    if (e != cudaSuccess || !p) {
      cudaGetLastError();
      return ZOACT_ERR_CUDA;
    }
    int sms = 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return ZOACT_ERR_CUDA;
    g_addr[dev] = static_cast<float*>(p);
    g_sm_count[dev] = sms;
    g_ctx_id[dev] = current_context_id();      // the context the lookup ran in (0: look up again next call)
  }
  *out = g_addr[dev];
  *sm_count = g_sm_count[dev];
  return ZOACT_OK;
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

}  // namespace
}  // namespace zoact

using namespace zoact;

extern "C" int zoact_pair_forward_noalloc(const zoact_layer* L, const void* X, int xdtype, int64_t T,
                                          int input_shared, float eps, uint64_t seed, uint64_t query, int act,
                                          void* Y, int ydtype, void* stream) {
  // argument checks: the same rules as zoact_pair_forward
  if (!L || !L->W || !L->U || !L->C || L->d_in <= 0 || L->d_out <= 0 || L->r <= 0) return ZOACT_ERR_INVALID_ARG;
  if (L->r > 32 || L->wtype == ZOACT_DT_INT4_G128) return ZOACT_ERR_UNSUPPORTED;
  const bool ok_x = xdtype == ZOACT_DT_FP32 || xdtype == ZOACT_DT_BF16 || xdtype == ZOACT_DT_FP16;
  const bool ok_y = ydtype == ZOACT_DT_FP32 || ydtype == ZOACT_DT_BF16 || ydtype == ZOACT_DT_FP16;
  if (T < 0 || !ok_x || !ok_y || xdtype != L->wtype) return ZOACT_ERR_INVALID_ARG;
  if (act < ZOACT_ACT_NONE || act > ZOACT_ACT_GELU) return ZOACT_ERR_INVALID_ARG;
  if (T == 0) return ZOACT_OK;
  if (!X || !Y || !aligned16(X) || !aligned16(Y) || !aligned16(L->W)) return ZOACT_ERR_INVALID_ARG;
  if (L->d_in % (xdtype == ZOACT_DT_FP32 ? 4 : 8) != 0 || L->d_out % 8 != 0) return ZOACT_ERR_INVALID_ARG;
  if ((int64_t)L->d_out * L->r >= (int64_t)1 << 34) return ZOACT_ERR_INVALID_ARG;
  const int64_t rows = input_shared ? T : 2 * T;
  if (rows * L->r > NOALLOC_FLOATS) return ZOACT_ERR_TOO_LARGE;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return ZOACT_ERR_CUDA;
  float* base = nullptr;
  Ctx c;
  int st = scratch_address(dev, &base, &c.sm_count);
  if (st) return st;
  c.device = dev;
  c.stream = static_cast<cudaStream_t>(stream);
  c.d_status = reinterpret_cast<int*>(base + NOALLOC_FLOATS);
  c.d_tickets = nullptr;
  c.may_allocate = false;
  ZOACT_CUDA_TRY(cudaMemsetAsync(c.d_status, 0, sizeof(int), c.stream));

  float* P = base;
  const int64_t p_floats = (rows * L->r + 63) / 64 * 64;     // keep the partials 256-byte aligned
  st = launch_lowrank_proj_into(&c, X, xdtype, rows, L->d_in, L->U, L->r, P, base + p_floats,
                                NOALLOC_FLOATS - p_floats);
  if (st) return st;
  PairArgs a{};
  a.X = X; a.W = L->W; a.w_scales = L->w_scales; a.P = P; a.C = L->C; a.Y = Y;
  a.rows = rows; a.T = T; a.d_in = L->d_in; a.d_out = L->d_out; a.r = L->r;
  a.shared = input_shared ? 1 : 0; a.act = act;
  a.xdtype = xdtype; a.wtype = L->wtype; a.ydtype = ydtype;
  set_pair_blocks(a, eps, query);
  a.seed = seed; a.layer_id = L->layer_id;
  return xdtype == ZOACT_DT_FP32 ? launch_pair_simt(&c, a) : launch_pair_tc(&c, a);
}
