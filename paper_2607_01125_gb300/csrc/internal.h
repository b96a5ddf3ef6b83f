// Internal declarations shared by the libzoact translation units.
#pragma once
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cstdint>
#include <cstddef>

#include "../../include/zoact.h"

#define ZOACT_CUDA_TRY(expr)                                  \
  do {                                                        \
    cudaError_t e_ = (expr);                                  \
    if (e_ != cudaSuccess) return zoact::cuda_fail(e_, #expr); \
  } while (0)

#define ZOACT_CHECK_LAUNCH() ZOACT_CUDA_TRY(cudaGetLastError())

namespace zoact {

// Scratch slots owned by a context.  Each slot grows on demand; growing
// synchronises the stream first so no queued kernel still uses the old buffer.
enum ScratchSlot {
  SLOT_P0 = 0,       // projection U^T x of the current call
  SLOT_P1,           // second projection (gated pair forward)
  SLOT_SPLITK,       // split-K partials of the projection
  SLOT_PARTIALS,     // per-block partial sums of grid reductions
  SLOT_BASIS,        // Gram matrix and subspace-iteration workspace
  SLOT_BASIS_X,      // transposed calibration activations
  SLOT_UT,           // 16-bit split copy of the basis for the tensor-core projection
  SLOT_WDQ0,         // bf16 copy of an INT4 weight (staged INT4 pair forward)
  SLOT_WDQ1,         // second copy (gated up weight)
  SLOT_AUG_A,        // 16-bit split of the projection P (extra K columns of the tensor-core pair forward)
  SLOT_AUG_B,        // 16-bit split of C (+ c_b Z_b) for those K columns (gate and up)
  SLOT_AUG_Z,        // Z of each query, transposed, for the epilogue (C on the tensor cores)
  SLOT_DIAG,         // partial products of the subspace diagnostics
  SLOT_STACKED_X,    // a shared input and its projection copied once per evaluation block (ranks above 32)
  SLOT_SK_PART,      // partial accumulators of the CTA-pair kernel's split tail
  SLOT_SK_TICKETS,   // its per-tile tickets (zero between launches)
  SLOT_COUNT
};

struct Ctx {
  int device = 0;
  cudaStream_t stream = nullptr;
  int sm_count = 0;
  int64_t n_launch = 0;              // kernels launched through this context (host counter)
  bool may_allocate = true;          // false: no scratch may be allocated (kernels that need none only)
  bool pdl = false;                   // step-path kernels launched with programmatic dependent launch
  int* d_status = nullptr;            // device status word (first error wins)
  unsigned int* d_tickets = nullptr;  // grid-reduction tickets, reset by their last block
  void* slot_ptr[SLOT_COUNT] = {};
  size_t slot_bytes[SLOT_COUNT] = {};
  // kernel timing (zoact_kernel_timing): event pairs around the tensor-core pair-forward launches
  bool timing = false;
  cudaEvent_t* tev = nullptr;        // 2 * tev_cap events, created on demand
  int tev_cap = 0;
  int tev_used = 0;                   // pairs recorded since the last read
  int64_t tev_dropped = 0;            // launches not timed (capacity reached)
  int tev_depth = 0;                  // nesting of timing_begin / timing_end (the outermost pair records)
};

// Record the start / end of a timed launch on the context's stream (no-ops unless timing is on).
int timing_begin(Ctx* ctx);
int timing_end(Ctx* ctx);

int cuda_fail(cudaError_t e, const char* what);
// Returns a device pointer of at least `bytes` for the slot, or nullptr on failure.
void* scratch(Ctx* ctx, ScratchSlot slot, size_t bytes);
// As scratch(), and a newly allocated buffer is zero-filled (on the context's stream).
void* scratch_zeroed(Ctx* ctx, ScratchSlot slot, size_t bytes);

// ---- programmatic dependent launch ----
// launch_pdl puts a kernel on the context's stream; with ctx->pdl the launch
// allows its blocks to be scheduled while the previous kernel on the stream
// drains (from the moment every block of that kernel has called pdl_trigger()
// or exited).  Every kernel launched this way calls pdl_wait() before its first
// global memory access, read or write: it returns once the previous kernel has
// completed and its writes are visible, so stream order holds for memory and
// only the launch latency and the block prologue overlap the previous kernel.
// A kernel calls pdl_trigger() only after its own pdl_wait(), which keeps the
// chain transitive (kernel i+2 cannot start before kernel i has completed).
// Both are no-ops in a kernel launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(Ctx* ctx, void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = ctx->stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = ctx->pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

// Device-side error recording: keeps the first non-zero code.
__device__ __forceinline__ void record_error(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// ---- dtype helpers ----
template <typename T> __device__ __forceinline__ float to_f32(T v);
template <> __device__ __forceinline__ float to_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ float to_f32<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }
template <> __device__ __forceinline__ float to_f32<__half>(__half v) { return __half2float(v); }

template <typename T> __device__ __forceinline__ T from_f32(float v);
template <> __device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <> __device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }
template <> __device__ __forceinline__ __half from_f32<__half>(float v) { return __float2half_rn(v); }

__device__ __forceinline__ float apply_act(float y, int act) {
  if (act == ZOACT_ACT_RELU) return fmaxf(y, 0.0f);
  if (act == ZOACT_ACT_GELU) return 0.5f * y * (1.0f + erff(y * 0.70710678118654752f));
  return y;
}

__device__ __forceinline__ float silu_f(float x) { return x / (1.0f + expf(-x)); }

inline size_t dtype_size(int dt) {
  return dt == ZOACT_DT_FP32 ? 4 : 2;
}

// ---- launchers (return ZOACT_* status) ----
int launch_philox_normals(Ctx* ctx, uint64_t seed, uint32_t layer_id, uint64_t query, int64_t n,
                          float* z, uint32_t* words);
int launch_lowrank_proj(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U,
                        int r, float* P);
// Tensor-core projection for 16-bit X (U split into three 16-bit terms).
int launch_lowrank_proj_tc(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U, int r,
                           float* P);
// The basis in the tensor-core projection's operand form: [basis_tc_rows(r), d_in] 16-bit (xdtype),
// rows [0, RT) / [RT, 2RT) / [2RT, 3RT) the three 16-bit terms of U^T (RT = r rounded up to 4, 8, 16, 32).
int basis_tc_rows(int r);
int launch_basis_prepare(Ctx* ctx, const float* U, int d_in, int r, int xdtype, void* Ut);
int launch_lowrank_proj_tc_prepared(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const void* Ut,
                                    int r, float* P);
// As launch_lowrank_proj, with split-K partials in `part` (part_floats floats) instead of context scratch.
int launch_lowrank_proj_into(Ctx* ctx, const void* X, int xdtype, int64_t rows, int d_in, const float* U,
                             int r, float* P, float* part, int64_t part_floats);

struct PairArgs {
  const void* X;        // [rows, d_in]
  const void* W;        // [d_out, d_in] (or INT4 packed)
  const void* w_scales;
  const float* P;       // [rows, r]
  const float* C;       // [d_out, r]
  void* Y;              // [nb T, d_out]
  int64_t rows;         // rows of X (T if shared else nb T)
  int64_t T;
  int d_in, d_out, r;
  int shared;
  int act;
  int xdtype, wtype, ydtype;
  // evaluation blocks: rows [b T, (b+1) T) of Y at C + coef[b] Z(seed, layer_id, qry[b])
  int nb;
  float coef[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t qry[ZOACT_MAX_EVAL_BLOCKS];
  uint64_t seed;
  uint32_t layer_id;
  // gated mode (second layer: up); W2 == nullptr for the plain pair forward
  const void* W2;
  const void* w_scales2;
  const float* P2;
  const float* C2;
  uint32_t layer_id2;
  // fused loss pair (zoact_pair_forward_loss): Y is not written; the losses of the rounded outputs
  int fuse_loss;
  const void* target;   // [T, d_out] of ydtype, or nullptr (mean of squares)
  double* loss_out;     // [4] = {L+, L-, D, a}
  float loss_eps;
  // row scales (zoact_pair_forward_rs): in_scale [rows] multiplies each output row before the activation;
  // out_sumsq [ceil(d_out / 64), nb T] receives per-64-column-part sums of squares of the stored outputs
  const float* in_scale;
  float* out_sumsq;
  // adapted linears that read one input, run as one (zoact_pair_forward_group_rs): output columns
  // [seg_off[s], seg_off[s + 1]) are layer s's, with coefficients seg_C[s] and Philox stream seg_lid[s]
  // (d_out is the sum, W the first layer's rows followed by the others'); nseg <= 1: one layer
  int nseg;
  int seg_off[ZOACT_MAX_GROUP + 1];
  const float* seg_C[ZOACT_MAX_GROUP];
  uint32_t seg_lid[ZOACT_MAX_GROUP];
};
// Whether a launch with row scales runs on a kernel that applies them (CTA pairs, stacked rows, the whole
// low-rank term on the MMA, staged output) -- decided before anything is launched.
bool pair_rowscale_supported(const Ctx* ctx, int64_t rows, int shared, int xdtype, int wtype, int nb);
// inv[t] = 1 / sqrt(sum_p parts[p][t] / n + eps) over the ceil(n / 64) parts, in part order.
int launch_rms_scale(Ctx* ctx, const float* parts, int64_t rows, int n, float eps, float* inv);
// The two-sided pair as evaluation blocks: {+eps, -eps} with the same query.
inline void set_pair_blocks(PairArgs& a, float eps, uint64_t query) {
  a.nb = 2;
  a.coef[0] = eps;
  a.coef[1] = -eps;
  a.qry[0] = a.qry[1] = query;
}
int launch_pair_simt(Ctx* ctx, const PairArgs& a);
// INT4 g128 weight [d_out, d_in/2] + fp16 scales -> bf16 [d_out, d_in].
int launch_dequant_int4(Ctx* ctx, const void* Wq, const void* Ws, void* Wb, int64_t d_out, int d_in);
// Row count from which the INT4 pair forward expands W to bf16 first instead of dequantising per M-tile.
constexpr int64_t INT4_STAGED_MIN_ROWS = 1024;
int launch_pair_tc(Ctx* ctx, const PairArgs& a);
// Plain product D[M, N] (fp32) = A[M, K] * B[N, K]^T with 16-bit A, B (K-major), on tcgen05.
// Low-rank term of the tensor-core pair forward (see k_aug.cu):
//   LOWRANK_EPILOGUE  (C + c_b Z_b) p summed in the epilogue (fp32 tables)
//   LOWRANK_C_ON_TC   C p as extra K columns of the MMA, c_b Z_b p in the epilogue
//   LOWRANK_ALL_ON_TC (C + c_b Z_b) p as extra K columns (stacked rows): one K slot when every tile lies in
//                     one evaluation block, two slots (block parity) when tiles straddle two blocks
enum LowrankMode { LOWRANK_EPILOGUE = 0, LOWRANK_C_ON_TC = 1, LOWRANK_ALL_ON_TC = 2 };
// Extra K columns per layer for rank r: the three 16-bit products P_hi T_hi, P_hi T_lo, P_lo T_hi
// padded to whole 64-column K-blocks.
inline int aug_cols(int r) { return (3 * r + 63) / 64 * 64; }
// Writes A_aug [rows, ka_tot] and B_aug / B_aug2 [nbB * d_out, ka_tot] (bf16) for one pair forward.
// distinct: gate and up have their own projections (A_aug holds both, B_aug zero-pads the other half).
// Zt / Zt2 (optional): Z of the nzq queries zq, transposed, [nzq][r][d_out] fp32 each.
// slots (LOWRANK_ALL_ON_TC): S > 1 puts row t's parts in K slot block(t) mod S of an A_aug row of S ka columns.
int launch_aug_prep(Ctx* ctx, const PairArgs& a, int mode, int ka, int distinct, int slots, void* A_aug,
                    void* B_aug, void* B_aug2, float* Zt, float* Zt2, const uint64_t* zq, int nzq);
int launch_gemm_tc_f32out(Ctx* ctx, const void* A, const void* B, int dtype, int M, int N, int K,
                          float* D);

int launch_loss_pair(Ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n,
                     float eps, double* out, double* partials, int max_blocks);
int loss_pair_max_blocks(Ctx* ctx);

int launch_loss_multi(Ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n, int nb,
                      float mu, double* out, double* partials, int max_blocks);

// g = (1/q) sum_j a[j] Z(seed, layer_id, queries[j]) (q = 1: the two-sided a * Z).
int launch_adam(Ctx* ctx, float* C, float* m, float* v, const zoact_coeff_block* blocks, int n_blocks,
                const double* a, int q, const uint64_t* queries, float lr, float b1, float b2, float adam_eps,
                int64_t step, uint64_t seed, int sgd);

int launch_rms_norm(Ctx* ctx, const void* X, int dtype, int64_t rows, int n, float eps, void* Y);
int launch_mix_rms(Ctx* ctx, const void* q, const void* k, const void* v, int dtype, int64_t rows,
                   int n, int n_rep, int head_dim, float eps, void* Y, int64_t ld_q, int64_t ld_kv);

// Section 5.3 diagnostics (k_diag.cu): out[0] = ||Ua^T Ub||_F^2, out[2] = out[0] / ra;
// energy: out[0] = ||U^T G||_F^2, out[1] = ||G||_F^2, out[2] = their ratio.  out: device fp64 [3].
int launch_subspace_overlap(Ctx* ctx, const float* Ua, const float* Ub, int d, int ra, int rb, double* out);
int launch_gradient_energy(Ctx* ctx, const float* U, int d_in, int r, const void* G, int gdtype, int64_t n,
                           double* out);

// Data-parallel replicas (k_replica.cu): the SplitMix64-tagged sum of an arena's words; v /= world.
int launch_arena_hash(Ctx* ctx, const void* data, int64_t n_words, uint64_t* out);
int launch_mean_over_ranks(Ctx* ctx, double* v, int64_t n, int world);

int run_basis_init(Ctx* ctx, const void* X, int xdtype, int64_t n_tok, int d_in, int r, int oversample,
                   int n_iter, uint64_t seed, float* U_out, float* evals_out);

}  // namespace zoact

struct zoact_ctx : public zoact::Ctx {};
