/*
 * zoact.h -- C ABI of libzoact, the GB300 (sm_103a) hot path of one ZO-Act step.
 *
 * ZO-Act (arXiv 2607.01125) fine-tunes a frozen model forward-only: every
 * adapted linear layer keeps its weight W frozen and learns only a small
 * coefficient matrix on a frozen activation basis (Section 3):
 *
 *     y = W x + (C + sigma * eps * Z)(U^T x),      sigma in {+1, -1}
 *
 * with U [d_in, r] the top-r right singular vectors of the layer's calibration
 * activations (Algorithm 1), C [d_out, r] the coefficients (the paper's B,
 * transposed; zero at initialisation) and Z [d_out, r] ~ N(0, I) a perturbation
 * regenerated from a seed (never stored).  One ZO step (Algorithm 2, in
 * two-sided form) runs the forward pass at +eps and -eps, forms
 * a = (L+ - L-) / (2 eps) and updates C with Adam on g = a * Z.
 *
 * Conventions for every call:
 *  - All tensor pointers are DEVICE pointers owned by the caller; the library
 *    never frees caller memory and keeps no pointer after a call returns.
 *  - Every call is asynchronous on the context's stream; none synchronises with
 *    the host except zoact_get_device_status and zoact_destroy.
 *  - Errors in arguments (shape, dtype, alignment, NULL) are found on the host
 *    before any launch and returned as a negative status; nothing is launched
 *    then.  Errors found on the device (non-finite loss, a bounded wait that
 *    timed out) are recorded in the context's device status word.
 *  - Row-major layouts throughout.  "Stacked" activations hold 2T rows: rows
 *    [0, T) belong to sigma = +1 and rows [T, 2T) to sigma = -1.
 *  - Z for a layer is a pure function of (seed, layer_id, query): element
 *    e = i * r + j of Z is word (e & 3) of Philox4x32-10 with
 *    key = (seed_lo, seed_hi) and counter = (e >> 2, layer_id, query_lo, query_hi),
 *    turned into normals by Box-Muller on word pairs (w0, w1), (w2, w3) with
 *    u1 = ((w_a >> 8) + 1) 2^-24, u2 = (w_b >> 8) 2^-24, z_a = sqrt(-2 ln u1) cos(2 pi u2),
 *    z_b = sqrt(-2 ln u1) sin(2 pi u2).  The forward pass and the optimizer step
 *    must be given the same (seed, query) to see the same Z.
 */
#ifndef ZOACT_H_
#define ZOACT_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- status codes ---- */
#define ZOACT_OK               0
#define ZOACT_ERR_INVALID_ARG (-1)  /* bad shape, dtype, NULL or misaligned pointer */
#define ZOACT_ERR_UNSUPPORTED (-2)  /* valid request this build does not implement */
#define ZOACT_ERR_CUDA        (-3)  /* a CUDA runtime call failed */
#define ZOACT_ERR_NONFINITE   (-4)  /* device: a loss or the estimator scalar was NaN/Inf */
#define ZOACT_ERR_TIMEOUT     (-5)  /* device: a bounded wait in a kernel gave up */
#define ZOACT_ERR_NOMEM       (-6)  /* the context could not allocate its scratch */
#define ZOACT_ERR_TOO_LARGE   (-7)  /* request exceeds the fixed scratch of zoact_pair_forward_noalloc */

/* ---- storage types ---- */
#define ZOACT_DT_FP32       0
#define ZOACT_DT_BF16       1
#define ZOACT_DT_FP16       2
#define ZOACT_DT_INT4_G128  3  /* weights only: see zoact_layer.W */

/* ---- activations fused into the pair-forward epilogue ---- */
#define ZOACT_ACT_NONE  0
#define ZOACT_ACT_RELU  1
#define ZOACT_ACT_GELU  2  /* exact: 0.5 x (1 + erf(x / sqrt 2)) */

typedef struct zoact_ctx zoact_ctx;

/* One adapted linear layer (Section 3: W_eff = W + V_r B).  All pointers are
 * caller-owned device memory that must stay valid until the work using them
 * has run on the stream.                                                     */
typedef struct zoact_layer {
  int32_t d_in;        /* input width  (the paper's m) */
  int32_t d_out;       /* output width (the paper's n) */
  int32_t r;           /* basis rank, 1 <= r <= 256 (above 32 with 16-bit activations only when
                          the pair forward may use context scratch; see zoact_pair_forward) */
  int32_t wtype;       /* ZOACT_DT_* of W */
  const void* W;       /* frozen weight [d_out, d_in] row-major.  INT4_G128:
                          [d_out, d_in/2] bytes, element k in byte k/2, low nibble
                          for even k, 4-bit two's complement q in [-8, 7]      */
  const void* w_scales;/* INT4_G128 only: [d_out, d_in/128] fp16 scales, w = q*s;
                          NULL otherwise                                        */
  const float* U;      /* frozen basis [d_in, r] fp32 (the paper's V_r)        */
  const float* C;      /* coefficients [d_out, r] fp32 (the paper's B^T)       */
  uint32_t layer_id;   /* Philox stream id of this layer's Z; unique per layer */
} zoact_layer;

/* A block of coefficients inside the flat C/m/v arenas given to the
 * optimizer: elements [offset, offset + d_out*r) hold one layer's [d_out, r]. */
typedef struct zoact_coeff_block {
  int64_t offset;      /* element offset into the arenas; multiple of 4 */
  int32_t d_out;
  int32_t r;
  uint32_t layer_id;
  uint32_t reserved;
} zoact_coeff_block;

/* Create a context on CUDA device `device` that launches on `stream`
 * (a cudaStream_t; NULL = the legacy default stream).  The context owns only
 * scratch (projection buffer, reduction partials, basis workspace, the device
 * status word); it allocates device memory here and may grow its scratch on
 * later calls.  Returns ZOACT_OK and sets *out, or a negative status.          */
int zoact_create(zoact_ctx** out, int device, void* stream);

/* Destroy a context: synchronises its stream, frees its scratch.  NULL is a no-op. */
int zoact_destroy(zoact_ctx* ctx);

/* Change the stream later launches go to (cudaStream_t).                       */
int zoact_set_stream(zoact_ctx* ctx, void* stream);

/* Human-readable text of a status code (static storage).                       */
const char* zoact_status_string(int status);

/* Synchronise the stream and read the device status word (ZOACT_OK or the
 * first device-side error recorded since the last reset).  reset != 0 clears it.
 * On ZOACT_ERR_TIMEOUT the outputs of the launches since the last read are
 * undefined; the context's grid-reduction tickets are zeroed here, so the
 * context serves later calls normally.                                          */
int zoact_get_device_status(zoact_ctx* ctx, int* status, int reset);

/* Failure-detection test hook: one kernel that leaves every ticket of the
 * context part-counted (as a launch that gave up can), then waits for a device
 * flag that nothing sets, for at most wait_ns nanoseconds (0 < wait_ns <= 1e9),
 * and records ZOACT_ERR_TIMEOUT in the device status word.  It shows that a
 * bounded wait ends with a readable status and that zoact_get_device_status
 * repairs the tickets; nothing faults or traps.  Returns ZOACT_ERR_INVALID_ARG
 * for a wait_ns outside that range.                                              */
int zoact_debug_timeout(zoact_ctx* ctx, int64_t wait_ns);

/* Number of SMs of the context's device (host query, no launch).               */
int zoact_device_sm_count(zoact_ctx* ctx, int* sm_count);

/* Number of kernels this context has launched since it was created (a host
 * counter, incremented at every launch; no synchronisation).                   */
int zoact_get_launch_count(zoact_ctx* ctx, int64_t* count);

/* Kernel timing: with enable != 0 the context records CUDA events on its stream
 * around every tensor-core pair-forward kernel (the MMA kernel alone, without
 * the preparation kernels of the same call -- except that INT4 weights expanded
 * to bf16 first are timed with that expansion; up to 4096 launches between
 * reads, later ones are not timed and not counted).
 * Switching it on creates the event pool (ZOACT_ERR_CUDA if that fails).  The
 * events themselves lengthen a step: measure throughput with timing off.
 * zoact_kernel_timing(ctx, 0/1) switches it and forgets recorded launches;
 * zoact_kernel_time synchronises the stream and returns the summed duration (ms)
 * and the number of timed launches since the last read, then forgets them.      */
int zoact_kernel_timing(zoact_ctx* ctx, int enable);
int zoact_kernel_time(zoact_ctx* ctx, double* ms_total, int64_t* launches);

/* ---- Z: the perturbation generator (Section 3, Z ~ N(0, I)) ----
 * Writes the first n elements of the (seed, layer_id, query) stream:
 * z_out[e] (fp32 normal) and, if words_out != NULL, the raw Philox word of
 * element e.  The pair forward and the optimizer use the same device function. */
int zoact_philox_normals(zoact_ctx* ctx, uint64_t seed, uint32_t layer_id, uint64_t query,
                         int64_t n, float* z_out, uint32_t* words_out);

/* ---- the low-rank projection p = U^T x (Section 3: the factor X V_r) ----
 * X [rows, d_in] of xdtype (FP32/BF16/FP16), U [d_in, r] fp32 -> P [rows, r] fp32, r <= 256.
 * d_in % 8 == 0 for BF16/FP16, % 4 for FP32.                                    */
int zoact_lowrank_proj(zoact_ctx* ctx, const void* X, int xdtype, int64_t rows, int32_t d_in,
                       const float* U, int32_t r, float* P);

/* ---- the frozen basis in the projection's tensor-core operand form ----
 * Algorithm 1 freezes U; the tensor-core projection multiplies 16-bit X by U
 * split into three 16-bit terms (U = U0 + U1 + U2, each the rounding of what
 * the previous terms left), which keeps the product at fp32 accuracy.
 * zoact_basis_prepare writes that operand once (U_tc: zoact_basis_prepared_bytes
 * bytes of device memory, 16-byte aligned, caller-owned; xdtype BF16 or FP16 is
 * the dtype of the X it will multiply; d_in % 8 == 0) so that
 * zoact_lowrank_proj_prepared computes P = X U from it without re-splitting U.
 * U_tc must be prepared again if U changes.  zoact_basis_prepared_bytes returns -1
 * for unsupported sizes (r > 256).                                              */
int64_t zoact_basis_prepared_bytes(int32_t d_in, int32_t r);
int zoact_basis_prepare(zoact_ctx* ctx, const float* U, int32_t d_in, int32_t r, int32_t xdtype,
                        void* U_tc);
int zoact_lowrank_proj_prepared(zoact_ctx* ctx, const void* X, int xdtype, int64_t rows, int32_t d_in,
                                const void* U_tc, int32_t r, float* P);

/* ---- the pair forward (Section 3, perturbed forward pass; Algorithm 2) ----
 * Y = the stacked outputs y(+1), y(-1) of one adapted linear:
 *   input_shared == 0: X is [2T, d_in] stacked; row t of Y uses sigma(t).
 *   input_shared == 1: X is [T, d_in], the same input for both signs; W x is
 *                      computed once per row and Y rows t and T + t are written.
 * X has xdtype == the weight's compute type (FP32 for FP32 weights; BF16 for
 * BF16 and INT4_G128; FP16 for FP16).  Y [2T, d_out] of ydtype (same as xdtype,
 * or FP32).  `act` (ZOACT_ACT_*) is applied to y before it is stored.
 * P: optional [rows(X), r] fp32 projection U^T x computed earlier (e.g. by
 * zoact_lowrank_proj, or shared by layers with the same input and basis); when
 * NULL the call computes it into context scratch first.
 * Requirements: d_in % 8 == 0 (BF16/FP16), d_in % 128 == 0 (INT4), d_out % 8 == 0,
 * 16-byte aligned X, W, Y.  Ranks above 32 (16-bit X) add the whole low-rank term on
 * the tensor cores, which needs stacked rows: a shared input is first copied once
 * per sign into context scratch.                                                 */
int zoact_pair_forward(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype,
                       int64_t T, int input_shared, const float* P, float eps, uint64_t seed,
                       uint64_t query, int act, void* Y, int ydtype);

/* ---- RMS-normalised inputs without a normalisation pass ----
 * The synthetic stacks normalise a linear's input, rms(x) = x / sqrt(mean(x^2)
 * + eps) per row (zoact_rms_norm), before the next adapted linear.  That is a
 * per-row scale 1/s, and the pair forward is linear in its input:
 *     W (x/s) + (C +- eps Z) U^T (x/s) = (W x + (C +- eps Z) U^T x) / s,
 * so a pair forward can take x itself (and its projection U^T x) and scale its
 * accumulator rows.  zoact_rowscale, passed by HOST pointer, read during the call:
 *   in_scale  [rows(X)] fp32 (DEVICE, or NULL): output row t (both the W x and
 *             the low-rank terms) is multiplied by in_scale[t] before the
 *             activation / SiLU gate.
 *   out_sumsq [ceil(d_out / 64), rows(Y)] fp32 (DEVICE, or NULL): element
 *             [p][t] receives the sum of squares of Y's stored values (after
 *             rounding to ydtype) in columns [64 p, 64 p + 64) of row t, ready
 *             for zoact_rms_scale.
 * zoact_pair_forward_rs / zoact_pair_forward_gated_rs / zoact_multi_forward_rs /
 * zoact_multi_forward_gated_rs are zoact_pair_forward / _gated and
 * zoact_multi_forward / _gated (declared below) with row scales; out_sumsq then
 * has n_blocks T rows.  They apply them on the CTA-pair kernel's stacked-row
 * path only: input_shared == 0, rows(X) >= 256, 16-bit X, and INT4 weights from
 * 1024 rows; any other request returns ZOACT_ERR_UNSUPPORTED before anything is
 * launched (callers then normalise explicitly).  rs == NULL or both pointers
 * NULL is the plain call.  Relative to normalising the stored input first, the
 * outputs skip one rounding of the normalised input to the activation dtype.
 * zoact_rms_scale: inv_scale[t] = 1 / sqrt(sum_p sumsq[p][t] / n + eps) over the
 * ceil(n / 64) parts of a [ceil(n / 64), rows] array, in part order (n = the
 * producer's d_out).  The paper has no counterpart: this is how the device
 * runs the synthetic graphs' normalisations.                                    */
typedef struct zoact_rowscale {
  const float* in_scale;
  float* out_sumsq;
} zoact_rowscale;
int zoact_pair_forward_rs(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype,
                          int64_t T, int input_shared, const float* P, float eps, uint64_t seed,
                          uint64_t query, int act, void* Y, int ydtype, const zoact_rowscale* rs);
int zoact_pair_forward_gated_rs(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up,
                                const void* X, int xdtype, int64_t T, int input_shared,
                                const float* P_gate, const float* P_up, float eps, uint64_t seed,
                                uint64_t query, void* H, int ydtype, const zoact_rowscale* rs);
int zoact_rms_scale(zoact_ctx* ctx, const float* sumsq, int64_t rows, int32_t n, float eps,
                    float* inv_scale);
struct zoact_eval_blocks;
int zoact_multi_forward_rs(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype,
                           int64_t T, int input_shared, const float* P,
                           const struct zoact_eval_blocks* blocks, uint64_t seed, int act, void* Y,
                           int ydtype, const zoact_rowscale* rs);
int zoact_multi_forward_gated_rs(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up,
                                 const void* X, int xdtype, int64_t T, int input_shared,
                                 const float* P_gate, const float* P_up,
                                 const struct zoact_eval_blocks* blocks, uint64_t seed, void* H,
                                 int ydtype, const zoact_rowscale* rs);

/* ---- the pair forward without any allocation ----
 * The paper has no counterpart: this entry point exists for callers that must
 * not allocate device memory (a framework whose allocator owns all device
 * memory, a real-time loop that cannot afford a synchronising cudaMalloc, a
 * process under a hard memory budget).  It computes the pair forward of
 * zoact_pair_forward with P == NULL, on `stream` (a cudaStream_t), without a
 * context and without calling cudaMalloc, cudaFree or any allocating library
 * routine.  It adds the low-rank term from fp32 epilogue tables, so its
 * outputs agree with zoact_pair_forward within the pair forward's tolerance
 * (1e-4 of the output scale for fp32 outputs), not bit for bit.  Limits beyond
 * zoact_pair_forward's: r <= 32, and weights of type FP32, BF16 or FP16 (INT4
 * returns ZOACT_ERR_UNSUPPORTED).  Its only scratch is one file-scope device array of
 * ZOACT_NOALLOC_MAX_PROJ_FLOATS floats (4 MiB) plus a status slot, which every
 * GPU that loads the library holds until the process exits; it holds the
 * projection U^T x of the rows(X) x r inputs, so rows(X) * r above
 * ZOACT_NOALLOC_MAX_PROJ_FLOATS returns ZOACT_ERR_TOO_LARGE and launches nothing.
 * The first call on each device looks up the array's device address (with that
 * device current); make that first call before any stream capture.  The address
 * belongs to the CUDA context it was looked up in: after cudaDeviceReset (or
 * with another context current) the next call looks it up again, so that call
 * too should come before any stream capture.  All calls
 * share the array: calls that overlap on the GPU (other streams or threads)
 * race and must be ordered by the caller.  Device-side errors are not
 * reported back (there is no context); the returned status covers argument
 * and launch errors.  Other requirements (alignment, d_in and d_out multiples)
 * as for zoact_pair_forward.                                                    */
#define ZOACT_NOALLOC_MAX_PROJ_FLOATS (1 << 20)
int zoact_pair_forward_noalloc(const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                               int input_shared, float eps, uint64_t seed, uint64_t query, int act,
                               void* Y, int ydtype, void* stream);

/* ---- evaluation blocks: the forward pass at several coefficient points ----
 * Algorithm 2 evaluates each mini-batch at the unperturbed C (loss L) and at
 * C + mu Z^(j) for q independent perturbations (losses L^(j,+)).  A
 * zoact_eval_blocks lists n_blocks such points; a stacked activation then holds
 * n_blocks * T rows, rows [b T, (b + 1) T) evaluated at
 *     C + coef[b] * Z(seed, layer_id, query[b]).
 * coef[b] == 0 draws no Z (query[b] is ignored).  The paper's estimator with q
 * queries is n_blocks = q + 1, coef = {0, mu, ..., mu}, query = {-, q_1, ..., q_q};
 * the two-sided pair of zoact_pair_forward is n_blocks = 2, coef = {eps, -eps},
 * query = {q, q}.  Passed by HOST pointer; read during the call only.          */
#define ZOACT_MAX_EVAL_BLOCKS 17
typedef struct zoact_eval_blocks {
  int32_t n_blocks;                          /* 1 .. ZOACT_MAX_EVAL_BLOCKS */
  int32_t reserved;                          /* 0 */
  float coef[ZOACT_MAX_EVAL_BLOCKS];         /* finite */
  uint64_t query[ZOACT_MAX_EVAL_BLOCKS];
} zoact_eval_blocks;

/* ---- the multi-point forward (Algorithm 2: the unperturbed pass and the q
 * forward-perturbed passes of one adapted linear in one launch) ----
 * As zoact_pair_forward with the two signs replaced by the blocks of `blocks`:
 *   input_shared == 0: X is [n_blocks T, d_in]; row t of Y uses block t / T.
 *   input_shared == 1: X is [T, d_in]; W x is computed once per row and Y rows
 *                      b T + t are written for every block b.
 * Y is [n_blocks T, d_out].  Other arguments and requirements as for
 * zoact_pair_forward.                                                          */
int zoact_multi_forward(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype,
                        int64_t T, int input_shared, const float* P, const zoact_eval_blocks* blocks,
                        uint64_t seed, int act, void* Y, int ydtype);

/* ---- SiLU-gated multi-point forward: H = silu(y_gate) * y_up per block ---- */
int zoact_multi_forward_gated(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up,
                              const void* X, int xdtype, int64_t T, int input_shared,
                              const float* P_gate, const float* P_up, const zoact_eval_blocks* blocks,
                              uint64_t seed, void* H, int ydtype);

/* ---- SiLU-gated pair forward (the Llama MLP gate/up pair) ----
 * H = silu(y_gate) * y_up for both signs, with y_gate, y_up the pair forwards of
 * `gate` and `up` on the same X (same d_in, d_out, r and wtype).  H [2T, d_out]
 * of ydtype.  Gate and up keep their own U, C and layer_id (P_gate / P_up may be
 * the same pointer when the bases are equal; NULL computes them, once when gate
 * and up point at the same U).                                                 */
int zoact_pair_forward_gated(zoact_ctx* ctx, const zoact_layer* gate, const zoact_layer* up,
                             const void* X, int xdtype, int64_t T, int input_shared,
                             const float* P_gate, const float* P_up, float eps, uint64_t seed,
                             uint64_t query, void* H, int ydtype);

/* ---- adapted linears that read one input, as one launch (Section 3 perturbed
 * forward of each; Algorithm 2) ----
 * Linears with the same input have, by Algorithm 1, the same basis U, hence one
 * projection P = X U: attention's q, k and v.  Run one by one, the narrow ones
 * (k and v of a grouped-query model) leave pairs of SMs idle in their last wave;
 * run as one pair forward over their concatenated weights they do not.
 * layers[0 .. n_layers), 1 <= n_layers <= ZOACT_MAX_GROUP: the same d_in, r,
 * wtype and U (pointer), and W rows that follow one another in memory: layers[i].W
 * is layers[0].W advanced by d_out_0 + ... + d_out_{i-1} rows (INT4: the packed
 * rows and the scale rows both).  Each layer keeps its own C and layer_id, so
 * every output element is the one its layer's own pair forward computes: the
 * same Z and the same K order (a tile of a last wave whose K range is split sums
 * its pieces in fixed order, and the split can fall on other tiles than in the
 * per-layer calls: equal within rounding there).
 * X: stacked [n_blocks T, d_in] (a shared input has no grouped form).  Y
 * [n_blocks T, sum d_out] of ydtype holds the layers' outputs side by side:
 * layer i in columns [d_out_0 + ... + d_out_{i-1}, that + d_out_i).  P: optional
 * [n_blocks T, r] fp32 projection (NULL: computed once into context scratch).
 * rs: row scales as for zoact_pair_forward_rs over the sum d_out columns (NULL:
 * none).  zoact_pair_forward_group_rs evaluates the two-sided pair ({+eps, -eps},
 * one query), zoact_multi_forward_group_rs the blocks of `blocks`.
 * One launch serves the request where the kernel takes the whole low-rank term
 * from the tensor-core operand tables: stacked rows from 256 on CTA pairs, 16-bit
 * X (INT4 from 1024 rows); any other request returns ZOACT_ERR_UNSUPPORTED before
 * anything is launched, and the caller runs the layers one by one.  Layers that
 * differ in d_in, r, wtype or U, or whose W (or scales) do not follow one
 * another: ZOACT_ERR_INVALID_ARG.  n_layers == 1 is zoact_pair_forward_rs /
 * zoact_multi_forward_rs on stacked rows.                                       */
#define ZOACT_MAX_GROUP 4
int zoact_pair_forward_group_rs(zoact_ctx* ctx, const zoact_layer* layers, int32_t n_layers, const void* X,
                                int xdtype, int64_t T, const float* P, float eps, uint64_t seed,
                                uint64_t query, int act, void* Y, int ydtype, const zoact_rowscale* rs);
int zoact_multi_forward_group_rs(zoact_ctx* ctx, const zoact_layer* layers, int32_t n_layers, const void* X,
                                 int xdtype, int64_t T, const float* P, const zoact_eval_blocks* blocks,
                                 uint64_t seed, int act, void* Y, int ydtype, const zoact_rowscale* rs);

/* ---- the last pair forward fused with its loss pair (Section 3; Algorithm 2) ----
 * The losses zoact_loss_pair would return for Y = zoact_pair_forward(layer, X,
 * stacked rows, eps, seed, query, act) rounded to ydtype, computed inside the
 * pair forward's epilogue without writing Y.  X [2T, d_in] stacked (+ rows then
 * - rows), target [T, d_out] of ydtype (16-byte aligned) or NULL for the mean
 * square loss, out[4] = {L+, L-, D, a} fp64 in DEVICE memory, D = L+ - L- (the
 * difference of the two sums, each over T * d_out rounded outputs; every square
 * split exactly into two fp32 terms, compensated fp32 sums, fp64 partials: L+ and
 * L- within ~1e-11 relative of their exact values), a = D / (2 eps).  Qualifies:
 * two-sided stacked rows, T a multiple of 256, 16-bit ydtype, the CTA-pair
 * tensor-core path with the whole low-rank term on the MMA; otherwise
 * ZOACT_ERR_UNSUPPORTED is returned before
 * any launch of the pair forward itself (a projection U^T x, when P is NULL, may
 * already have run) and the caller uses zoact_pair_forward + zoact_loss_pair.
 * T = 0 writes nothing.  A non-finite result sets ZOACT_ERR_NONFINITE; a launch
 * that timed out (ZOACT_ERR_TIMEOUT) writes no loss.                            */
int zoact_pair_forward_loss(zoact_ctx* ctx, const zoact_layer* layer, const void* X, int xdtype, int64_t T,
                            const float* P, float eps, uint64_t seed, uint64_t query, int act, int ydtype,
                            const void* target, double* out);

/* ---- the loss pair (Section 3 estimator, two-sided; Algorithm 2) ----
 * Y [2T, n] stacked outputs of ydtype; target [T, n] of ydtype, or NULL for the
 * mean square loss.  Writes out[0] = L+ = mean((y+ - t)^2), out[1] = L-,
 * out[2] = D = L+ - L- (formed as mean((y+ - y-)(y+ + y- - 2t)), without
 * cancellation), out[3] = a = D / (2 eps), all fp64, to DEVICE memory out[4].
 * A non-finite result sets ZOACT_ERR_NONFINITE in the device status word.       */
int zoact_loss_pair(zoact_ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T,
                    int64_t n, float eps, double* out);

/* ---- the losses of a multi-point evaluation (Algorithm 2, one-sided) ----
 * Y [n_blocks T, n] of ydtype, block 0 the unperturbed pass; target [T, n] or
 * NULL (mean square).  Writes to DEVICE memory out[2 n_blocks - 1] (fp64):
 *   out[b]                = L_b = mean((y_b - t)^2),            b = 0 .. n_blocks-1
 *   out[n_blocks + j - 1] = a_j = (L_j - L_0) / mu,             j = 1 .. n_blocks-1
 * with L_j - L_0 formed as mean((y_j - y_0)(y_j + y_0 - 2t)), without
 * cancellation.  n_blocks >= 2, mu > 0.  A non-finite result sets
 * ZOACT_ERR_NONFINITE in the device status word.                               */
int zoact_loss_multi(zoact_ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T,
                     int64_t n, int32_t n_blocks, float mu, double* out);

/* ---- ZO-Adam (Section 3: Adam on g = a * Z; Appendix B: weight decay 0) ----
 * Updates the flat fp32 arenas C, m, v (n_total elements) in place for every
 * block: g = a * Z(seed, layer_id, query) with a = loss_out[3] (device fp64),
 *   m = b1 m + (1-b1) g;  v = b2 v + (1-b2) g^2;
 *   C -= lr * (m / (1 - b1^step)) / (sqrt(v / (1 - b2^step)) + adam_eps).
 * step is 1-based.  If a is not finite nothing is updated and the device status
 * word gets ZOACT_ERR_NONFINITE.  blocks is a HOST array of n_blocks entries.    */
int zoact_adam_step(zoact_ctx* ctx, float* C, float* m, float* v, int64_t n_total,
                    const zoact_coeff_block* blocks, int32_t n_blocks, const double* loss_out,
                    float lr, float beta1, float beta2, float adam_eps, int64_t step,
                    uint64_t seed, uint64_t query);

/* ---- ZO-SGD (Table 1, "ZO-Act Full SGD"): C -= lr * a * Z, same layout. ---- */
int zoact_sgd_step(zoact_ctx* ctx, float* C, int64_t n_total, const zoact_coeff_block* blocks,
                   int32_t n_blocks, const double* loss_out, float lr, uint64_t seed,
                   uint64_t query);

/* ---- ZO-Adam / ZO-SGD on the q-query average (Algorithm 2) ----
 * As zoact_adam_step / zoact_sgd_step with
 *   g = (1/q) sum_j a[j] * Z(seed, layer_id, queries[j]),   j = 0 .. q-1,
 * a: DEVICE fp64 [q] (e.g. zoact_loss_multi's out + n_blocks), queries: HOST
 * array of q ids, 1 <= q <= ZOACT_MAX_EVAL_BLOCKS - 1.  If any a[j] is not
 * finite nothing is updated and the device status word gets ZOACT_ERR_NONFINITE. */
int zoact_adam_step_multi(zoact_ctx* ctx, float* C, float* m, float* v, int64_t n_total,
                          const zoact_coeff_block* blocks, int32_t n_blocks, const double* a, int32_t q,
                          const uint64_t* queries, float lr, float beta1, float beta2, float adam_eps,
                          int64_t step, uint64_t seed);
int zoact_sgd_step_multi(zoact_ctx* ctx, float* C, int64_t n_total, const zoact_coeff_block* blocks,
                         int32_t n_blocks, const double* a, int32_t q, const uint64_t* queries, float lr,
                         uint64_t seed);

/* ---- the one-shot basis (Algorithm 1) ----
 * U_out [d_in, r] fp32 = the top-r right singular vectors of the calibration
 * activations X_cal [n_tok, d_in] (xdtype FP32/BF16/FP16), i.e. the top-r
 * eigenvectors of G = X^T X (uncentred), by randomised subspace iteration:
 * k = r + oversample columns, Omega from the Z generator with (seed, 0, 0)
 * (element i*k + j), Q0 = orth(Omega), Q <- orth(G Q) n_iter times, then
 * Rayleigh-Ritz.  Columns in descending eigenvalue order, each flipped so its
 * largest-magnitude entry is positive.  Optional evals_out [k] fp32 (device)
 * receives the Ritz values.  Requires k <= 512 and k <= d_in; uses d_in^2 * 4
 * bytes of context scratch.  Non-finite calibration data gives a non-finite
 * basis and sets the device status word to ZOACT_ERR_NONFINITE (a column with
 * no finite entry is left unflipped).                                          */
int zoact_basis_init(zoact_ctx* ctx, const void* X_cal, int xdtype, int64_t n_tok, int32_t d_in,
                     int32_t r, int32_t oversample, int32_t n_iter, uint64_t seed, float* U_out,
                     float* evals_out);

/* ---- subspace diagnostics (Section 5.3) ----
 * zoact_subspace_overlap: out[0] = ||U_a^T U_b||_F^2, out[1] = ||U_b||_F^2,
 *   out[2] = ||U_a^T U_b||_F^2 / r_a  (the basis-stability metric; 1 for the same
 *   subspace, 0 for orthogonal ones).  U_a [d, r_a], U_b [d, r_b] fp32 row-major.
 * zoact_gradient_energy: out[0] = ||U^T G||_F^2, out[1] = ||G||_F^2, out[2] = their
 *   ratio (the share of a weight gradient's energy inside the basis; 0 when G = 0).
 *   U [d_in, r] fp32, G [d_in, n] row-major of gdtype (FP32/BF16/FP16), i.e. the
 *   gradient of W in the paper's [d_in, d_out] orientation.
 * out: DEVICE fp64 [3].  1 <= r, r_a, r_b <= 256.  Deterministic; two launches each.  */
int zoact_subspace_overlap(zoact_ctx* ctx, const float* U_a, const float* U_b, int32_t d, int32_t r_a,
                           int32_t r_b, double* out);
int zoact_gradient_energy(zoact_ctx* ctx, const float* U, int32_t d_in, int32_t r, const void* G, int gdtype,
                          int64_t n, double* out);

/* ---- glue ops of the synthetic graphs (row-wise; activations of one dtype) ----
 * zoact_rms_norm:  Y = X / sqrt(mean(X^2, row) + eps), no gain.                  */
int zoact_rms_norm(zoact_ctx* ctx, const void* X, int dtype, int64_t rows, int32_t n, float eps,
                   void* Y);
/* zoact_mix_rms: Y = rms_norm(q + rep(k) + rep(v)) with q [rows, n], k and v
 * [rows, n / n_rep]; rep repeats each head_dim-wide kv head for n_rep
 * consecutive query heads (n_rep = 1: plain sum).                              */
int zoact_mix_rms(zoact_ctx* ctx, const void* q, const void* k, const void* v, int dtype,
                  int64_t rows, int32_t n, int32_t n_rep, int32_t head_dim, float eps, void* Y);
/* zoact_mix_rms_strided: the same with row strides in elements: row t of q at
 * q + t ld_q (ld_q >= n), of k and v at k + t ld_kv, v + t ld_kv (ld_kv >=
 * n / n_rep), e.g. column views of a zoact_pair_forward_group_rs output; Y is
 * [rows, n] contiguous.                                                        */
int zoact_mix_rms_strided(zoact_ctx* ctx, const void* q, const void* k, const void* v, int dtype,
                          int64_t rows, int32_t n, int32_t n_rep, int32_t head_dim, int64_t ld_q,
                          int64_t ld_kv, float eps, void* Y);

/* ---- data-parallel replicas ----
 * A data-parallel ZO step shares everything but the tokens: every rank holds
 * the same W, U, C, m, v and seed, runs its token shard, and the ranks
 * all-reduce the loss vector once (MeZO's property, which Section 3 keeps: Z
 * is regenerated from the seed, so C stays identical on every rank without a
 * gradient exchange).
 * zoact_mean_over_ranks: v[i] = v[i] / world for the n doubles of the
 *   all-reduced (summed) loss vector v (DEVICE): every entry is a mean over a
 *   rank's equal token share and a is linear in the losses, so the result is
 *   the whole batch's vector.  1 <= world; n >= 0.
 * zoact_arena_hash: a 64-bit fingerprint of n_words 32-bit words at `data`
 *   (DEVICE, 4-byte aligned; 16-byte aligned for full speed), written to
 *   *hash_out (DEVICE uint64):
 *       h = sum_i mix64(((i << 32) | w_i) + 0x9E3779B97F4A7C15)  mod 2^64
 *   with mix64 the output function of SplitMix64 (Steele, Lea, Flood, OOPSLA
 *   2014): z ^= z >> 30; z *= 0xBF58476D1CE4E5B9; z ^= z >> 27;
 *   z *= 0x94D049BB133111EB; z ^= z >> 31.  The same on every GPU and launch
 *   configuration (integer sums).  Replicas compare their fingerprints of C
 *   (and m, v) to detect one that diverged; ZOACT_ERR_REPLICA_MISMATCH is the
 *   status the Python layer reports then.  0 <= n_words < 2^32.
 * The paper has no counterpart of either call (it runs on one device).        */
#define ZOACT_ERR_REPLICA_MISMATCH (-8)  /* data-parallel replicas hold different coefficients */
int zoact_mean_over_ranks(zoact_ctx* ctx, double* v, int64_t n, int32_t world);
int zoact_arena_hash(zoact_ctx* ctx, const void* data, int64_t n_words, uint64_t* hash_out);

#ifdef __cplusplus
}
#endif
#endif /* ZOACT_H_ */
