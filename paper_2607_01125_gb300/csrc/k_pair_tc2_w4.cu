// Instantiations of the CTA-pair pair forward with INT4 weights dequantised in the kernel (stacked rows,
// whole low-rank term on the MMA, staged bf16 or fp32 output).
#include "pair_tc2_kernel.cuh"

namespace zoact {
namespace pairtc {

template <typename TO, int MODE>
static int launch_two_w4(Ctx* ctx, const TmaSet& tm, const Params& p) {
  auto kern = pair_tc2_kernel<TO, 4, MODE, 1, STAGE_ALL, true>;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM2_BYTES));
  // every pair when the tail is split (its pieces are laid out over all of them)
  const int clusters = p.sk_tiles > 0 || p.num_tiles >= ctx->sm_count / 2 ? ctx->sm_count / 2 : p.num_tiles;
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3(2 * clusters), dim3(num_threads2(true)), SMEM2_BYTES, tm, p));
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

int dispatch2_w4(Ctx* ctx, int mode, int ydtype, const TmaSet& tm, const Params& p) {
  if (p.y_staged != STAGE_ALL || p.aug_mode != LOWRANK_ALL_ON_TC || !p.Wq || !p.Ws) return ZOACT_ERR_UNSUPPORTED;
  if (mode == MODE_GATED && (!p.Wq2 || !p.Ws2)) return ZOACT_ERR_UNSUPPORTED;
  if (ydtype == ZOACT_DT_FP32)
    return mode == MODE_GATED ? launch_two_w4<float, MODE_GATED>(ctx, tm, p) : launch_two_w4<float, MODE_PAIR>(ctx, tm, p);
  if (ydtype == ZOACT_DT_BF16)
    return mode == MODE_GATED ? launch_two_w4<__nv_bfloat16, MODE_GATED>(ctx, tm, p)
                              : launch_two_w4<__nv_bfloat16, MODE_PAIR>(ctx, tm, p);
  return ZOACT_ERR_UNSUPPORTED;
}

}  // namespace pairtc
}  // namespace zoact
