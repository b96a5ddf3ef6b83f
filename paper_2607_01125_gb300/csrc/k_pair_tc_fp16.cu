// Instantiations of the tensor-core pair forward for fp16 inputs.
#include "pair_tc_kernel.cuh"

namespace zoact {
namespace pairtc {

template <typename TO, int RT, int MODE>
static int launch_one(Ctx* ctx, const TmaSet& tm, const Params& p) {
  auto kern = pair_tc_kernel<TO, RT, MODE, 0, false>;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES));
  const int grid = p.num_tiles < ctx->sm_count ? p.num_tiles : ctx->sm_count;
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3(grid), dim3(num_threads(false)), SMEM_BYTES, tm, p)); ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

template <typename TO>
static int by_rank(Ctx* ctx, int mode, int rt, const TmaSet& tm, const Params& p) {
  if (mode == MODE_GATED) {
    switch (rt) {
      case 4: return launch_one<TO, 4, MODE_GATED>(ctx, tm, p);
      case 8: return launch_one<TO, 8, MODE_GATED>(ctx, tm, p);
      case 16: return launch_one<TO, 16, MODE_GATED>(ctx, tm, p);
      case 32: return launch_one<TO, 32, MODE_GATED>(ctx, tm, p);
      default: return ZOACT_ERR_UNSUPPORTED;
    }
  }
  switch (rt) {
    case 4: return launch_one<TO, 4, MODE_PAIR>(ctx, tm, p);
    case 8: return launch_one<TO, 8, MODE_PAIR>(ctx, tm, p);
    case 16: return launch_one<TO, 16, MODE_PAIR>(ctx, tm, p);
    case 32: return launch_one<TO, 32, MODE_PAIR>(ctx, tm, p);
    default: return ZOACT_ERR_UNSUPPORTED;
  }
}

int dispatch_fp16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p) {
  if (mode == MODE_PLAIN) return launch_one<float, 4, MODE_PLAIN>(ctx, tm, p);
  if (ydtype == ZOACT_DT_FP32) return by_rank<float>(ctx, mode, rt, tm, p);
  return by_rank<__half>(ctx, mode, rt, tm, p);
}

}  // namespace pairtc
}  // namespace zoact
