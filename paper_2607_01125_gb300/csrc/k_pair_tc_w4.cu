// Instantiations of the tensor-core pair forward for INT4 (g128) weights with bf16 activations.
#include "pair_tc_kernel.cuh"

namespace zoact {
namespace pairtc {

template <typename TO, int RT, int MODE>
static int launch_one(Ctx* ctx, const CUtensorMap& a, const Params& p) {
  auto kern = pair_tc_kernel<TO, RT, MODE, 1, true>;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES));
  const int grid = p.num_tiles < ctx->sm_count ? p.num_tiles : ctx->sm_count;
  TmaSet tm;
  tm.a = tm.b = tm.b2 = tm.aa = tm.ba = tm.ba2 = tm.y = tm.y16 = a;   // only X comes by TMA
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3(grid), dim3(num_threads(true)), SMEM_BYTES, tm, p));
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

template <typename TO>
static int by_rank(Ctx* ctx, int mode, int rt, const CUtensorMap& a, const Params& p) {
  if (mode == MODE_GATED) {
    switch (rt) {
      case 4: return launch_one<TO, 4, MODE_GATED>(ctx, a, p);
      case 8: return launch_one<TO, 8, MODE_GATED>(ctx, a, p);
      case 16: return launch_one<TO, 16, MODE_GATED>(ctx, a, p);
      case 32: return launch_one<TO, 32, MODE_GATED>(ctx, a, p);
      default: return ZOACT_ERR_UNSUPPORTED;
    }
  }
  switch (rt) {
    case 4: return launch_one<TO, 4, MODE_PAIR>(ctx, a, p);
    case 8: return launch_one<TO, 8, MODE_PAIR>(ctx, a, p);
    case 16: return launch_one<TO, 16, MODE_PAIR>(ctx, a, p);
    case 32: return launch_one<TO, 32, MODE_PAIR>(ctx, a, p);
    default: return ZOACT_ERR_UNSUPPORTED;
  }
}

int dispatch_w4(Ctx* ctx, int mode, int rt, int ydtype, const CUtensorMap& a, const Params& p) {
  if (ydtype == ZOACT_DT_FP32) return by_rank<float>(ctx, mode, rt, a, p);
  return by_rank<__nv_bfloat16>(ctx, mode, rt, a, p);
}

}  // namespace pairtc
}  // namespace zoact
