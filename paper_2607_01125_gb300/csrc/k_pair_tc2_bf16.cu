// Instantiations of the CTA-pair tensor-core pair forward for bf16 inputs.
#include "pair_tc2_kernel.cuh"

namespace zoact {
namespace pairtc {

template <typename TO, int RT, int MODE, int SMODE = STAGE_NONE>
static int launch_two(Ctx* ctx, const TmaSet& tm, const Params& p) {
  auto kern = pair_tc2_kernel<TO, RT, MODE, 1, SMODE>;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM2_BYTES));
  // every pair when the tail is split (its pieces are laid out over all of them)
  const int clusters = p.sk_tiles > 0 || p.num_tiles >= ctx->sm_count / 2 ? ctx->sm_count / 2 : p.num_tiles;
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3(2 * clusters), dim3(num_threads(false)), SMEM2_BYTES, tm, p));
  ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

template <typename TO>
static int by_rank_two(Ctx* ctx, int mode, int rt, const TmaSet& tm, const Params& p) {
  // the whole low-rank term on the MMA (rank tile 4, no epilogue tables): output staged for bulk stores
  if (p.y_staged == STAGE_ALL && p.aug_mode == LOWRANK_ALL_ON_TC && rt == 4)
    return mode == MODE_GATED ? launch_two<TO, 4, MODE_GATED, STAGE_ALL>(ctx, tm, p)
                              : launch_two<TO, 4, MODE_PAIR, STAGE_ALL>(ctx, tm, p);
  // the two signs on a shared input with 16-bit outputs: both signs staged for bulk stores
  if constexpr (sizeof(TO) == 2) {
    if (p.y_staged == STAGE_LOSS)
      return mode == MODE_PAIR && rt == 4 ? launch_two<TO, 4, MODE_PAIR, STAGE_LOSS>(ctx, tm, p) : ZOACT_ERR_UNSUPPORTED;
    if (p.y_staged == STAGE_MULTI4) {
      switch (rt) {
        case 4: return mode == MODE_GATED ? launch_two<TO, 4, MODE_GATED, STAGE_MULTI4>(ctx, tm, p)
                                          : launch_two<TO, 4, MODE_PAIR, STAGE_MULTI4>(ctx, tm, p);
        case 8: return mode == MODE_GATED ? launch_two<TO, 8, MODE_GATED, STAGE_MULTI4>(ctx, tm, p)
                                          : launch_two<TO, 8, MODE_PAIR, STAGE_MULTI4>(ctx, tm, p);
        case 16: return mode == MODE_GATED ? launch_two<TO, 16, MODE_GATED, STAGE_MULTI4>(ctx, tm, p)
                                           : launch_two<TO, 16, MODE_PAIR, STAGE_MULTI4>(ctx, tm, p);
        default: return ZOACT_ERR_UNSUPPORTED;
      }
    }
    if (p.y_staged == STAGE_MIRROR4) {
      switch (rt) {
        case 4: return mode == MODE_GATED ? launch_two<TO, 4, MODE_GATED, STAGE_MIRROR4>(ctx, tm, p)
                                          : launch_two<TO, 4, MODE_PAIR, STAGE_MIRROR4>(ctx, tm, p);
        case 8: return mode == MODE_GATED ? launch_two<TO, 8, MODE_GATED, STAGE_MIRROR4>(ctx, tm, p)
                                          : launch_two<TO, 8, MODE_PAIR, STAGE_MIRROR4>(ctx, tm, p);
        case 16: return mode == MODE_GATED ? launch_two<TO, 16, MODE_GATED, STAGE_MIRROR4>(ctx, tm, p)
                                           : launch_two<TO, 16, MODE_PAIR, STAGE_MIRROR4>(ctx, tm, p);
        default: return ZOACT_ERR_UNSUPPORTED;
      }
    }
    if (p.y_staged == STAGE_MIRROR) {
      switch (rt) {
        case 4: return mode == MODE_GATED ? launch_two<TO, 4, MODE_GATED, STAGE_MIRROR>(ctx, tm, p)
                                          : launch_two<TO, 4, MODE_PAIR, STAGE_MIRROR>(ctx, tm, p);
        case 8: return mode == MODE_GATED ? launch_two<TO, 8, MODE_GATED, STAGE_MIRROR>(ctx, tm, p)
                                          : launch_two<TO, 8, MODE_PAIR, STAGE_MIRROR>(ctx, tm, p);
        case 16: return mode == MODE_GATED ? launch_two<TO, 16, MODE_GATED, STAGE_MIRROR>(ctx, tm, p)
                                           : launch_two<TO, 16, MODE_PAIR, STAGE_MIRROR>(ctx, tm, p);
        case 32: return mode == MODE_GATED ? launch_two<TO, 32, MODE_GATED, STAGE_MIRROR>(ctx, tm, p)
                                           : launch_two<TO, 32, MODE_PAIR, STAGE_MIRROR>(ctx, tm, p);
        default: return ZOACT_ERR_UNSUPPORTED;
      }
    }
  }
  if (mode == MODE_GATED) {
    switch (rt) {
      case 4: return launch_two<TO, 4, MODE_GATED>(ctx, tm, p);
      case 8: return launch_two<TO, 8, MODE_GATED>(ctx, tm, p);
      case 16: return launch_two<TO, 16, MODE_GATED>(ctx, tm, p);
      case 32: return launch_two<TO, 32, MODE_GATED>(ctx, tm, p);
      default: return ZOACT_ERR_UNSUPPORTED;
    }
  }
  switch (rt) {
    case 4: return launch_two<TO, 4, MODE_PAIR>(ctx, tm, p);
    case 8: return launch_two<TO, 8, MODE_PAIR>(ctx, tm, p);
    case 16: return launch_two<TO, 16, MODE_PAIR>(ctx, tm, p);
    case 32: return launch_two<TO, 32, MODE_PAIR>(ctx, tm, p);
    default: return ZOACT_ERR_UNSUPPORTED;
  }
}

int dispatch2_bf16(Ctx* ctx, int mode, int rt, int ydtype, const TmaSet& tm, const Params& p) {
  if (ydtype == ZOACT_DT_FP32) return by_rank_two<float>(ctx, mode, rt, tm, p);
  return by_rank_two<__nv_bfloat16>(ctx, mode, rt, tm, p);
}

}  // namespace pairtc
}  // namespace zoact
