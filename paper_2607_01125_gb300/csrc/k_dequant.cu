// INT4 (g128) weight -> bf16, for the staged INT4 pair forward.
//
// With many token rows the fused kernel would dequantise every weight once per
// 128-row M-tile (64 times at 8192 rows), so for large row counts the pair
// forward first expands the layer's weight into a bf16 scratch copy with this
// HBM-bound kernel (0.5 B read + 2 B written per weight) and then runs the bf16
// tensor-core kernel.  w = q * s is formed in fp32 (exact: |q| <= 8, s fp16)
// and rounded once to bf16.
#include "internal.h"

namespace zoact {
namespace {

__global__ void dequant_int4_kernel(const uint8_t* __restrict__ Wq, const __half* __restrict__ Ws,
                                    __nv_bfloat16* __restrict__ Wb, int64_t d_out, int d_in) {
  pdl_wait();                              // the previous kernel may still read the scratch copy Wb
  pdl_trigger();
  const int words_per_row = d_in / 8;                  // 8 nibbles per 32-bit word
  const int64_t n_words = d_out * words_per_row;
  const uint32_t* src = reinterpret_cast<const uint32_t*>(Wq);
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n_words;
       i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = i / words_per_row;
    const int k0 = (int)(i % words_per_row) * 8;
    const float s = __half2float(Ws[row * (d_in / 128) + k0 / 128]);
    const uint32_t w = __ldg(src + i);
    uint32_t out[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      int q0 = (int)((w >> (8 * j)) & 0xFu), q1 = (int)((w >> (8 * j + 4)) & 0xFu);
      q0 = q0 >= 8 ? q0 - 16 : q0;
      q1 = q1 >= 8 ? q1 - 16 : q1;
      __nv_bfloat162 h = __floats2bfloat162_rn((float)q0 * s, (float)q1 * s);
      out[j] = *reinterpret_cast<uint32_t*>(&h);
    }
    *reinterpret_cast<uint4*>(Wb + row * d_in + k0) = make_uint4(out[0], out[1], out[2], out[3]);
  }
}

}  // namespace

int launch_dequant_int4(Ctx* ctx, const void* Wq, const void* Ws, void* Wb, int64_t d_out, int d_in) {
  const int64_t n_words = d_out * (d_in / 8);
  int64_t blocks = (n_words + 255) / 256;
  if (blocks > 16LL * ctx->sm_count) blocks = 16LL * ctx->sm_count;
  ZOACT_CUDA_TRY(launch_pdl(ctx, dequant_int4_kernel, dim3((unsigned)blocks), dim3(256), 0,
                            static_cast<const uint8_t*>(Wq), static_cast<const __half*>(Ws),
                            static_cast<__nv_bfloat16*>(Wb), d_out, d_in));
  ++ctx->n_launch;
  return ZOACT_OK;
}

}  // namespace zoact
