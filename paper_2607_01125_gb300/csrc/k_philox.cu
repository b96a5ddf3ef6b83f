// Z dump kernel: the first n elements of one (seed, layer_id, query) stream.
// Uses the same device generator as the pair forward and the optimizer.
#include "internal.h"
#include "philox.cuh"

namespace zoact {

__global__ void philox_normals_kernel(uint64_t seed, uint32_t layer_id, uint64_t query, int64_t n,
                                      float* __restrict__ z, uint32_t* __restrict__ words) {
  const int64_t n_groups = (n + 3) >> 2;
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; g < n_groups;
       g += (int64_t)gridDim.x * blockDim.x) {
    const uint4 w = z_words(seed, layer_id, query, (uint64_t)g);
    float4 v;
    box_muller(w.x, w.y, v.x, v.y);
    box_muller(w.z, w.w, v.z, v.w);
    const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
    const float zv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t e = 4 * g + i;
      if (e < n) {
        z[e] = zv[i];
        if (words) words[e] = wv[i];
      }
    }
  }
}

int launch_philox_normals(Ctx* ctx, uint64_t seed, uint32_t layer_id, uint64_t query, int64_t n,
                          float* z, uint32_t* words) {
  if (n <= 0) return ZOACT_OK;
  const int64_t n_groups = (n + 3) >> 2;
  const int threads = 256;
  int64_t blocks = (n_groups + threads - 1) / threads;
  const int64_t cap = (int64_t)ctx->sm_count * 8;
  if (blocks > cap) blocks = cap;
  philox_normals_kernel<<<(unsigned)blocks, threads, 0, ctx->stream>>>(seed, layer_id, query, n, z, words); ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
