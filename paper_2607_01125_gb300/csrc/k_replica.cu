// Data-parallel replicas: the fingerprint of a coefficient arena and the rank mean of the loss vector.
//
// In a data-parallel ZO step every rank holds the same C, m, v and applies the same update with the same
// regenerated Z, so the arenas stay bit-identical without a gradient exchange; the only exchange is one
// all-reduce of the loss vector.  Two kernels support that:
//
//  * arena_hash_kernel: h = sum_i mix64(((i << 32) | w_i) + GAMMA) mod 2^64 over the arena's 32-bit words
//    w_i, with mix64 the output function of SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom
//    number generators", OOPSLA 2014) and GAMMA its golden-ratio increment.  Every word is tagged with its
//    index, so a moved or changed word changes h; integer addition mod 2^64 is associative and commutative,
//    so the sum is the same whatever the order the blocks finish in.  Ranks compare their h to find a
//    diverged replica.
//  * mean_over_ranks_kernel: the all-reduced sum of the loss vector divided by the number of ranks (each
//    entry is a mean over a rank's equal share of the tokens, and a is linear in the losses, so the mean of
//    the ranks' vectors is the whole batch's).
#include "internal.h"

namespace zoact {
namespace {

constexpr uint64_t SM64_GAMMA = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

constexpr int HASH_THREADS = 256;

// Grid-stride over 16-byte vectors of the word array (a ragged tail of < 4 words by thread 0 of block 0),
// per-thread sums, a warp and block reduction, one 64-bit atomic add per block into *out (zeroed before).
__global__ void __launch_bounds__(HASH_THREADS) arena_hash_kernel(const uint32_t* __restrict__ w, int64_t n,
                                                                  unsigned long long* out) {
  pdl_wait();
  pdl_trigger();
  uint64_t h = 0;
  const int64_t n4 = n / 4;
  const uint4* w4 = reinterpret_cast<const uint4*>(w);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < n4; v += stride) {
    const uint4 q = __ldg(w4 + v);
    const uint64_t i = (uint64_t)v * 4;
    h += mix64(((i << 32) | q.x) + SM64_GAMMA);
    h += mix64((((i + 1) << 32) | q.y) + SM64_GAMMA);
    h += mix64((((i + 2) << 32) | q.z) + SM64_GAMMA);
    h += mix64((((i + 3) << 32) | q.w) + SM64_GAMMA);
  }
  if (blockIdx.x == 0 && threadIdx.x == 0)
    for (int64_t i = n4 * 4; i < n; ++i) h += mix64((((uint64_t)i << 32) | w[i]) + SM64_GAMMA);
  for (int o = 16; o > 0; o >>= 1) h += __shfl_xor_sync(0xffffffffu, h, o);
  __shared__ uint64_t warp_sum[HASH_THREADS / 32];
  if ((threadIdx.x & 31) == 0) warp_sum[threadIdx.x >> 5] = h;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint64_t s = 0;
    for (int k = 0; k < HASH_THREADS / 32; ++k) s += warp_sum[k];
    atomicAdd(out, (unsigned long long)s);
  }
}

__global__ void mean_over_ranks_kernel(double* v, int64_t n, int world) {
  pdl_wait();
  pdl_trigger();
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
    v[i] = v[i] / (double)world;
}

}  // namespace

int launch_arena_hash(Ctx* ctx, const void* data, int64_t n_words, uint64_t* out) {
  ZOACT_CUDA_TRY(cudaMemsetAsync(out, 0, sizeof(uint64_t), ctx->stream));
  if (n_words == 0) return ZOACT_OK;
  const int64_t vecs = n_words / 4;
  const int64_t want = (vecs + HASH_THREADS - 1) / HASH_THREADS;
  const int blocks = (int)(want < 1 ? 1 : want > 8 * (int64_t)ctx->sm_count ? 8 * (int64_t)ctx->sm_count : want);
  ZOACT_CUDA_TRY(launch_pdl(ctx, arena_hash_kernel, dim3(blocks), dim3(HASH_THREADS), 0,
                            static_cast<const uint32_t*>(data), n_words,
                            reinterpret_cast<unsigned long long*>(out)));
  ++ctx->n_launch;
  return ZOACT_OK;
}

int launch_mean_over_ranks(Ctx* ctx, double* v, int64_t n, int world) {
  if (n == 0) return ZOACT_OK;
  const int blocks = (int)((n + 255) / 256 < 64 ? (n + 255) / 256 : 64);
  ZOACT_CUDA_TRY(launch_pdl(ctx, mean_over_ranks_kernel, dim3(blocks), dim3(256), 0, v, n, world));
  ++ctx->n_launch;
  return ZOACT_OK;
}

}  // namespace zoact
