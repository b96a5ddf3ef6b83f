// Glue ops of the synthetic graphs: per-row RMS normalisation (no gain) and the
// attention-free mixer rms(q + rep(k) + rep(v)).  One block per row; the row is
// read twice (sum of squares, then scale), the second time from L1/L2.
#include "internal.h"

namespace zoact {
namespace {

constexpr int GLUE_THREADS = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float s = 0.f;
  for (int w = 0; w < GLUE_THREADS / 32; ++w) s += red[w];
  return s;
}

template <typename T>
__global__ void __launch_bounds__(GLUE_THREADS)
rms_norm_kernel(const T* __restrict__ X, T* __restrict__ Y, int n, float eps) {
  __shared__ float red[GLUE_THREADS / 32];
  const int64_t row = blockIdx.x;
  const T* x = X + row * n;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) {
    const float f = to_f32<T>(x[i]);
    ss = fmaf(f, f, ss);
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)n + eps);
  T* y = Y + row * n;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) y[i] = from_f32<T>(to_f32<T>(x[i]) * inv);
}

template <typename T>
__device__ __forceinline__ float mix_at(const T* q, const T* k, const T* v, int i, int n_rep, int head_dim) {
  const int kv = (i / head_dim) / n_rep * head_dim + (i % head_dim);
  return to_f32<T>(q[i]) + to_f32<T>(k[kv]) + to_f32<T>(v[kv]);
}

template <typename T>
__global__ void __launch_bounds__(GLUE_THREADS)
mix_rms_kernel(const T* __restrict__ Q, const T* __restrict__ K, const T* __restrict__ V, T* __restrict__ Y, int n,
               int n_rep, int head_dim, float eps) {
  __shared__ float red[GLUE_THREADS / 32];
  const int64_t row = blockIdx.x;
  const int nk = n / n_rep;
  const T* q = Q + row * n;
  const T* k = K + row * nk;
  const T* v = V + row * nk;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) {
    const float f = mix_at(q, k, v, i, n_rep, head_dim);
    ss = fmaf(f, f, ss);
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)n + eps);
  T* y = Y + row * n;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) y[i] = from_f32<T>(mix_at(q, k, v, i, n_rep, head_dim) * inv);
}

}  // namespace

int launch_rms_norm(Ctx* ctx, const void* X, int dtype, int64_t rows, int n, float eps, void* Y) {
  if (rows <= 0) return ZOACT_OK;
  switch (dtype) {
    case ZOACT_DT_FP32:
      rms_norm_kernel<float><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const float*>(X), static_cast<float*>(Y), n, eps); ++ctx->n_launch;
      break;
    case ZOACT_DT_BF16:
      rms_norm_kernel<__nv_bfloat16><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const __nv_bfloat16*>(X), static_cast<__nv_bfloat16*>(Y), n, eps); ++ctx->n_launch;
      break;
    case ZOACT_DT_FP16:
      rms_norm_kernel<__half><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const __half*>(X), static_cast<__half*>(Y), n, eps); ++ctx->n_launch;
      break;
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

int launch_mix_rms(Ctx* ctx, const void* q, const void* k, const void* v, int dtype, int64_t rows, int n, int n_rep,
                   int head_dim, float eps, void* Y) {
  if (rows <= 0) return ZOACT_OK;
  switch (dtype) {
    case ZOACT_DT_FP32:
      mix_rms_kernel<float><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const float*>(q), static_cast<const float*>(k), static_cast<const float*>(v),
          static_cast<float*>(Y), n, n_rep, head_dim, eps); ++ctx->n_launch;
      break;
    case ZOACT_DT_BF16:
      mix_rms_kernel<__nv_bfloat16><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(k),
          static_cast<const __nv_bfloat16*>(v), static_cast<__nv_bfloat16*>(Y), n, n_rep, head_dim, eps); ++ctx->n_launch;
      break;
    case ZOACT_DT_FP16:
      mix_rms_kernel<__half><<<(unsigned)rows, GLUE_THREADS, 0, ctx->stream>>>(
          static_cast<const __half*>(q), static_cast<const __half*>(k), static_cast<const __half*>(v),
          static_cast<__half*>(Y), n, n_rep, head_dim, eps); ++ctx->n_launch;
      break;
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
