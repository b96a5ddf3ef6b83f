// Glue ops of the synthetic graphs: per-row RMS normalisation (no gain) and the
// attention-free mixer rms(q + rep(k) + rep(v)).  One block per row.  When the
// row is a whole number of 16-byte vectors (and fits), each thread keeps its
// vectors in registers, so the row is read once and written once; otherwise a
// two-pass kernel reads it twice (the second time from L1/L2).
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
  pdl_wait();                              // the input rows written by the previous kernel
  pdl_trigger();
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
               int n_rep, int head_dim, float eps, int64_t ld_q, int64_t ld_kv) {
  pdl_wait();                              // the input rows written by the previous kernel
  pdl_trigger();
  __shared__ float red[GLUE_THREADS / 32];
  const int64_t row = blockIdx.x;
  const T* q = Q + row * ld_q;
  const T* k = K + row * ld_kv;
  const T* v = V + row * ld_kv;
  float ss = 0.f;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) {
    const float f = mix_at(q, k, v, i, n_rep, head_dim);
    ss = fmaf(f, f, ss);
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)n + eps);
  T* y = Y + row * n;
  for (int i = threadIdx.x; i < n; i += GLUE_THREADS) y[i] = from_f32<T>(mix_at(q, k, v, i, n_rep, head_dim) * inv);
}

// ---- single-pass versions: VPT 16-byte vectors per thread held in registers ----
template <typename T>
struct Vec {
  static constexpr int N = 16 / sizeof(T);           // elements per 16-byte vector
};

template <typename T>
__device__ __forceinline__ void vec_to_f32(const uint4& u, float* f) {
  const T* e = reinterpret_cast<const T*>(&u);
#pragma unroll
  for (int i = 0; i < Vec<T>::N; ++i) f[i] = to_f32<T>(e[i]);
}

template <typename T>
__device__ __forceinline__ uint4 f32_to_vec(const float* f) {
  uint4 u;
  T* e = reinterpret_cast<T*>(&u);
#pragma unroll
  for (int i = 0; i < Vec<T>::N; ++i) e[i] = from_f32<T>(f[i]);
  return u;
}

template <typename T, int VPT>
__global__ void __launch_bounds__(GLUE_THREADS)
rms_norm_reg_kernel(const T* __restrict__ X, T* __restrict__ Y, int n, float eps) {
  pdl_wait();                              // the input rows written by the previous kernel
  pdl_trigger();
  constexpr int E = Vec<T>::N;
  __shared__ float red[GLUE_THREADS / 32];
  const int64_t row = blockIdx.x;
  const uint4* x = reinterpret_cast<const uint4*>(X + row * n);
  const int nv = n / E;
  float v[VPT][E];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int idx = threadIdx.x + j * GLUE_THREADS;
    if (idx < nv) {
      vec_to_f32<T>(__ldg(x + idx), v[j]);
#pragma unroll
      for (int i = 0; i < E; ++i) ss = fmaf(v[j][i], v[j][i], ss);
    }
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)n + eps);
  uint4* y = reinterpret_cast<uint4*>(Y + row * n);
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int idx = threadIdx.x + j * GLUE_THREADS;
    if (idx < nv) {
#pragma unroll
      for (int i = 0; i < E; ++i) v[j][i] *= inv;
      y[idx] = f32_to_vec<T>(v[j]);
    }
  }
}

template <typename T, int VPT>
__global__ void __launch_bounds__(GLUE_THREADS)
mix_rms_reg_kernel(const T* __restrict__ Q, const T* __restrict__ K, const T* __restrict__ V, T* __restrict__ Y,
                   int n, int n_rep, int head_dim, float eps, int64_t ld_q, int64_t ld_kv) {
  pdl_wait();                              // the input rows written by the previous kernel
  pdl_trigger();
  constexpr int E = Vec<T>::N;
  __shared__ float red[GLUE_THREADS / 32];
  const int64_t row = blockIdx.x;
  const uint4* q = reinterpret_cast<const uint4*>(Q + row * ld_q);
  const T* k = K + row * ld_kv;
  const T* v = V + row * ld_kv;
  const int nv = n / E;
  float m[VPT][E];
  float ss = 0.f;
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int idx = threadIdx.x + j * GLUE_THREADS;
    if (idx < nv) {
      const int i0 = idx * E;                            // head_dim % E == 0: one kv head per vector
      const int kv = (i0 / head_dim) / n_rep * head_dim + (i0 % head_dim);
      float a[E], b[E];
      vec_to_f32<T>(__ldg(q + idx), m[j]);
      vec_to_f32<T>(__ldg(reinterpret_cast<const uint4*>(k + kv)), a);
      vec_to_f32<T>(__ldg(reinterpret_cast<const uint4*>(v + kv)), b);
#pragma unroll
      for (int i = 0; i < E; ++i) {
        m[j][i] = m[j][i] + a[i] + b[i];
        ss = fmaf(m[j][i], m[j][i], ss);
      }
    }
  }
  const float inv = rsqrtf(block_sum(ss, red) / (float)n + eps);
  uint4* y = reinterpret_cast<uint4*>(Y + row * n);
#pragma unroll
  for (int j = 0; j < VPT; ++j) {
    const int idx = threadIdx.x + j * GLUE_THREADS;
    if (idx < nv) {
#pragma unroll
      for (int i = 0; i < E; ++i) m[j][i] *= inv;
      y[idx] = f32_to_vec<T>(m[j]);
    }
  }
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

// vectors per thread for a row of n elements, or 0 when the register path does not apply
template <typename T>
int reg_vpt(int n) {
  constexpr int E = Vec<T>::N;
  if (n % E != 0) return 0;
  const int vecs = n / E;
  const int vpt = (vecs + GLUE_THREADS - 1) / GLUE_THREADS;
  if (vpt <= 2) return 2;
  if (vpt <= 4) return 4;
  if (vpt <= 8) return 8;
  if (vpt <= 12) return 12;
  return 0;
}

template <typename T>
int rms_dispatch(Ctx* ctx, const T* X, T* Y, int64_t rows, int n, float eps) {
  const int vpt = (aligned16(X) && aligned16(Y)) ? reg_vpt<T>(n) : 0;
  void (*kern)(const T*, T*, int, float) = rms_norm_kernel<T>;
  switch (vpt) {
    case 2: kern = rms_norm_reg_kernel<T, 2>; break;
    case 4: kern = rms_norm_reg_kernel<T, 4>; break;
    case 8: kern = rms_norm_reg_kernel<T, 8>; break;
    case 12: kern = rms_norm_reg_kernel<T, 12>; break;
    default: break;
  }
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3((unsigned)rows), dim3(GLUE_THREADS), 0, X, Y, n, eps));
  ++ctx->n_launch;
  return ZOACT_OK;
}

template <typename T>
int mix_dispatch(Ctx* ctx, const T* q, const T* k, const T* v, T* Y, int64_t rows, int n, int n_rep, int head_dim,
                 float eps, int64_t ld_q, int64_t ld_kv) {
  constexpr int E = Vec<T>::N;
  // 16-byte vectors need every row of q, k and v to start on a 16-byte boundary
  const bool ok = aligned16(q) && aligned16(k) && aligned16(v) && aligned16(Y) && head_dim % E == 0 &&
                  (n / n_rep) % E == 0 && ld_q % E == 0 && ld_kv % E == 0;
  const int vpt = ok ? reg_vpt<T>(n) : 0;
  void (*kern)(const T*, const T*, const T*, T*, int, int, int, float, int64_t, int64_t) = mix_rms_kernel<T>;
  switch (vpt) {
    case 2: kern = mix_rms_reg_kernel<T, 2>; break;
    case 4: kern = mix_rms_reg_kernel<T, 4>; break;
    case 8: kern = mix_rms_reg_kernel<T, 8>; break;
    case 12: kern = mix_rms_reg_kernel<T, 12>; break;
    default: break;
  }
  ZOACT_CUDA_TRY(launch_pdl(ctx, kern, dim3((unsigned)rows), dim3(GLUE_THREADS), 0, q, k, v, Y, n, n_rep, head_dim,
                            eps, ld_q, ld_kv));
  ++ctx->n_launch;
  return ZOACT_OK;
}

// 1/s per row from the per-part sums of squares a pair forward's epilogue wrote: 32 rows per block (one per
// lane), the parts split over the 8 warps (warp w takes parts w, w + 8, ...), the 8 warp sums added in warp
// order -- a fixed order, so the result is bit-reproducible.
constexpr int RS_WARPS = 8;
__global__ void __launch_bounds__(32 * RS_WARPS)
rms_scale_kernel(const float* __restrict__ parts, int64_t rows, int n_parts, int n, float eps, float* __restrict__ inv) {
  pdl_wait();                              // the partial sums written by the previous kernel
  pdl_trigger();
  __shared__ float red[RS_WARPS][32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t t = (int64_t)blockIdx.x * 32 + lane;
  float s = 0.f;
  if (t < rows) {
#pragma unroll 4
    for (int p = warp; p < n_parts; p += RS_WARPS) s += __ldg(parts + (int64_t)p * rows + t);
  }
  red[warp][lane] = s;
  __syncthreads();
  if (warp == 0 && t < rows) {
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < RS_WARPS; ++w) tot += red[w][lane];
    inv[t] = rsqrtf(tot / (float)n + eps);
  }
}

}  // namespace

int launch_rms_scale(Ctx* ctx, const float* parts, int64_t rows, int n, float eps, float* inv) {
  if (rows <= 0) return ZOACT_OK;
  const int64_t blocks = (rows + 31) / 32;
  if (blocks > 0x7fffffff) return ZOACT_ERR_UNSUPPORTED;
  ZOACT_CUDA_TRY(launch_pdl(ctx, rms_scale_kernel, dim3((unsigned)blocks), dim3(32 * RS_WARPS), 0, parts, rows,
                            (n + 63) / 64, n, eps, inv));
  ++ctx->n_launch;
  return ZOACT_OK;
}

int launch_rms_norm(Ctx* ctx, const void* X, int dtype, int64_t rows, int n, float eps, void* Y) {
  if (rows <= 0) return ZOACT_OK;
  switch (dtype) {
    case ZOACT_DT_FP32:
      return rms_dispatch(ctx, static_cast<const float*>(X), static_cast<float*>(Y), rows, n, eps);
    case ZOACT_DT_BF16:
      return rms_dispatch(ctx, static_cast<const __nv_bfloat16*>(X), static_cast<__nv_bfloat16*>(Y), rows, n, eps);
    case ZOACT_DT_FP16:
      return rms_dispatch(ctx, static_cast<const __half*>(X), static_cast<__half*>(Y), rows, n, eps);
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
}

int launch_mix_rms(Ctx* ctx, const void* q, const void* k, const void* v, int dtype, int64_t rows, int n, int n_rep,
                   int head_dim, float eps, void* Y, int64_t ld_q, int64_t ld_kv) {
  if (rows <= 0) return ZOACT_OK;
  switch (dtype) {
    case ZOACT_DT_FP32:
      return mix_dispatch(ctx, static_cast<const float*>(q), static_cast<const float*>(k),
                          static_cast<const float*>(v), static_cast<float*>(Y), rows, n, n_rep, head_dim, eps, ld_q,
                          ld_kv);
    case ZOACT_DT_BF16:
      return mix_dispatch(ctx, static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(k),
                          static_cast<const __nv_bfloat16*>(v), static_cast<__nv_bfloat16*>(Y), rows, n, n_rep,
                          head_dim, eps, ld_q, ld_kv);
    case ZOACT_DT_FP16:
      return mix_dispatch(ctx, static_cast<const __half*>(q), static_cast<const __half*>(k),
                          static_cast<const __half*>(v), static_cast<__half*>(Y), rows, n, n_rep, head_dim, eps, ld_q,
                          ld_kv);
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
}

}  // namespace zoact
