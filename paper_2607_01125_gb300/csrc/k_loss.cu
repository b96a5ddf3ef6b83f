// Loss pair and estimator scalar (Section 3 estimator in two-sided form; Algorithm 2):
//   L+ = mean((y+ - t)^2),  L- = mean((y- - t)^2),
//   D  = mean((y+ - y-)(y+ + y- - 2t))   (= L+ - L-, without cancellation),
//   a  = D / (2 eps).
// One pass over the stacked outputs (HBM-bound).  Each thread reads 16-byte
// vectors of y+, y- and t (kept as raw words until used; 64 registers, four
// 256-thread blocks per SM), sums a round of two vectors' terms (16 per
// accumulator) in fp32 and adds the round's sum to a compensated fp32 running
// sum (fp64 units are scarce on this part); each block adds its threads' sums
// in fp64 in a fixed order, writes the block partials to scratch, and the last
// block to finish (an atomic ticket) adds the partials in block order, so the
// result is deterministic.  The ticket is reset by that
// block, leaving the scratch ready for the next call.
#include "internal.h"

namespace zoact {
namespace {

constexpr int LOSS_THREADS = 256;

__device__ __forceinline__ void unpack2(uint32_t w, float* out, const __nv_bfloat16*) {
  out[0] = __uint_as_float(w << 16);
  out[1] = __uint_as_float(w & 0xffff0000u);
}
__device__ __forceinline__ void unpack2(uint32_t w, float* out, const __half*) {
  const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w));
  out[0] = f.x;
  out[1] = f.y;
}

// 8 consecutive elements as raw 16-byte words (unpacked only when used, so a
// round of loads in flight costs 4 registers per 8 elements of 16-bit data)
template <typename TY> struct Raw8 { uint4 w; };
template <> struct Raw8<float> { float4 a, b; };

template <typename TY>
__device__ __forceinline__ Raw8<TY> ld8(const TY* p) {
  Raw8<TY> r;
  r.w = __ldg(reinterpret_cast<const uint4*>(p));
  return r;
}
template <>
__device__ __forceinline__ Raw8<float> ld8<float>(const float* p) {
  Raw8<float> r;
  r.a = __ldg(reinterpret_cast<const float4*>(p));
  r.b = __ldg(reinterpret_cast<const float4*>(p + 4));
  return r;
}
template <typename TY>
__device__ __forceinline__ void unpack8(const Raw8<TY>& r, float* out) {
  unpack2(r.w.x, out + 0, (const TY*)nullptr);
  unpack2(r.w.y, out + 2, (const TY*)nullptr);
  unpack2(r.w.z, out + 4, (const TY*)nullptr);
  unpack2(r.w.w, out + 6, (const TY*)nullptr);
}
template <>
__device__ __forceinline__ void unpack8<float>(const Raw8<float>& r, float* out) {
  out[0] = r.a.x; out[1] = r.a.y; out[2] = r.a.z; out[3] = r.a.w;
  out[4] = r.b.x; out[5] = r.b.y; out[6] = r.b.z; out[7] = r.b.w;
}

template <typename TY>
__device__ __forceinline__ void load8(const TY* p, float* out) {
  const uint4 raw = __ldg(reinterpret_cast<const uint4*>(p));
  unpack2(raw.x, out + 0, p);
  unpack2(raw.y, out + 2, p);
  unpack2(raw.z, out + 4, p);
  unpack2(raw.w, out + 6, p);
}
template <>
__device__ __forceinline__ void load8<float>(const float* p, float* out) {
  const float4 a = *reinterpret_cast<const float4*>(p);
  const float4 b = *reinterpret_cast<const float4*>(p + 4);
  out[0] = a.x; out[1] = a.y; out[2] = a.z; out[3] = a.w;
  out[4] = b.x; out[5] = b.y; out[6] = b.z; out[7] = b.w;
}

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// A running sum in fp32 with Neumaier compensation: s + c carries the sum of the
// added values to about twice fp32 precision, without the scarce fp64 units.
struct CSum {
  float s = 0.f, c = 0.f;
  __device__ __forceinline__ void add(float x) {
    const float t = s + x;
    c += fabsf(s) >= fabsf(x) ? (s - t) + x : (x - t) + s;
    s = t;
  }
  __device__ __forceinline__ double value() const { return (double)s + (double)c; }
};

// Sum v over the block's threads in fp64 (one conversion per thread; warp 0 adds the
// per-thread values in a fixed order).  Result valid in thread 0.
template <int NV>
__device__ __forceinline__ void block_sum(const double (&v)[NV], double (&out)[NV], double (*sm)[LOSS_THREADS]) {
#pragma unroll
  for (int i = 0; i < NV; ++i) sm[i][threadIdx.x] = v[i];
  __syncthreads();
  if (threadIdx.x < 32) {
#pragma unroll
    for (int i = 0; i < NV; ++i) {
      double a = 0.0;
      for (int t = threadIdx.x; t < LOSS_THREADS; t += 32) a += sm[i][t];
      out[i] = warp_sum(a);
    }
  }
}

template <typename TY>
__global__ void __launch_bounds__(LOSS_THREADS, 4)
loss_pair_kernel(const TY* __restrict__ Y, const TY* __restrict__ tgt, int64_t count, int vec_ok, float eps,
                 double* __restrict__ out, double* __restrict__ partials, unsigned int* __restrict__ ticket,
                 int* __restrict__ status) {
  pdl_wait();                              // Y written by the previous kernel
  pdl_trigger();
  const TY* yp = Y;
  const TY* ym = Y + count;
  CSum ap, am, ad;
  // 16-byte vectors need y+, y- and t 16-byte aligned (host checks the bases;
  // y- = y+ + count is aligned when count % 8 == 0)
  const int64_t n_vec = vec_ok ? count / 8 : 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  // R vectors per round, all of their 16-byte loads issued before any use
  constexpr int R = sizeof(TY) == 4 ? 1 : 2;   // vectors per round (fp32 words take twice the registers)
  for (; v + (R - 1) * stride < n_vec; v += R * stride) {
    Raw8<TY> rp[R], rm[R], rt[R];
#pragma unroll
    for (int u = 0; u < R; ++u) {
      rp[u] = ld8<TY>(yp + 8 * (v + u * stride));
      rm[u] = ld8<TY>(ym + 8 * (v + u * stride));
      if (tgt) rt[u] = ld8<TY>(tgt + 8 * (v + u * stride));
    }
    float sp = 0.f, sm = 0.f, sd = 0.f;
#pragma unroll
    for (int u = 0; u < R; ++u) {
      float p[8], m[8], t[8];
      unpack8<TY>(rp[u], p);
      unpack8<TY>(rm[u], m);
      if (tgt) {
        unpack8<TY>(rt[u], t);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) t[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float dp = p[i] - t[i], dm = m[i] - t[i];
        sp = fmaf(dp, dp, sp);
        sm = fmaf(dm, dm, sm);
        sd = fmaf(p[i] - m[i], dp + dm, sd);
      }
    }
    ap.add(sp); am.add(sm); ad.add(sd);
  }
  for (; v < n_vec; v += stride) {
    float p[8], m[8], t[8];
    load8<TY>(yp + 8 * v, p);
    load8<TY>(ym + 8 * v, m);
    if (tgt) {
      load8<TY>(tgt + 8 * v, t);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) t[i] = 0.f;
    }
    float sp = 0.f, sm = 0.f, sd = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float dp = p[i] - t[i], dm = m[i] - t[i];
      sp = fmaf(dp, dp, sp);
      sm = fmaf(dm, dm, sm);
      sd = fmaf(p[i] - m[i], dp + dm, sd);
    }
    ap.add(sp); am.add(sm); ad.add(sd);
  }
  // scalar remainder (everything when the vector path is off)
  for (int64_t i = 8 * n_vec + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < count; i += stride) {
    const float tv = tgt ? to_f32<TY>(tgt[i]) : 0.f;
    const float dp = to_f32<TY>(yp[i]) - tv, dm = to_f32<TY>(ym[i]) - tv;
    ap.add(dp * dp); am.add(dm * dm);
    ad.add((to_f32<TY>(yp[i]) - to_f32<TY>(ym[i])) * (dp + dm));
  }
  __shared__ double tree[3][LOSS_THREADS];
  __shared__ bool is_last;
  double bs[3];
  block_sum<3>({ap.value(), am.value(), ad.value()}, bs, tree);
  if (threadIdx.x == 0) {
    const double s0 = bs[0], s1 = bs[1], s2 = bs[2];
    partials[3 * blockIdx.x + 0] = s0;
    partials[3 * blockIdx.x + 1] = s1;
    partials[3 * blockIdx.x + 2] = s2;
    __threadfence();
    const unsigned int prev = atomicAdd(ticket, 1u);
    is_last = (prev == gridDim.x - 1);
  }
  __syncthreads();
  if (!is_last) return;
  // the last block adds the partials: thread t takes blocks t, t + 256, ... in order, then a fixed
  // shared-memory tree combines the threads, so the result does not depend on scheduling
  __threadfence();
  double s0 = 0.0, s1 = 0.0, s2 = 0.0;
  for (unsigned int b = threadIdx.x; b < gridDim.x; b += LOSS_THREADS) {
    s0 += __ldcg(partials + 3 * b);
    s1 += __ldcg(partials + 3 * b + 1);
    s2 += __ldcg(partials + 3 * b + 2);
  }
  __syncthreads();                 // the block sum's readers of `tree` are done
  tree[0][threadIdx.x] = s0; tree[1][threadIdx.x] = s1; tree[2][threadIdx.x] = s2;
  __syncthreads();
  for (int h = LOSS_THREADS / 2; h > 0; h >>= 1) {
    if (threadIdx.x < h) {
      tree[0][threadIdx.x] += tree[0][threadIdx.x + h];
      tree[1][threadIdx.x] += tree[1][threadIdx.x + h];
      tree[2][threadIdx.x] += tree[2][threadIdx.x + h];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    const double inv = 1.0 / (double)count;
    const double Lp = tree[0][0] * inv, Lm = tree[1][0] * inv, D = tree[2][0] * inv;
    const double a = D / (2.0 * (double)eps);
    out[0] = Lp; out[1] = Lm; out[2] = D; out[3] = a;
    if (!isfinite(Lp) || !isfinite(Lm) || !isfinite(a)) record_error(status, ZOACT_ERR_NONFINITE);
    *ticket = 0u;
  }
}

template <typename TY>
int loss_dispatch(Ctx* ctx, const TY* Y, const TY* tgt, int64_t count, float eps, double* out,
                  double* partials, int max_blocks, unsigned int* ticket) {
  const int vec_ok = (count % 8 == 0) && ((uintptr_t)Y % 16 == 0) && ((uintptr_t)tgt % 16 == 0);
  int64_t blocks = ((vec_ok ? count / 8 : count) + LOSS_THREADS - 1) / LOSS_THREADS;
  if (blocks < 1) blocks = 1;
  if (blocks > max_blocks) blocks = max_blocks;
  ZOACT_CUDA_TRY(launch_pdl(ctx, loss_pair_kernel<TY>, dim3((unsigned)blocks), dim3(LOSS_THREADS), 0, Y, tgt, count,
                            vec_ok, eps, out, partials, ticket, ctx->d_status));
  ++ctx->n_launch;
  return ZOACT_OK;
}

// Losses of a multi-point evaluation (Algorithm 2, one-sided, q queries):
//   L_b = mean((y_b - t)^2) for every block b,
//   D_j = mean((y_j - y_0)(y_j + y_0 - 2t)) (= L_j - L_0),  a_j = D_j / mu.
// blockIdx.y is the block b; each CTA reads y_b, y_0 and t over its share of
// the elements (y_0 and t are re-read once per block, from L2 when they fit).
// Partials [nb][gridDim.x][2] are added in a fixed order by the last CTA.
template <typename TY>
__global__ void __launch_bounds__(LOSS_THREADS, 4)
loss_multi_kernel(const TY* __restrict__ Y, const TY* __restrict__ tgt, int64_t count, int vec_ok, int nb, float mu,
                  double* __restrict__ out, double* __restrict__ partials, unsigned int* __restrict__ ticket,
                  int* __restrict__ status) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y;
  const TY* yb = Y + (int64_t)b * count;
  const TY* y0 = Y;
  CSum as, ad;
  const int64_t n_vec = vec_ok ? count / 8 : 0;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  const int64_t first = blockIdx.x * (int64_t)blockDim.x + threadIdx.x;
  // rounds of two vectors, all loads issued first; one compensated add per accumulator per round
  int64_t v = first;
  constexpr int R = sizeof(TY) == 4 ? 1 : 2;   // vectors per round (fp32 words take twice the registers)
  for (; v + (R - 1) * stride < n_vec; v += R * stride) {
    Raw8<TY> ry[R], rz[R], rt[R];
#pragma unroll
    for (int u = 0; u < R; ++u) {
      ry[u] = ld8<TY>(yb + 8 * (v + u * stride));
      if (b > 0) rz[u] = ld8<TY>(y0 + 8 * (v + u * stride));
      if (tgt) rt[u] = ld8<TY>(tgt + 8 * (v + u * stride));
    }
    float ss = 0.f, sd = 0.f;
#pragma unroll
    for (int u = 0; u < R; ++u) {
      float y[8], z[8], t[8];
      unpack8<TY>(ry[u], y);
      if (b > 0) unpack8<TY>(rz[u], z);
      if (tgt) {
        unpack8<TY>(rt[u], t);
      } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) t[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float dy = y[i] - t[i];
        ss = fmaf(dy, dy, ss);
        if (b > 0) sd = fmaf(y[i] - z[i], dy + (z[i] - t[i]), sd);
      }
    }
    as.add(ss); ad.add(sd);
  }
  for (; v < n_vec; v += stride) {
    float y[8], z[8], t[8];
    load8<TY>(yb + 8 * v, y);
    if (b > 0) load8<TY>(y0 + 8 * v, z);
    if (tgt) {
      load8<TY>(tgt + 8 * v, t);
    } else {
#pragma unroll
      for (int i = 0; i < 8; ++i) t[i] = 0.f;
    }
    float ss = 0.f, sd = 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float dy = y[i] - t[i];
      ss = fmaf(dy, dy, ss);
      if (b > 0) sd = fmaf(y[i] - z[i], dy + (z[i] - t[i]), sd);
    }
    as.add(ss); ad.add(sd);
  }
  for (int64_t i = 8 * n_vec + first; i < count; i += stride) {
    const float tv = tgt ? to_f32<TY>(tgt[i]) : 0.f;
    const float yv = to_f32<TY>(yb[i]);
    const float dy = yv - tv;
    as.add(dy * dy);
    if (b > 0) {
      const float zv = to_f32<TY>(y0[i]);
      ad.add((yv - zv) * (dy + (zv - tv)));
    }
  }
  __shared__ double red[2][LOSS_THREADS];
  __shared__ bool is_last;
  double bs[2];
  block_sum<2>({as.value(), ad.value()}, bs, red);
  if (threadIdx.x == 0) {
    const double s0 = bs[0], s1 = bs[1];
    double* pb = partials + 2 * ((int64_t)b * gridDim.x + blockIdx.x);
    pb[0] = s0;
    pb[1] = s1;
    __threadfence();
    const unsigned int prev = atomicAdd(ticket, 1u);
    is_last = (prev == gridDim.x * gridDim.y - 1);
  }
  __syncthreads();
  if (!is_last) return;
  __threadfence();
  __shared__ double tree[2][LOSS_THREADS];
  const double inv = 1.0 / (double)count;
  bool finite = true;
  for (int bb = 0; bb < nb; ++bb) {
    double s0 = 0.0, s1 = 0.0;
    for (unsigned int x = threadIdx.x; x < gridDim.x; x += LOSS_THREADS) {
      const double* pb = partials + 2 * ((int64_t)bb * gridDim.x + x);
      s0 += __ldcg(pb);
      s1 += __ldcg(pb + 1);
    }
    tree[0][threadIdx.x] = s0; tree[1][threadIdx.x] = s1;
    __syncthreads();
    for (int h = LOSS_THREADS / 2; h > 0; h >>= 1) {
      if (threadIdx.x < h) {
        tree[0][threadIdx.x] += tree[0][threadIdx.x + h];
        tree[1][threadIdx.x] += tree[1][threadIdx.x + h];
      }
      __syncthreads();
    }
    if (threadIdx.x == 0) {
      const double L = tree[0][0] * inv;
      out[bb] = L;
      finite = finite && isfinite(L);
      if (bb > 0) {
        const double a = tree[1][0] * inv / (double)mu;
        out[nb + bb - 1] = a;
        finite = finite && isfinite(a);
      }
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    if (!finite) record_error(status, ZOACT_ERR_NONFINITE);
    *ticket = 0u;
  }
}

template <typename TY>
int loss_multi_dispatch(Ctx* ctx, const TY* Y, const TY* tgt, int64_t count, int nb, float mu, double* out,
                        double* partials, int max_blocks, unsigned int* ticket) {
  const int vec_ok = (count % 8 == 0) && ((uintptr_t)Y % 16 == 0) && ((uintptr_t)tgt % 16 == 0);
  int64_t bx = ((vec_ok ? count / 8 : count) + LOSS_THREADS - 1) / LOSS_THREADS;
  if (bx < 1) bx = 1;
  int64_t cap = max_blocks / nb;
  if (cap < 1) cap = 1;
  if (bx > cap) bx = cap;
  dim3 grid((unsigned)bx, (unsigned)nb);
  ZOACT_CUDA_TRY(launch_pdl(ctx, loss_multi_kernel<TY>, grid, dim3(LOSS_THREADS), 0, Y, tgt, count, vec_ok, nb, mu,
                            out, partials, ticket, ctx->d_status));
  ++ctx->n_launch;
  return ZOACT_OK;
}

}  // namespace

// Two blocks per SM: the reduction tail (block sums, the ticket, the last block's pass over the
// partials) grows with the block count and outweighs the extra loads in flight of a larger grid
// (measured on the 4096 x 4096 bf16 MLP output: 13.6 us at 2 per SM, 14.4 at 4, 20.4 at 8).
int loss_pair_max_blocks(Ctx* ctx) { return 2 * ctx->sm_count; }

int launch_loss_multi(Ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n, int nb, float mu,
                      double* out, double* partials, int max_blocks) {
  const int64_t count = T * n;
  unsigned int* ticket = ctx->d_tickets;
  switch (ydtype) {
    case ZOACT_DT_FP32:
      return loss_multi_dispatch(ctx, static_cast<const float*>(Y), static_cast<const float*>(target), count, nb, mu,
                                 out, partials, max_blocks, ticket);
    case ZOACT_DT_BF16:
      return loss_multi_dispatch(ctx, static_cast<const __nv_bfloat16*>(Y),
                                 static_cast<const __nv_bfloat16*>(target), count, nb, mu, out, partials, max_blocks,
                                 ticket);
    case ZOACT_DT_FP16:
      return loss_multi_dispatch(ctx, static_cast<const __half*>(Y), static_cast<const __half*>(target), count, nb,
                                 mu, out, partials, max_blocks, ticket);
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
}

int launch_loss_pair(Ctx* ctx, const void* Y, int ydtype, const void* target, int64_t T, int64_t n, float eps,
                     double* out, double* partials, int max_blocks) {
  const int64_t count = T * n;
  unsigned int* ticket = ctx->d_tickets;
  switch (ydtype) {
    case ZOACT_DT_FP32:
      return loss_dispatch(ctx, static_cast<const float*>(Y), static_cast<const float*>(target), count, eps, out,
                           partials, max_blocks, ticket);
    case ZOACT_DT_BF16:
      return loss_dispatch(ctx, static_cast<const __nv_bfloat16*>(Y), static_cast<const __nv_bfloat16*>(target),
                           count, eps, out, partials, max_blocks, ticket);
    case ZOACT_DT_FP16:
      return loss_dispatch(ctx, static_cast<const __half*>(Y), static_cast<const __half*>(target), count, eps, out,
                           partials, max_blocks, ticket);
    default:
      return ZOACT_ERR_INVALID_ARG;
  }
}

}  // namespace zoact
