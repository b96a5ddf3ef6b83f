// One-shot activation basis (Algorithm 1: top-r right singular vectors of the
// calibration activations X, i.e. the top-r eigenvectors of G = X^T X).
//
// Device pipeline (no host round trip, every step a kernel):
//   1. G = X^T X in fp32: for 16-bit X, X is transposed into a zero-padded
//      [d, n_pad] copy and multiplied with itself on the tcgen05 GEMM;
//      for fp32 X a CUDA-core kernel forms X^T X directly.
//   2. Omega [d, k] from the Z generator (seed, layer 0, query 0), k = r + oversample.
//   3. Q = orth(Omega); n_iter times Q = orth(G Q).  orth() is CholeskyQR2:
//      S = Y^T Y accumulated in fp64, Cholesky S = R^T R and R^-1 in one block
//      (fp64), Q = Y R^-1; done twice for orthogonality.
//   4. Rayleigh-Ritz: S = Q^T G Q (fp64), cyclic Jacobi in one block (fp64),
//      eigenpairs sorted by value, U = Q V[:, :r], each column flipped so its
//      largest-magnitude entry is positive (first index on ties).
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

constexpr int KMAX = 64;

// ---- X [n, d] (16-bit) -> Xt [d, n_pad], zero in columns n .. n_pad-1 ----
template <typename T>
__global__ void transpose_pad_kernel(const T* __restrict__ X, T* __restrict__ Xt, int64_t n, int d, int64_t n_pad) {
  __shared__ T tile[32][33];
  const int64_t t0 = (int64_t)blockIdx.x * 32;
  const int i0 = blockIdx.y * 32;
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int64_t t = t0 + y;
    const int i = i0 + threadIdx.x;
    tile[y][threadIdx.x] = (t < n && i < d) ? X[t * d + i] : from_f32<T>(0.f);
  }
  __syncthreads();
  for (int y = threadIdx.y; y < 32; y += 8) {
    const int i = i0 + y;
    const int64_t t = t0 + threadIdx.x;
    if (i < d && t < n_pad) Xt[(int64_t)i * n_pad + t] = tile[threadIdx.x][y];
  }
}

// ---- G = X^T X for fp32 X [n, d] (CUDA cores, 64x64 tiles) ----
__global__ void __launch_bounds__(256) gram_f32_kernel(const float* __restrict__ X, float* __restrict__ G, int64_t n,
                                                       int d) {
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64 + 4];
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int i0 = blockIdx.y * 64, j0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int64_t t0 = 0; t0 < n; t0 += 16) {
    __syncthreads();
    for (int v = threadIdx.x; v < 16 * 64; v += 256) {
      const int kk = v / 64, c = v % 64;
      const int64_t t = t0 + kk;
      As[kk][c] = (t < n && i0 + c < d) ? X[t * d + i0 + c] : 0.f;
      Bs[kk][c] = (t < n && j0 + c < d) ? X[t * d + j0 + c] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int q = 0; q < 4; ++q) { a[q] = As[kk][ty * 4 + q]; b[q] = Bs[kk][tx * 4 + q]; }
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[p][q] = fmaf(a[p], b[q], acc[p][q]);
    }
  }
  for (int p = 0; p < 4; ++p)
    for (int q = 0; q < 4; ++q) {
      const int i = i0 + ty * 4 + p, j = j0 + tx * 4 + q;
      if (i < d && j < d) G[(int64_t)i * d + j] = acc[p][q];
    }
}

// ---- Omega [d, k]: element i*k + j of the (seed, 0, 0) stream ----
__global__ void omega_kernel(float* __restrict__ Om, int64_t n, uint64_t seed) {
  for (int64_t g = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; 4 * g < n; g += (int64_t)gridDim.x * blockDim.x) {
    const float4 z = z_normals4(seed, 0u, 0ull, (uint64_t)g);
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (4 * g + i < n) Om[4 * g + i] = z_select(z, i);
  }
}

// ---- Y [d, k] = G [d, d] * Q [d, k] (fp32, 64-row blocks, K staged in chunks of 32) ----
__global__ void __launch_bounds__(256) gemm_gq_kernel(const float* __restrict__ G, const float* __restrict__ Q,
                                                      float* __restrict__ Y, int d, int k) {
  __shared__ float Gs[64][33];
  __shared__ __align__(16) float Qs[32][KMAX];
  const int cg = threadIdx.x % 16, rg = threadIdx.x / 16;  // 16 col groups x 16 row groups (4x4 each)
  const int64_t i0 = (int64_t)blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < d; k0 += 32) {
    __syncthreads();
    for (int v = threadIdx.x; v < 64 * 32; v += 256) {
      const int rr = v / 32, kk = v % 32;
      Gs[rr][kk] = (i0 + rr < d && k0 + kk < d) ? G[(i0 + rr) * d + k0 + kk] : 0.f;
    }
    for (int v = threadIdx.x; v < 32 * KMAX; v += 256) {
      const int kk = v / KMAX, c = v % KMAX;
      Qs[kk][c] = (k0 + kk < d && c < k) ? Q[(int64_t)(k0 + kk) * k + c] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < 32; ++kk) {
      const float4 q = *reinterpret_cast<const float4*>(&Qs[kk][cg * 4]);
#pragma unroll
      for (int p = 0; p < 4; ++p) {
        const float g = Gs[rg * 4 + p][kk];
        acc[p][0] = fmaf(g, q.x, acc[p][0]);
        acc[p][1] = fmaf(g, q.y, acc[p][1]);
        acc[p][2] = fmaf(g, q.z, acc[p][2]);
        acc[p][3] = fmaf(g, q.w, acc[p][3]);
      }
    }
  }
  for (int p = 0; p < 4; ++p) {
    const int64_t i = i0 + rg * 4 + p;
    if (i >= d) continue;
    for (int c = 0; c < 4; ++c) {
      const int j = cg * 4 + c;
      if (j < k) Y[i * k + j] = acc[p][c];
    }
  }
}

// ---- partial S = A^T B over a chunk of ATB_ROWS rows, fp64, A, B [d, k] ----
constexpr int ATB_ROWS = 64;
__global__ void __launch_bounds__(256) atb_partial_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                          double* __restrict__ part, int d, int k) {
  __shared__ float As[ATB_ROWS][KMAX + 1];
  __shared__ float Bs[ATB_ROWS][KMAX + 1];
  const int64_t r0 = (int64_t)blockIdx.x * ATB_ROWS;
  const int nrow = (int)((int64_t)d - r0 < ATB_ROWS ? (int64_t)d - r0 : ATB_ROWS);
  for (int v = threadIdx.x; v < ATB_ROWS * k; v += 256) {
    const int rr = v / k, c = v % k;
    As[rr][c] = rr < nrow ? A[(r0 + rr) * k + c] : 0.f;
    Bs[rr][c] = rr < nrow ? B[(r0 + rr) * k + c] : 0.f;
  }
  __syncthreads();
  double* out = part + (int64_t)blockIdx.x * k * k;
  for (int pq = threadIdx.x; pq < k * k; pq += 256) {
    const int p = pq / k, q = pq % k;
    double s = 0.0;
    for (int rr = 0; rr < nrow; ++rr) s += (double)As[rr][p] * (double)Bs[rr][q];
    out[pq] = s;
  }
}

__global__ void sum_partials_kernel(const double* __restrict__ part, double* __restrict__ S, int nblk, int kk) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < kk; i += gridDim.x * blockDim.x) {
    double s = 0.0;
    for (int b = 0; b < nblk; ++b) s += part[(int64_t)b * kk + i];
    S[i] = s;
  }
}

// ---- Cholesky S = R^T R (R upper) and Rinv, one block; shift on breakdown ----
constexpr int CHOL_SMEM = 2 * KMAX * KMAX * 8;
__global__ void chol_inv_kernel(const double* __restrict__ S, double* __restrict__ Rinv, int k, int* status) {
  extern __shared__ double chol_sm[];
  double (*R)[KMAX] = reinterpret_cast<double (*)[KMAX]>(chol_sm);
  double (*Ri)[KMAX] = reinterpret_cast<double (*)[KMAX]>(chol_sm + KMAX * KMAX);
  __shared__ int bad;
  __shared__ double shift;
  const int t = threadIdx.x;
  if (t == 0) {
    double tr = 0.0;
    for (int i = 0; i < k; ++i) tr += S[i * k + i];
    shift = 0.0;
    bad = 0;
    (void)tr;
  }
  __syncthreads();
  for (int attempt = 0; attempt < 4; ++attempt) {
    for (int v = t; v < k * k; v += blockDim.x) {
      const int i = v / k, j = v % k;
      R[i][j] = (j >= i) ? S[i * k + j] + (i == j ? shift : 0.0) : 0.0;
    }
    __syncthreads();
    if (t == 0) {
      bad = 0;
      for (int j = 0; j < k && !bad; ++j) {
        double djj = R[j][j];
        for (int p = 0; p < j; ++p) djj -= R[p][j] * R[p][j];
        if (!(djj > 0.0)) { bad = 1; break; }
        const double rjj = sqrt(djj);
        R[j][j] = rjj;
        for (int q = j + 1; q < k; ++q) {
          double s = R[j][q];
          for (int p = 0; p < j; ++p) s -= R[p][j] * R[p][q];
          R[j][q] = s / rjj;
        }
      }
      if (bad) {
        double tr = 0.0;
        for (int i = 0; i < k; ++i) tr += S[i * k + i];
        shift = (shift == 0.0) ? 1e-12 * tr : shift * 1e3;
      }
    }
    __syncthreads();
    if (!bad) break;
  }
  if (bad) {
    if (t == 0) record_error(status, ZOACT_ERR_NONFINITE);
    return;
  }
  // Rinv: solve R * Ri = I column by column (column c per thread)
  for (int c = t; c < k; c += blockDim.x) {
    for (int i = k - 1; i >= 0; --i) {
      double s = (i == c) ? 1.0 : 0.0;
      for (int p = i + 1; p < k; ++p) s -= R[i][p] * Ri[p][c];
      Ri[i][c] = s / R[i][i];
    }
  }
  __syncthreads();
  for (int v = t; v < k * k; v += blockDim.x) Rinv[v] = Ri[v / k][v % k];
}

// ---- Q [d, k] = Y [d, k] * Rinv [k, k] (fp64 accumulate, fp32 out); Q may alias Y ----
// One warp per row: every lane reads the row before any lane writes it.
__global__ void apply_rinv_kernel(const float* Y, const double* __restrict__ Rinv, float* Q, int d, int k) {
  __shared__ double Rs[KMAX * KMAX];
  for (int v = threadIdx.y * blockDim.x + threadIdx.x; v < k * k; v += blockDim.x * blockDim.y) Rs[v] = Rinv[v];
  __syncthreads();
  for (int64_t i = blockIdx.x * (int64_t)blockDim.y + threadIdx.y; i < d; i += (int64_t)gridDim.x * blockDim.y) {
    float out[KMAX / 32];
#pragma unroll
    for (int h = 0; h < KMAX / 32; ++h) {
      const int c = threadIdx.x + 32 * h;
      double s = 0.0;
      if (c < k)
        for (int p = 0; p <= c; ++p) s += (double)Y[i * k + p] * Rs[p * k + c];
      out[h] = (float)s;
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < KMAX / 32; ++h) {
      const int c = threadIdx.x + 32 * h;
      if (c < k) Q[i * k + c] = out[h];
    }
    __syncwarp();
  }
}

// ---- cyclic Jacobi on S (k x k, fp64), eigenvalues descending; V columns ----
constexpr int JACOBI_SMEM = 2 * KMAX * (KMAX + 1) * 8;
__global__ void jacobi_kernel(const double* __restrict__ S, double* __restrict__ Vout, double* __restrict__ evals,
                              int k) {
  extern __shared__ double jac_sm[];
  double (*A)[KMAX + 1] = reinterpret_cast<double (*)[KMAX + 1]>(jac_sm);
  double (*V)[KMAX + 1] = reinterpret_cast<double (*)[KMAX + 1]>(jac_sm + KMAX * (KMAX + 1));
  __shared__ double cs[2];
  __shared__ int done;
  __shared__ int order[KMAX];
  const int t = threadIdx.x;  // blockDim.x >= k
  for (int v = t; v < k * k; v += blockDim.x) {
    const int i = v / k, j = v % k;
    A[i][j] = 0.5 * (S[i * k + j] + S[j * k + i]);
    V[i][j] = (i == j) ? 1.0 : 0.0;
  }
  __syncthreads();
  for (int sweep = 0; sweep < 60; ++sweep) {
    if (t == 0) {
      double off = 0.0, tot = 0.0;
      for (int i = 0; i < k; ++i)
        for (int j = 0; j < k; ++j) {
          tot += A[i][j] * A[i][j];
          if (i != j) off += A[i][j] * A[i][j];
        }
      done = (off <= 1e-30 * tot) ? 1 : 0;
    }
    __syncthreads();
    if (done) break;
    for (int p = 0; p < k - 1; ++p) {
      for (int q = p + 1; q < k; ++q) {
        if (t == 0) {
          const double apq = A[p][q];
          double c = 1.0, s = 0.0;
          if (fabs(apq) > 1e-300) {
            const double theta = (A[q][q] - A[p][p]) / (2.0 * apq);
            double tt;
            if (fabs(theta) > 1e150) tt = 0.5 / theta;
            else tt = (theta >= 0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
            c = 1.0 / sqrt(1.0 + tt * tt);
            s = tt * c;
          }
          cs[0] = c; cs[1] = s;
        }
        __syncthreads();
        const double c = cs[0], s = cs[1];
        if (s != 0.0) {
          if (t < k) {  // columns p, q
            const double ap = A[t][p], aq = A[t][q];
            A[t][p] = c * ap - s * aq;
            A[t][q] = s * ap + c * aq;
            const double vp = V[t][p], vq = V[t][q];
            V[t][p] = c * vp - s * vq;
            V[t][q] = s * vp + c * vq;
          }
          __syncthreads();
          if (t < k) {  // rows p, q
            const double ap = A[p][t], aq = A[q][t];
            A[p][t] = c * ap - s * aq;
            A[q][t] = s * ap + c * aq;
          }
        }
        __syncthreads();
      }
    }
  }
  if (t == 0) {
    for (int i = 0; i < k; ++i) order[i] = i;
    for (int i = 0; i < k; ++i) {  // selection sort, descending
      int best = i;
      for (int j = i + 1; j < k; ++j)
        if (A[order[j]][order[j]] > A[order[best]][order[best]]) best = j;
      const int tmp = order[i]; order[i] = order[best]; order[best] = tmp;
    }
  }
  __syncthreads();
  for (int v = t; v < k * k; v += blockDim.x) {
    const int i = v / k, j = v % k;
    Vout[i * k + j] = V[i][order[j]];
  }
  for (int j = t; j < k; j += blockDim.x) evals[j] = A[order[j]][order[j]];
}

// ---- U [d, r] = Q [d, k] * V[:, :r] ----
__global__ void ritz_kernel(const float* __restrict__ Q, const double* __restrict__ V, float* __restrict__ U, int d,
                            int k, int r) {
  for (int64_t v = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; v < (int64_t)d * r;
       v += (int64_t)gridDim.x * blockDim.x) {
    const int64_t i = v / r;
    const int j = (int)(v % r);
    double s = 0.0;
    for (int p = 0; p < k; ++p) s += (double)Q[i * k + p] * V[p * k + j];
    U[v] = (float)s;
  }
}

// ---- flip column j so its largest-|.| entry (first index on ties) is positive ----
__global__ void sign_fix_kernel(float* __restrict__ U, int d, int r) {
  const int j = blockIdx.x;
  __shared__ float bv[256];
  __shared__ int bi[256];
  float best = -1.f;
  int idx = 0x7fffffff;
  for (int i = threadIdx.x; i < d; i += blockDim.x) {
    const float a = fabsf(U[(int64_t)i * r + j]);
    if (a > best || (a == best && i < idx)) { best = a; idx = i; }
  }
  bv[threadIdx.x] = best;
  bi[threadIdx.x] = idx;
  __syncthreads();
  for (int s = blockDim.x / 2; s > 0; s >>= 1) {
    if (threadIdx.x < s) {
      const float a = bv[threadIdx.x + s];
      const int ia = bi[threadIdx.x + s];
      if (a > bv[threadIdx.x] || (a == bv[threadIdx.x] && ia < bi[threadIdx.x])) {
        bv[threadIdx.x] = a;
        bi[threadIdx.x] = ia;
      }
    }
    __syncthreads();
  }
  const bool flip = U[(int64_t)bi[0] * r + j] < 0.f;
  __syncthreads();
  if (flip)
    for (int i = threadIdx.x; i < d; i += blockDim.x) U[(int64_t)i * r + j] = -U[(int64_t)i * r + j];
}

__global__ void f64_to_f32_kernel(const double* __restrict__ a, float* __restrict__ b, int n) {
  for (int i = threadIdx.x; i < n; i += blockDim.x) b[i] = (float)a[i];
}

struct Work {
  float* G;
  float* Q;
  float* Y;
  double* part;
  double* S;
  double* Rinv;
  double* V;
  double* ev;
};

int orth(Ctx* ctx, Work& w, float* Y, float* Q, int d, int k) {
  // CholeskyQR2: Q = Y R^-1 twice
  const int nblk = (d + ATB_ROWS - 1) / ATB_ROWS;
  const float* src = Y;
  for (int pass = 0; pass < 2; ++pass) {
    atb_partial_kernel<<<nblk, 256, 0, ctx->stream>>>(src, src, w.part, d, k); ++ctx->n_launch;
    sum_partials_kernel<<<(k * k + 255) / 256, 256, 0, ctx->stream>>>(w.part, w.S, nblk, k * k); ++ctx->n_launch;
    chol_inv_kernel<<<1, 64, CHOL_SMEM, ctx->stream>>>(w.S, w.Rinv, k, ctx->d_status); ++ctx->n_launch;
    apply_rinv_kernel<<<(d + 7) / 8 < 4096 ? (d + 7) / 8 : 4096, dim3(32, 8), 0, ctx->stream>>>(src, w.Rinv, Q, d, k); ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
    src = Q;
  }
  return ZOACT_OK;
}

}  // namespace

int run_basis_init(Ctx* ctx, const void* X, int xdtype, int64_t n_tok, int d, int r, int oversample, int n_iter,
                   uint64_t seed, float* U_out, float* evals_out) {
  int k = r + oversample;
  if (k > d) k = d;
  if (k > KMAX || r > k) return ZOACT_ERR_UNSUPPORTED;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(chol_inv_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, CHOL_SMEM));
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(jacobi_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, JACOBI_SMEM));
  const int nblk = (d + ATB_ROWS - 1) / ATB_ROWS;
  // workspace: G d*d f32 | Q, Y d*k f32 | part nblk*k*k f64 | S, Rinv, V k*k f64 | ev k f64
  const size_t bytes = (size_t)d * d * 4 + 2 * (size_t)d * k * 4 + (size_t)nblk * k * k * 8 + 3 * (size_t)k * k * 8 +
                       (size_t)k * 8 + 1024;
  uint8_t* base = static_cast<uint8_t*>(scratch(ctx, SLOT_BASIS, bytes));
  if (!base) return ZOACT_ERR_NOMEM;
  Work w;
  size_t off = 0;
  auto take = [&](size_t b) { uint8_t* p = base + off; off += (b + 255) / 256 * 256; return p; };
  w.G = reinterpret_cast<float*>(take((size_t)d * d * 4));
  w.Q = reinterpret_cast<float*>(take((size_t)d * k * 4));
  w.Y = reinterpret_cast<float*>(take((size_t)d * k * 4));
  w.part = reinterpret_cast<double*>(take((size_t)nblk * k * k * 8));
  w.S = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.Rinv = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.V = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.ev = reinterpret_cast<double*>(take((size_t)k * 8));
  (void)off;

  // 1. Gram
  if (xdtype == ZOACT_DT_FP32) {
    dim3 grid((d + 63) / 64, (d + 63) / 64);
    gram_f32_kernel<<<grid, 256, 0, ctx->stream>>>(static_cast<const float*>(X), w.G, n_tok, d); ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
  } else {
    const int64_t n_pad = (n_tok + 7) / 8 * 8;
    void* Xt = scratch(ctx, SLOT_BASIS_X, (size_t)d * n_pad * 2);
    if (!Xt) return ZOACT_ERR_NOMEM;
    dim3 grid((unsigned)((n_pad + 31) / 32), (unsigned)((d + 31) / 32));
    if (xdtype == ZOACT_DT_BF16) {
      transpose_pad_kernel<__nv_bfloat16><<<grid, dim3(32, 8), 0, ctx->stream>>>(
          static_cast<const __nv_bfloat16*>(X), static_cast<__nv_bfloat16*>(Xt), n_tok, d, n_pad);
    } else {
      transpose_pad_kernel<__half><<<grid, dim3(32, 8), 0, ctx->stream>>>(static_cast<const __half*>(X),
                                                                          static_cast<__half*>(Xt), n_tok, d, n_pad);
    }
    ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
    const int st = launch_gemm_tc_f32out(ctx, Xt, Xt, xdtype, d, d, (int)n_pad, w.G);
    if (st) return st;
  }
  // 2-3. sketch and subspace iteration
  const int64_t nq = (int64_t)d * k;
  omega_kernel<<<(unsigned)((nq / 4 + 255) / 256 + 1), 256, 0, ctx->stream>>>(w.Y, nq, seed); ++ctx->n_launch;
  ZOACT_CHECK_LAUNCH();
  int st = orth(ctx, w, w.Y, w.Q, d, k);
  if (st) return st;
  const unsigned gq_blocks = (unsigned)((d + 63) / 64);
  for (int it = 0; it < n_iter; ++it) {
    gemm_gq_kernel<<<gq_blocks, 256, 0, ctx->stream>>>(w.G, w.Q, w.Y, d, k); ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
    st = orth(ctx, w, w.Y, w.Q, d, k);
    if (st) return st;
  }
  // 4. Rayleigh-Ritz
  gemm_gq_kernel<<<gq_blocks, 256, 0, ctx->stream>>>(w.G, w.Q, w.Y, d, k); ++ctx->n_launch;
  atb_partial_kernel<<<nblk, 256, 0, ctx->stream>>>(w.Q, w.Y, w.part, d, k); ++ctx->n_launch;
  sum_partials_kernel<<<(k * k + 255) / 256, 256, 0, ctx->stream>>>(w.part, w.S, nblk, k * k); ++ctx->n_launch;
  jacobi_kernel<<<1, KMAX, JACOBI_SMEM, ctx->stream>>>(w.S, w.V, w.ev, k); ++ctx->n_launch;
  ritz_kernel<<<(unsigned)(((int64_t)d * r + 255) / 256), 256, 0, ctx->stream>>>(w.Q, w.V, U_out, d, k, r); ++ctx->n_launch;
  sign_fix_kernel<<<r, 256, 0, ctx->stream>>>(U_out, d, r); ++ctx->n_launch;
  if (evals_out) {
    f64_to_f32_kernel<<<1, 64, 0, ctx->stream>>>(w.ev, evals_out, k);
    ++ctx->n_launch;
  }
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
