// One-shot activation basis (Algorithm 1: top-r right singular vectors of the
// calibration activations X, i.e. the top-r eigenvectors of G = X^T X).
//
// Device pipeline (no host round trip, every step a kernel):
//   1. G = X^T X in fp32: for 16-bit X, X is transposed into a zero-padded
//      [d, n_pad] copy and multiplied with itself on the tcgen05 GEMM;
//      for fp32 X a CUDA-core kernel forms X^T X directly.
//   2. Omega [d, k] from the Z generator (seed, layer 0, query 0), k = r + oversample.
//   3. Q = orth(Omega); n_iter times Q = orth(G Q).  orth() is CholeskyQR2:
//      S = Y^T Y (64 x 64 output tiles; fp32 over 32-row slabs, fp64 across
//      slabs and row chunks), Cholesky S = R^T R and R^-1 in one block (fp64,
//      in global memory), Q = Y R^-1; done twice for orthogonality.
//   4. Rayleigh-Ritz: S = Q^T G Q (fp64), Jacobi in one block (fp64): cyclic in
//      shared memory for k <= 64, parallel round-robin pairs in global memory
//      above; eigenpairs sorted by value, U = Q V[:, :r], each column flipped so
//      its largest-magnitude entry is positive (first index on ties).
//   k = r + oversample <= 512.
#include "internal.h"
#include "philox.cuh"

namespace zoact {
namespace {

constexpr int KMAX = 64;        // k handled by the shared-memory Jacobi and R^-1 application
constexpr int KLIM = 512;       // largest k

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

// ---- Y [d, k] = G [d, d] * Q [d, k] (fp32, 64-row x 64-column blocks, K staged in chunks of 32) ----
__global__ void __launch_bounds__(256) gemm_gq_kernel(const float* __restrict__ G, const float* __restrict__ Q,
                                                      float* __restrict__ Y, int d, int k) {
  const int c0 = blockIdx.y * KMAX;
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
      Qs[kk][c] = (k0 + kk < d && c0 + c < k) ? Q[(int64_t)(k0 + kk) * k + c0 + c] : 0.f;
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
      const int j = c0 + cg * 4 + c;
      if (j < k) Y[i * k + j] = acc[p][c];
    }
  }
}

// ---- partial S = A^T B over a chunk of rows, A, B [d, k]: 64 x 64 output tiles per block (grid x, y),
// row chunks on grid z; fp32 products over 32-row slabs, added into fp64 per slab ----
constexpr int ATB_CHUNK = 2048;
__global__ void __launch_bounds__(256) atb_partial_kernel(const float* __restrict__ A, const float* __restrict__ B,
                                                          double* __restrict__ part, int d, int k) {
  __shared__ float As[32][KMAX + 4];
  __shared__ float Bs[32][KMAX + 4];
  const int p0 = blockIdx.y * KMAX, q0 = blockIdx.x * KMAX;
  const int tx = threadIdx.x % 16, ty = threadIdx.x / 16;
  const int64_t r_begin = (int64_t)blockIdx.z * ATB_CHUNK;
  const int64_t r_end = r_begin + ATB_CHUNK < d ? r_begin + ATB_CHUNK : d;
  double acc[4][4] = {};
  for (int64_t s0 = r_begin; s0 < r_end; s0 += 32) {
    __syncthreads();
    for (int v = threadIdx.x; v < 32 * KMAX; v += 256) {
      const int rr = v / KMAX, c = v % KMAX;
      const int64_t row = s0 + rr;
      As[rr][c] = (row < r_end && p0 + c < k) ? A[row * k + p0 + c] : 0.f;
      Bs[rr][c] = (row < r_end && q0 + c < k) ? B[row * k + q0 + c] : 0.f;
    }
    __syncthreads();
    float a32[4][4] = {};
#pragma unroll 8
    for (int rr = 0; rr < 32; ++rr) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) { a[i] = As[rr][ty * 4 + i]; b[i] = Bs[rr][tx * 4 + i]; }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) a32[i][j] = fmaf(a[i], b[j], a32[i][j]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] += (double)a32[i][j];
  }
  double* out = part + (int64_t)blockIdx.z * k * k;
  for (int i = 0; i < 4; ++i)
    for (int j = 0; j < 4; ++j) {
      const int p = p0 + ty * 4 + i, q = q0 + tx * 4 + j;
      if (p < k && q < k) out[(int64_t)p * k + q] = acc[i][j];
    }
}

__global__ void sum_partials_kernel(const double* __restrict__ part, double* __restrict__ S, int nblk, int kk) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < kk; i += gridDim.x * blockDim.x) {
    double s = 0.0;
    for (int b = 0; b < nblk; ++b) s += part[(int64_t)b * kk + i];
    S[i] = s;
  }
}

// ---- Cholesky S = R^T R (R upper) and Rinv, one block, R in global memory (k x k fp64); shift on breakdown ----
__global__ void __launch_bounds__(256) chol_inv_kernel(const double* __restrict__ S, double* __restrict__ R,
                                                       double* __restrict__ Rinv, int k, int* status) {
  __shared__ int bad;
  __shared__ double shift, rjj_s;
  __shared__ double red[256];
  const int t = threadIdx.x;
  if (t == 0) { shift = 0.0; bad = 0; }
  __syncthreads();
  for (int attempt = 0; attempt < 4; ++attempt) {
    for (int v = t; v < k * k; v += blockDim.x) {
      const int i = v / k, j = v % k;
      R[v] = (j >= i) ? S[v] + (i == j ? shift : 0.0) : 0.0;
    }
    if (t == 0) bad = 0;
    __syncthreads();
    for (int j = 0; j < k; ++j) {
      // r_jj = sqrt(R[j][j] - sum_{p<j} R[p][j]^2)
      double part = 0.0;
      for (int p = t; p < j; p += blockDim.x) part += R[(int64_t)p * k + j] * R[(int64_t)p * k + j];
      red[t] = part;
      __syncthreads();
      for (int h = blockDim.x / 2; h > 0; h >>= 1) {
        if (t < h) red[t] += red[t + h];
        __syncthreads();
      }
      if (t == 0) {
        const double djj = R[(int64_t)j * k + j] - red[0];
        if (!(djj > 0.0)) {
          bad = 1;
        } else {
          rjj_s = sqrt(djj);
          R[(int64_t)j * k + j] = rjj_s;
        }
      }
      __syncthreads();
      if (bad) break;
      // R[j][q] = (R[j][q] - sum_{p<j} R[p][j] R[p][q]) / r_jj for q > j
      for (int q = j + 1 + t; q < k; q += blockDim.x) {
        double s2 = R[(int64_t)j * k + q];
        for (int p = 0; p < j; ++p) s2 -= R[(int64_t)p * k + j] * R[(int64_t)p * k + q];
        R[(int64_t)j * k + q] = s2 / rjj_s;
      }
      __syncthreads();
    }
    if (!bad) break;
    if (t == 0) {
      double tr = 0.0;
      for (int i = 0; i < k; ++i) tr += S[(int64_t)i * k + i];
      shift = (shift == 0.0) ? 1e-12 * tr : shift * 1e3;
    }
    __syncthreads();
  }
  if (bad) {
    if (t == 0) record_error(status, ZOACT_ERR_NONFINITE);
    return;
  }
  // Rinv: solve R * Ri = I column by column (column c per thread)
  for (int c = t; c < k; c += blockDim.x) {
    for (int i = k - 1; i >= 0; --i) {
      double s2 = (i == c) ? 1.0 : 0.0;
      for (int p = i + 1; p <= c; ++p) s2 -= R[(int64_t)i * k + p] * Rinv[(int64_t)p * k + c];
      Rinv[(int64_t)i * k + c] = i > c ? 0.0 : s2 / R[(int64_t)i * k + i];
    }
  }
}

// ---- Q [d, k] = Y [d, k] * Rinv [k, k] (fp64 accumulate, fp32 out); Q may alias Y ----
// One warp per row: every lane reads the row before any lane writes it.
// R^-1 is read from shared memory for k <= KMAX, else from global memory (L2).
__global__ void apply_rinv_kernel(const float* Y, const double* __restrict__ Rinv, float* Q, int d, int k) {
  __shared__ double Rs[KMAX * KMAX];
  const bool in_smem = k <= KMAX;
  if (in_smem)
    for (int v = threadIdx.y * blockDim.x + threadIdx.x; v < k * k; v += blockDim.x * blockDim.y) Rs[v] = Rinv[v];
  __syncthreads();
  const double* Rm = in_smem ? Rs : Rinv;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.y + threadIdx.y; i < d; i += (int64_t)gridDim.x * blockDim.y) {
    float out[KLIM / 32];
#pragma unroll
    for (int h = 0; h < KLIM / 32; ++h) {
      const int c = threadIdx.x + 32 * h;
      double s = 0.0;
      if (c < k)
        for (int p = 0; p <= c; ++p) s += (double)Y[i * k + p] * Rm[(int64_t)p * k + c];
      out[h] = (float)s;
    }
    __syncwarp();
#pragma unroll
    for (int h = 0; h < KLIM / 32; ++h) {
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

// ---- Jacobi for k > KMAX: A, V in global memory (k x k fp64 each), one block; every sweep runs the
// round-robin schedule of k' - 1 rounds (k' = k rounded up to even; index k' - 1 is a dummy when k is odd)
// of k'/2 disjoint rotations: angles from the current A, then A <- A J (columns), A <- J^T A (rows),
// V <- V J.  Eigenvalues descending in evals, eigenvectors as the columns of Vout. ----
__device__ __forceinline__ int rr_member(int slot, int round, int n) {
  // slot 0 stays; slots 1 .. n-1 rotate by `round`
  return slot == 0 ? 0 : 1 + (slot - 1 + round) % (n - 1);
}
__global__ void __launch_bounds__(1024) jacobi_big_kernel(const double* __restrict__ S, double* __restrict__ A,
                                                          double* __restrict__ V, double* __restrict__ Vout,
                                                          double* __restrict__ evals, int k) {
  __shared__ double cs_c[KLIM / 2], cs_s[KLIM / 2];
  __shared__ int pp[KLIM / 2], qq[KLIM / 2];
  __shared__ int done;
  __shared__ double red[1024];
  __shared__ int order[KLIM];
  const int t = threadIdx.x, nt = blockDim.x;
  const int n = (k + 1) / 2 * 2;
  const int npair = n / 2;
  for (int64_t v = t; v < (int64_t)k * k; v += nt) {
    const int i = (int)(v / k), j = (int)(v % k);
    A[v] = 0.5 * (S[(int64_t)i * k + j] + S[(int64_t)j * k + i]);
    V[v] = (i == j) ? 1.0 : 0.0;
  }
  __syncthreads();
  for (int sweep = 0; sweep < 60; ++sweep) {
    double off = 0.0, tot = 0.0;
    for (int64_t v = t; v < (int64_t)k * k; v += nt) {
      const double a = A[v];
      tot += a * a;
      if (v / k != v % k) off += a * a;
    }
    red[t] = off;
    __syncthreads();
    for (int h = nt / 2; h > 0; h >>= 1) {
      if (t < h) red[t] += red[t + h];
      __syncthreads();
    }
    const double off_all = red[0];
    __syncthreads();
    red[t] = tot;
    __syncthreads();
    for (int h = nt / 2; h > 0; h >>= 1) {
      if (t < h) red[t] += red[t + h];
      __syncthreads();
    }
    if (t == 0) done = (off_all <= 1e-30 * red[0]) ? 1 : 0;
    __syncthreads();
    if (done) break;
    for (int round = 0; round < n - 1; ++round) {
      for (int i = t; i < npair; i += nt) {
        int p = rr_member(i, round, n), q = rr_member(n - 1 - i, round, n);
        if (p > q) { const int tmp = p; p = q; q = tmp; }
        double c = 1.0, s2 = 0.0;
        if (q < k) {
          const double apq = A[(int64_t)p * k + q];
          if (fabs(apq) > 1e-300) {
            const double theta = (A[(int64_t)q * k + q] - A[(int64_t)p * k + p]) / (2.0 * apq);
            double tt;
            if (fabs(theta) > 1e150) tt = 0.5 / theta;
            else tt = (theta >= 0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
            c = 1.0 / sqrt(1.0 + tt * tt);
            s2 = tt * c;
          }
        }
        pp[i] = p; qq[i] = q; cs_c[i] = c; cs_s[i] = s2;
      }
      __syncthreads();
      // columns of A and V: for every row and pair
      for (int64_t v = t; v < (int64_t)k * npair; v += nt) {
        const int row = (int)(v / npair), i = (int)(v % npair);
        const int p = pp[i], q = qq[i];
        const double c = cs_c[i], s2 = cs_s[i];
        if (q >= k || s2 == 0.0) continue;
        const double ap = A[(int64_t)row * k + p], aq = A[(int64_t)row * k + q];
        A[(int64_t)row * k + p] = c * ap - s2 * aq;
        A[(int64_t)row * k + q] = s2 * ap + c * aq;
        const double vp = V[(int64_t)row * k + p], vq = V[(int64_t)row * k + q];
        V[(int64_t)row * k + p] = c * vp - s2 * vq;
        V[(int64_t)row * k + q] = s2 * vp + c * vq;
      }
      __syncthreads();
      // rows of A
      for (int64_t v = t; v < (int64_t)k * npair; v += nt) {
        const int col = (int)(v / npair), i = (int)(v % npair);
        const int p = pp[i], q = qq[i];
        const double c = cs_c[i], s2 = cs_s[i];
        if (q >= k || s2 == 0.0) continue;
        const double ap = A[(int64_t)p * k + col], aq = A[(int64_t)q * k + col];
        A[(int64_t)p * k + col] = c * ap - s2 * aq;
        A[(int64_t)q * k + col] = s2 * ap + c * aq;
      }
      __syncthreads();
    }
  }
  if (t == 0) {
    for (int i = 0; i < k; ++i) order[i] = i;
    for (int i = 0; i < k; ++i) {  // selection sort, descending
      int best = i;
      for (int j = i + 1; j < k; ++j)
        if (A[(int64_t)order[j] * k + order[j]] > A[(int64_t)order[best] * k + order[best]]) best = j;
      const int tmp = order[i]; order[i] = order[best]; order[best] = tmp;
    }
  }
  __syncthreads();
  for (int64_t v = t; v < (int64_t)k * k; v += nt) {
    const int i = (int)(v / k), j = (int)(v % k);
    Vout[v] = V[(int64_t)i * k + order[j]];
  }
  for (int j = t; j < k; j += nt) evals[j] = A[(int64_t)order[j] * k + order[j]];
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
// A column without a finite entry (non-finite calibration data) is left as it is and
// the status word records ZOACT_ERR_NONFINITE.
__global__ void sign_fix_kernel(float* __restrict__ U, int d, int r, int* __restrict__ status) {
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
  const int top = bi[0];
  if (top < 0 || top >= d) {                 // no finite |U| in this column
    if (threadIdx.x == 0) record_error(status, ZOACT_ERR_NONFINITE);
    return;
  }
  const bool flip = U[(int64_t)top * r + j] < 0.f;
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
  double* R;      // Cholesky factor / Jacobi matrix (k x k)
  double* Vw;     // Jacobi rotations (k x k)
  int nchunk;     // row chunks of the A^T B partials
};

void launch_atb(Ctx* ctx, const Work& w, const float* A, const float* B, int d, int k) {
  const unsigned tiles = (unsigned)((k + KMAX - 1) / KMAX);
  atb_partial_kernel<<<dim3(tiles, tiles, (unsigned)w.nchunk), 256, 0, ctx->stream>>>(A, B, w.part, d, k);
  ++ctx->n_launch;
  sum_partials_kernel<<<(k * k + 255) / 256, 256, 0, ctx->stream>>>(w.part, w.S, w.nchunk, k * k);
  ++ctx->n_launch;
}

int orth(Ctx* ctx, Work& w, float* Y, float* Q, int d, int k) {
  // CholeskyQR2: Q = Y R^-1 twice
  const float* src = Y;
  for (int pass = 0; pass < 2; ++pass) {
    launch_atb(ctx, w, src, src, d, k);
    chol_inv_kernel<<<1, 256, 0, ctx->stream>>>(w.S, w.R, w.Rinv, k, ctx->d_status); ++ctx->n_launch;
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
  if (k > KLIM || r > k) return ZOACT_ERR_UNSUPPORTED;
  ZOACT_CUDA_TRY(cudaFuncSetAttribute(jacobi_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, JACOBI_SMEM));
  const int nchunk = (d + ATB_CHUNK - 1) / ATB_CHUNK;
  // workspace: G d*d f32 | Q, Y d*k f32 | part nchunk*k*k f64 | S, Rinv, V, R, Vw k*k f64 | ev k f64
  const size_t bytes = (size_t)d * d * 4 + 2 * (size_t)d * k * 4 + (size_t)nchunk * k * k * 8 +
                       5 * (size_t)k * k * 8 + (size_t)k * 8 + 4096;
  uint8_t* base = static_cast<uint8_t*>(scratch(ctx, SLOT_BASIS, bytes));
  if (!base) return ZOACT_ERR_NOMEM;
  Work w;
  size_t off = 0;
  auto take = [&](size_t b) { uint8_t* p = base + off; off += (b + 255) / 256 * 256; return p; };
  w.G = reinterpret_cast<float*>(take((size_t)d * d * 4));
  w.Q = reinterpret_cast<float*>(take((size_t)d * k * 4));
  w.Y = reinterpret_cast<float*>(take((size_t)d * k * 4));
  w.part = reinterpret_cast<double*>(take((size_t)nchunk * k * k * 8));
  w.S = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.Rinv = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.V = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.ev = reinterpret_cast<double*>(take((size_t)k * 8));
  w.R = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.Vw = reinterpret_cast<double*>(take((size_t)k * k * 8));
  w.nchunk = nchunk;
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
  const dim3 gq_blocks((unsigned)((d + 63) / 64), (unsigned)((k + KMAX - 1) / KMAX));
  for (int it = 0; it < n_iter; ++it) {
    gemm_gq_kernel<<<gq_blocks, 256, 0, ctx->stream>>>(w.G, w.Q, w.Y, d, k); ++ctx->n_launch;
    ZOACT_CHECK_LAUNCH();
    st = orth(ctx, w, w.Y, w.Q, d, k);
    if (st) return st;
  }
  // 4. Rayleigh-Ritz
  gemm_gq_kernel<<<gq_blocks, 256, 0, ctx->stream>>>(w.G, w.Q, w.Y, d, k); ++ctx->n_launch;
  launch_atb(ctx, w, w.Q, w.Y, d, k);
  if (k <= KMAX) {
    jacobi_kernel<<<1, KMAX, JACOBI_SMEM, ctx->stream>>>(w.S, w.V, w.ev, k);
  } else {
    jacobi_big_kernel<<<1, 1024, 0, ctx->stream>>>(w.S, w.R, w.Vw, w.V, w.ev, k);
  }
  ++ctx->n_launch;
  ritz_kernel<<<(unsigned)(((int64_t)d * r + 255) / 256), 256, 0, ctx->stream>>>(w.Q, w.V, U_out, d, k, r); ++ctx->n_launch;
  sign_fix_kernel<<<r, 256, 0, ctx->stream>>>(U_out, d, r, ctx->d_status); ++ctx->n_launch;
  if (evals_out) {
    f64_to_f32_kernel<<<1, 256, 0, ctx->stream>>>(w.ev, evals_out, k);
    ++ctx->n_launch;
  }
  ZOACT_CHECK_LAUNCH();
  return ZOACT_OK;
}

}  // namespace zoact
