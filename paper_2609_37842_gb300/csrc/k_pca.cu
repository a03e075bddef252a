// PCA fit of the second stage (App. B.2 "PCA fitting"; Alg. 1 "fit P_u by
// uncentered PCA of {z_iu}"): the top-k eigenvectors of Z^T Z / n, obtained
// from the n x n Gram matrix Z Z^T / n when n < m (the route the paper
// describes). Everything runs on the device. Two solvers, by size
// (nn = min(n, m)):
//
// Dense (nn <= 1024, or k close to nn): every eigenpair of the nn x nn matrix.
//  1. A = Z^T Z / n (or Z Z^T): CUDA-core GEMM on the fp32 Z with fp64
//     accumulation.
//  2. Cyclic two-sided Jacobi (Golub & Van Loan, Sec. 8.5) in round-robin
//     ("circle") order: each step rotates nn'/2 disjoint (p, q) pairs. One
//     kernel forms the rotations (in double) from the current A; a second
//     applies J^T A J to rows p, q of A (row rotation, then the column
//     rotations of every pair inside the two rows held in shared memory) and
//     J^T to rows p, q of V^T. Sweeps repeat until the off-diagonal mass stops
//     shrinking or falls below 1e-11 of ||A||_F; A and V^T are kept in fp64.
//  3. Rank the eigenvalues (descending, ties to the lower index), keep the top
//     k, map Gram-route vectors through Z^T u / ||Z^T u||, normalise, and fix
//     each vector's sign so its largest-magnitude entry is positive.
//
// Subspace iteration (larger problems): only the top k eigenpairs.
//  1. A = Z^T Z / n (or Z Z^T / n) on the tensor cores: Z as a bf16 hi/lo pair
//     (about 16 significant bits), three MMAs per step (hi hi, hi lo, lo hi),
//     fp32 accumulation; A is symmetrised and kept as a hi/lo pair.
//  2. Block power iteration on p = k + max(64, k / 4) (rounded up to 32)
//     vectors, kept as rows of X^T: Y = A X on the tensor cores, then X =
//     orthonormal basis of Y by three Cholesky-QR passes (rows normalised,
//     Gram Y^T Y on the tensor cores, Cholesky of the Gram plus a shift of
//     1e-2 / 1e-4 / 0 of its mean diagonal in fp32, X = Y L^-T): the shifts keep
//     the factorisation defined when the columns of A X are nearly dependent.
//  3. Every 5 iterations a Rayleigh-Ritz step: H = X^T A X (p x p), its
//     eigenpairs by the Jacobi solver above in fp64, X and A X rotated onto the
//     Ritz vectors (ordered by Ritz value, descending). The iteration stops
//     when every one of the top k Ritz pairs has ||A x - theta x|| <= 1e-3 theta.
//  4. The top k Ritz vectors (mapped through Z^T u on the Gram route) are
//     normalised and signed as in the dense solver; eig = the Ritz values.
#include <algorithm>
#include <cmath>
#include <cstring>
#include <vector>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

namespace {

__device__ __forceinline__ void jac_pair(int s, int kidx, int np, int& p, int& q) {
  const int L = np - 1;
  if (kidx == 0) {
    p = s;
    q = L;
  } else {
    p = (s + kidx) % L;
    q = (s - kidx + L) % L;
  }
  if (p > q) {
    const int t = p;
    p = q;
    q = t;
  }
}

// C[i][j] = alpha * sum_k A(i,k) B(j,k) with A(i,k) = A[i*sai + k*sak] (fp32 in,
// fp64 accumulate and out). 32 x 32 tile per block, 2 x 2 per thread.
template <typename TA>
__global__ void __launch_bounds__(256) k_gemm_f64acc(int M, int N, int K, double alpha, int accumulate,
                                                     const TA* __restrict__ A, long long sai,
                                                     long long sak, const float* __restrict__ B,
                                                     long long sbj, long long sbk,
                                                     double* __restrict__ C, long long ldc) {
  __shared__ double As[16][33];
  __shared__ double Bs[16][33];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int i0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
  double acc[2][2] = {{0.0, 0.0}, {0.0, 0.0}};
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int r = 0; r < 2; ++r) {
      const int e = tid + 256 * r;
      int ii, kk;
      if (sak == 1) { ii = e >> 4; kk = e & 15; } else { kk = e >> 5; ii = e & 31; }
      double v = 0.0;
      if (i0 + ii < M && k0 + kk < K) v = static_cast<double>(A[(i0 + ii) * sai + (k0 + kk) * sak]);
      As[kk][ii] = v;
      int jj, kb;
      if (sbk == 1) { jj = e >> 4; kb = e & 15; } else { kb = e >> 5; jj = e & 31; }
      double w = 0.0;
      if (j0 + jj < N && k0 + kb < K) w = static_cast<double>(B[(j0 + jj) * sbj + (k0 + kb) * sbk]);
      Bs[kb][jj] = w;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      const double a0 = As[kk][ty], a1 = As[kk][ty + 16];
      const double b0 = Bs[kk][tx], b1 = Bs[kk][tx + 16];
      acc[0][0] = fma(a0, b0, acc[0][0]);
      acc[0][1] = fma(a0, b1, acc[0][1]);
      acc[1][0] = fma(a1, b0, acc[1][0]);
      acc[1][1] = fma(a1, b1, acc[1][1]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int x = 0; x < 2; ++x) {
    const int i = i0 + ty + 16 * x;
    if (i >= M) continue;
#pragma unroll
    for (int y = 0; y < 2; ++y) {
      const int j = j0 + tx + 16 * y;
      if (j < N) C[i * ldc + j] = accumulate ? C[i * ldc + j] + alpha * acc[x][y] : alpha * acc[x][y];
    }
  }
}

template <typename TA>
cudaError_t gemm_f64acc(int M, int N, int K, double alpha, const TA* A, long long sai, long long sak,
                        const float* B, long long sbj, long long sbk, double* C, long long ldc,
                        cudaStream_t st, int accumulate = 0) {
  dim3 grid((N + 31) / 32, (M + 31) / 32);
  k_gemm_f64acc<TA><<<grid, 256, 0, st>>>(M, N, K, alpha, accumulate, A, sai, sak, B, sbj, sbk, C, ldc);
  return cudaGetLastError();
}

// A[i][j] = scale * C[i][j] (dense n x n copy of a strided fp64 matrix)
__global__ void k_scale_copy(const double* __restrict__ C, int ldc, int n, double scale, double* __restrict__ A) {
  const long long tot = static_cast<long long>(n) * n;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x)
    A[e] = scale * C[(e / n) * ldc + e % n];
}

__global__ void k_eye(double* V, int n) {
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (idx >= static_cast<long long>(n) * n) return;
  V[idx] = (idx / n == idx % n) ? 1.0 : 0.0;
}

__global__ void k_jacobi_params(const double* __restrict__ A, int n, int np, int s,
                                double* __restrict__ cs) {
  const int kidx = blockIdx.x * blockDim.x + threadIdx.x;
  if (kidx >= np / 2) return;
  int p, q;
  jac_pair(s, kidx, np, p, q);
  double c = 1.0, sn = 0.0;
  if (q < n) {
    const double app = A[static_cast<size_t>(p) * n + p];
    const double aqq = A[static_cast<size_t>(q) * n + q];
    const double apq = A[static_cast<size_t>(p) * n + q];
    if (apq != 0.0) {
      const double tau = (aqq - app) / (2.0 * apq);
      double t;
      if (fabs(tau) > 1e150) {
        t = 0.5 / tau;
      } else {
        t = (tau >= 0.0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
      }
      c = 1.0 / sqrt(1.0 + t * t);
      sn = t * c;
    }
  }
  cs[2 * kidx] = c;
  cs[2 * kidx + 1] = sn;
}

__global__ void __launch_bounds__(256) k_jacobi_apply(double* __restrict__ A, double* __restrict__ Vt,
                                                      int n, int np, int s,
                                                      const double* __restrict__ cs) {
  extern __shared__ double rows[];
  double* rp = rows;
  double* rq = rows + n;
  const int kidx = blockIdx.x;
  int p, q;
  jac_pair(s, kidx, np, p, q);
  if (q >= n) return;
  const double c = cs[2 * kidx];
  const double sn = cs[2 * kidx + 1];
  double* Ap = A + static_cast<size_t>(p) * n;
  double* Aq = A + static_cast<size_t>(q) * n;
  for (int x = threadIdx.x; x < n; x += blockDim.x) {
    const double ap = Ap[x], aq = Aq[x];
    rp[x] = c * ap - sn * aq;
    rq[x] = sn * ap + c * aq;
  }
  __syncthreads();
  for (int j = threadIdx.x; j < np / 2; j += blockDim.x) {
    int pj, qj;
    jac_pair(s, j, np, pj, qj);
    if (qj >= n) continue;
    const double cj = cs[2 * j];
    const double sj = cs[2 * j + 1];
    double xp = rp[pj], xq = rp[qj];
    rp[pj] = cj * xp - sj * xq;
    rp[qj] = sj * xp + cj * xq;
    xp = rq[pj];
    xq = rq[qj];
    rq[pj] = cj * xp - sj * xq;
    rq[qj] = sj * xp + cj * xq;
  }
  __syncthreads();
  if (threadIdx.x == 0 && sn != 0.0) {
    rp[q] = 0.0;  // the annihilated pair
    rq[p] = 0.0;
  }
  __syncthreads();
  for (int x = threadIdx.x; x < n; x += blockDim.x) {
    Ap[x] = rp[x];
    Aq[x] = rq[x];
  }
  double* Vp = Vt + static_cast<size_t>(p) * n;
  double* Vq = Vt + static_cast<size_t>(q) * n;
  for (int x = threadIdx.x; x < n; x += blockDim.x) {
    const double vp = Vp[x], vq = Vq[x];
    Vp[x] = c * vp - sn * vq;
    Vq[x] = sn * vp + c * vq;
  }
}

__global__ void __launch_bounds__(256) k_offnorm(const double* __restrict__ A, int n,
                                                 double* __restrict__ red) {
  __shared__ double so[256], st[256];
  double off = 0.0, tot = 0.0;
  const long long N2 = static_cast<long long>(n) * n;
  for (long long idx = blockIdx.x * 256LL + threadIdx.x; idx < N2; idx += 256LL * gridDim.x) {
    const double v = A[idx];
    tot += v * v;
    if (idx / n != idx % n) off += v * v;
  }
  so[threadIdx.x] = off;
  st[threadIdx.x] = tot;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      so[threadIdx.x] += so[threadIdx.x + w];
      st[threadIdx.x] += st[threadIdx.x + w];
    }
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    atomicAdd(&red[0], so[0]);
    atomicAdd(&red[1], st[0]);
  }
}

// mu[i] = A[i][i]; sel[rank(i)] = i for the k largest (descending, ties to lower index).
__global__ void k_rank(const double* __restrict__ A, int n, int k, double* __restrict__ mu,
                       int* __restrict__ sel) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const double vi = A[static_cast<size_t>(i) * n + i];
  mu[i] = vi;
  int rank = 0;
  for (int j = 0; j < n; ++j) {
    const double vj = A[static_cast<size_t>(j) * n + j];
    rank += (vj > vi) || (vj == vi && j < i);
  }
  if (rank < k) sel[rank] = i;
}

// Pt row r = sign * src row (sel ? sel[r] : r) / ||row||, sign making the
// largest-magnitude entry (lowest index on ties) positive; eig[r] = mu[sel[r]] * eig_scale.
template <typename TS>
__global__ void __launch_bounds__(256) k_emit(const TS* __restrict__ src, int ld_src,
                                              const int* __restrict__ sel, int m,
                                              void* __restrict__ Pt, int ld_pt, int bf16_out,
                                              const double* __restrict__ mu, double eig_scale,
                                              float* __restrict__ eig) {
  __shared__ double s_ss[256];
  __shared__ double s_mx[256];
  __shared__ int s_ix[256];
  const int r = blockIdx.x;
  const TS* v = src + static_cast<size_t>(sel ? sel[r] : r) * ld_src;
  double ss = 0.0, mx = -1.0;
  int ix = 0x7fffffff;
  for (int c = threadIdx.x; c < m; c += blockDim.x) {
    const double x = static_cast<double>(v[c]);
    ss = fma(x, x, ss);
    const double a = fabs(x);
    if (a > mx) {
      mx = a;
      ix = c;
    }
  }
  s_ss[threadIdx.x] = ss;
  s_mx[threadIdx.x] = mx;
  s_ix[threadIdx.x] = ix;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) {
      s_ss[threadIdx.x] += s_ss[threadIdx.x + w];
      const double om = s_mx[threadIdx.x + w];
      const int oi = s_ix[threadIdx.x + w];
      if (om > s_mx[threadIdx.x] || (om == s_mx[threadIdx.x] && oi < s_ix[threadIdx.x])) {
        s_mx[threadIdx.x] = om;
        s_ix[threadIdx.x] = oi;
      }
    }
    __syncthreads();
  }
  const double nrm = sqrt(s_ss[0]);
  const double sgn = static_cast<double>(v[s_ix[0]]) < 0.0 ? -1.0 : 1.0;
  const double f = nrm > 0.0 ? sgn / nrm : 0.0;
  for (int c = threadIdx.x; c < m; c += blockDim.x) {
    const float o = static_cast<float>(static_cast<double>(v[c]) * f);
    if (bf16_out)
      static_cast<__nv_bfloat16*>(Pt)[static_cast<size_t>(r) * ld_pt + c] = __float2bfloat16_rn(o);
    else
      static_cast<float*>(Pt)[static_cast<size_t>(r) * ld_pt + c] = o;
  }
  if (threadIdx.x == 0 && eig) eig[r] = static_cast<float>(mu[sel ? sel[r] : r] * eig_scale);
}

__global__ void k_gather_f64_rows(const double* __restrict__ src, int ld, const int* __restrict__ sel,
                                  int len, double* __restrict__ dst) {
  const int r = blockIdx.x;
  for (int c = threadIdx.x; c < len; c += blockDim.x)
    dst[static_cast<size_t>(r) * len + c] = src[static_cast<size_t>(sel[r]) * ld + c];
}

__global__ void k_eig_out(const double* __restrict__ mu, const int* __restrict__ sel, int k,
                          double scale, float* __restrict__ eig) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r < k) eig[r] = static_cast<float>(mu[sel[r]] * scale);
}

size_t al256(size_t x) { return (x + 255) & ~size_t(255); }
inline int rup(int x, int a) { return (x + a - 1) / a * a; }

// ------------------------------------------------ subspace-iteration kernels
using bf16 = __nv_bfloat16;

__device__ __forceinline__ void split2(float v, bf16& h, bf16& l) {
  h = __float2bfloat16_rn(v);
  l = __float2bfloat16_rn(v - __bfloat162float(h));
}

// hi/lo [rows][ldd] of rscale[r] * src[r][c] for c < cols, zero in the padding.
__global__ void k_split_rows(const float* __restrict__ src, long long lds, int rows, int cols,
                             const float* __restrict__ rscale, bf16* __restrict__ hi,
                             bf16* __restrict__ lo, int ldd) {
  const long long tot = static_cast<long long>(rows) * ldd;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(e / ldd), c = static_cast<int>(e % ldd);
    float v = 0.f;
    if (c < cols) {
      v = src[static_cast<long long>(r) * lds + c];
      if (rscale) v *= rscale[r];
    }
    bf16 h, l;
    split2(v, h, l);
    hi[e] = h;
    lo[e] = l;
  }
}

// Transposed hi/lo [cols][ldd]: dst[c][r] = rscale[r] * src[r][c] for r < rows,
// zero for rows <= r < ldd. Grid (ceil(cols / 32), ceil(ldd / 32)), block 32 x 8.
__global__ void k_split_T(const float* __restrict__ src, long long lds, int rows, int cols,
                          const float* __restrict__ rscale, bf16* __restrict__ hi,
                          bf16* __restrict__ lo, int ldd) {
  __shared__ float t[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int j = ty; j < 32; j += 8) {
    const int r = r0 + j, c = c0 + tx;
    float v = 0.f;
    if (r < rows && c < cols) {
      v = src[static_cast<long long>(r) * lds + c];
      if (rscale) v *= rscale[r];
    }
    t[j][tx] = v;
  }
  __syncthreads();
  for (int j = ty; j < 32; j += 8) {
    const int c = c0 + j, r = r0 + tx;
    if (c < cols && r < ldd) {
      bf16 h, l;
      split2(t[tx][j], h, l);
      hi[static_cast<long long>(c) * ldd + r] = h;
      lo[static_cast<long long>(c) * ldd + r] = l;
    }
  }
}

// hi/lo [n][ldd] of (A + A^T) / 2 for a square fp32 A, zero in the padding.
// Grid (ceil(ldd / 32), ceil(n / 32)), block 32 x 8.
__global__ void k_split_sym(const float* __restrict__ A, long long lda, int n, bf16* __restrict__ hi,
                            bf16* __restrict__ lo, int ldd) {
  __shared__ float t[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x, ty = threadIdx.y;
  for (int j = ty; j < 32; j += 8) {
    const int rr = c0 + j, cc = r0 + tx;  // t[j][tx] = A[c0 + j][r0 + tx]
    t[j][tx] = (rr < n && cc < n) ? A[static_cast<long long>(rr) * lda + cc] : 0.f;
  }
  __syncthreads();
  for (int j = ty; j < 32; j += 8) {
    const int r = r0 + j, c = c0 + tx;
    if (r < n && c < ldd) {
      float v = 0.f;
      if (c < n) v = 0.5f * (A[static_cast<long long>(r) * lda + c] + t[tx][j]);
      bf16 h, l;
      split2(v, h, l);
      hi[static_cast<long long>(r) * ldd + c] = h;
      lo[static_cast<long long>(r) * ldd + c] = l;
    }
  }
}

// A32[i][j] = scale * C[i][j] (fp64 second moment -> fp32)
__global__ void k_f64_to_f32(const double* __restrict__ C, long long ldc, int n, double scale,
                             float* __restrict__ A, long long lda) {
  const long long tot = static_cast<long long>(n) * n;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x)
    A[(e / n) * lda + e % n] = static_cast<float>(scale * C[(e / n) * ldc + e % n]);
}

// rs[r] = 1 / ||src[r][0..cols)|| (0 for a zero row); one block per row.
__global__ void __launch_bounds__(256) k_row_invnorm(const float* __restrict__ src, long long lds, int cols,
                                                     float* __restrict__ rs) {
  __shared__ double red[256];
  const float* v = src + static_cast<long long>(blockIdx.x) * lds;
  double ss = 0.0;
  for (int c = threadIdx.x; c < cols; c += 256) {
    const double x = v[c];
    ss = fma(x, x, ss);
  }
  red[threadIdx.x] = ss;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) rs[blockIdx.x] = red[0] > 0.0 ? static_cast<float>(1.0 / sqrt(red[0])) : 0.f;
}

// Start vectors: standard normal entries from a counter-based generator
// (SplitMix64 of seed + element index, then the Box-Muller transform).
__device__ __forceinline__ unsigned long long splitmix64(unsigned long long x) {
  x += 0x9E3779B97F4A7C15ull;
  x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
  x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
  return x ^ (x >> 31);
}

__global__ void k_gauss(float* __restrict__ X, long long ld, int rows, int cols, unsigned long long seed) {
  const long long tot = static_cast<long long>(rows) * cols;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const unsigned long long h = splitmix64(seed * 0x100000001B3ull + static_cast<unsigned long long>(e));
    const float u1 = (static_cast<float>(h >> 40) + 0.5f) * (1.0f / 16777216.0f);
    const float u2 = static_cast<float>((h >> 16) & 0xFFFFFFull) * (1.0f / 16777216.0f);
    X[(e / cols) * ld + e % cols] = sqrtf(-2.0f * logf(u1)) * cospif(2.0f * u2);
  }
}

__global__ void k_add_diag(float* __restrict__ A, int lda, int n, const float* __restrict__ shift) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) A[static_cast<long long>(i) * lda + i] += *shift;
}

// shift[0] = rel * (mean diagonal of A) (the Cholesky-QR shift).
__global__ void __launch_bounds__(256) k_diag_shift(const float* __restrict__ A, int lda, int n, float rel,
                                                    float* __restrict__ shift) {
  __shared__ double red[256];
  double s = 0.0;
  for (int i = threadIdx.x; i < n; i += 256) s += A[static_cast<long long>(i) * lda + i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) shift[0] = static_cast<float>(rel * red[0] / n);
}

// ---- blocked Cholesky (lower, in place, fp32), panels of 32 columns
// Diagonal block at j0: 32 x 32 threads, one entry each.
__global__ void __launch_bounds__(1024) k_chol_diag(float* __restrict__ A, int lda, int n, int j0,
                                                    unsigned* status) {
  __shared__ float a[32][33];
  const int i = threadIdx.y, j = threadIdx.x;
  const int nb = min(32, n - j0);
  a[i][j] = (i < nb && j < nb) ? A[static_cast<long long>(j0 + i) * lda + j0 + j] : 0.f;
  __syncthreads();
  for (int c = 0; c < nb; ++c) {
    if (i == c && j == c) {
      float d = a[c][c];
      if (!(d > 0.f) || !isfinite(d)) {  // not positive definite: flag it, keep going
        eogp::flag_status(status, EOGP_ST_DEVICE);
        d = 1e-30f;
      }
      a[c][c] = sqrtf(d);
    }
    __syncthreads();
    if (j == c && i > c && i < nb) a[i][c] /= a[c][c];
    __syncthreads();
    if (i > c && j > c && j <= i && i < nb) a[i][j] -= a[i][c] * a[j][c];
    __syncthreads();
  }
  if (i < nb && j < nb) A[static_cast<long long>(j0 + i) * lda + j0 + j] = (j <= i) ? a[i][j] : 0.f;
}

// Rows i >= j0 + 32: A[i][j0..j0+32) <- A[i][j0..j0+32) L_d^-T (forward
// substitution, one thread per row).
__global__ void __launch_bounds__(128) k_chol_panel(float* __restrict__ A, int lda, int n, int j0) {
  __shared__ float L[32][33];
  for (int e = threadIdx.x; e < 1024; e += 128) {
    const int r = e >> 5, c = e & 31;
    L[r][c] = A[static_cast<long long>(j0 + r) * lda + j0 + c];
  }
  __syncthreads();
  const int i = j0 + 32 + blockIdx.x * 128 + threadIdx.x;
  if (i >= n) return;
  float* row = A + static_cast<long long>(i) * lda + j0;
  float x[32];
#pragma unroll
  for (int c = 0; c < 32; ++c) {
    float v = row[c];
#pragma unroll
    for (int t = 0; t < c; ++t) v -= x[t] * L[c][t];
    x[c] = v / L[c][c];
  }
#pragma unroll
  for (int c = 0; c < 32; ++c) row[c] = x[c];
}

// Trailing update of the lower triangle: A[i][j] -= sum_t A[i][j0 + t] A[j][j0 + t]
// for j0 + 32 <= j <= i < n; one block per 64 x 64 tile on or below the diagonal.
__global__ void __launch_bounds__(256) k_chol_update(float* __restrict__ A, int lda, int n, int j0) {
  __shared__ float Pi[64][33];
  __shared__ float Pj[64][33];
  const int j1 = j0 + 32;
  const int b = blockIdx.x;
  int ti = static_cast<int>((sqrt(8.0 * b + 1.0) - 1.0) * 0.5);
  while ((ti + 1) * (ti + 2) / 2 <= b) ++ti;
  while (ti * (ti + 1) / 2 > b) --ti;
  const int tj = b - ti * (ti + 1) / 2;
  const int r0 = j1 + ti * 64, c0 = j1 + tj * 64;
  for (int e = threadIdx.x; e < 64 * 32; e += 256) {
    const int r = e >> 5, t = e & 31;
    Pi[r][t] = (r0 + r < n) ? A[static_cast<long long>(r0 + r) * lda + j0 + t] : 0.f;
    Pj[r][t] = (c0 + r < n) ? A[static_cast<long long>(c0 + r) * lda + j0 + t] : 0.f;
  }
  __syncthreads();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};
#pragma unroll 8
  for (int t = 0; t < 32; ++t) {
    float a[4], bb[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      a[u] = Pi[ty + 16 * u][t];
      bb[u] = Pj[tx + 16 * u][t];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
      for (int v = 0; v < 4; ++v) acc[u][v] = fmaf(a[u], bb[v], acc[u][v]);
  }
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int i = r0 + ty + 16 * u;
    if (i >= n) continue;
#pragma unroll
    for (int v = 0; v < 4; ++v) {
      const int j = c0 + tx + 16 * v;
      if (j <= i) A[static_cast<long long>(i) * lda + j] -= acc[u][v];
    }
  }
}

// ---- inverse of a lower-triangular matrix (fp32), 32 x 32 blocks; Li zeroed first
// Diagonal blocks: one 32-thread block per block, one column each.
__global__ void k_trinv_diag(const float* __restrict__ L, int lda, float* __restrict__ Li, int ldi, int n) {
  __shared__ float Ls[32][33];
  const int j0 = blockIdx.x * 32, nb = min(32, n - j0), c = threadIdx.x;
  for (int r = 0; r < 32; ++r)
    Ls[r][c] = (r < nb && c < nb) ? L[static_cast<long long>(j0 + r) * lda + j0 + c] : 0.f;
  __syncthreads();
  if (c >= nb) return;
  float x[32];
#pragma unroll
  for (int i = 0; i < 32; ++i) {
    float v = 0.f;
    if (i >= c && i < nb) {
      v = (i == c) ? 1.f : 0.f;
      for (int t = c; t < i; ++t) v -= Ls[i][t] * x[t];
      v /= Ls[i][i];
    }
    x[i] = v;
  }
  for (int i = c; i < nb; ++i) Li[static_cast<long long>(j0 + i) * ldi + j0 + c] = x[i];
}

// Blocks at distance d below the diagonal: Li[I][J] = -Li[I][I] sum_{K=J}^{I-1} L[I][K] Li[K][J],
// I = J + d (grid = number of such blocks); 256 threads, 4 entries each.
__global__ void __launch_bounds__(256) k_trinv_off(const float* __restrict__ L, int lda, float* __restrict__ Li,
                                                   int ldi, int n, int d) {
  __shared__ float As[32][33];
  __shared__ float Bs[32][33];
  const int J = blockIdx.x, I = J + d;
  const int i0 = I * 32, j0 = J * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // ty 0..7: rows ty + 8u
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  for (int K = J; K < I; ++K) {
    const int k0 = K * 32;
    for (int e = threadIdx.x; e < 1024; e += 256) {
      const int r = e >> 5, c = e & 31;
      As[r][c] = (i0 + r < n) ? L[static_cast<long long>(i0 + r) * lda + k0 + c] : 0.f;
      Bs[r][c] = Li[static_cast<long long>(k0 + r) * ldi + j0 + c];
    }
    __syncthreads();
#pragma unroll 8
    for (int t = 0; t < 32; ++t) {
      const float bv = Bs[t][tx];
#pragma unroll
      for (int u = 0; u < 4; ++u) acc[u] = fmaf(As[ty + 8 * u][t], bv, acc[u]);
    }
    __syncthreads();
  }
  // T = acc (rows ty + 8u, column tx) -> Bs; Li[I][I] -> As
#pragma unroll
  for (int u = 0; u < 4; ++u) Bs[ty + 8 * u][tx] = acc[u];
  for (int e = threadIdx.x; e < 1024; e += 256) {
    const int r = e >> 5, c = e & 31;
    As[r][c] = (i0 + r < n && i0 + c < n) ? Li[static_cast<long long>(i0 + r) * ldi + i0 + c] : 0.f;
  }
  __syncthreads();
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    const int r = ty + 8 * u;
    float v = 0.f;
#pragma unroll 8
    for (int t = 0; t < 32; ++t) v = fmaf(As[r][t], Bs[t][tx], v);
    if (i0 + r < n) Li[static_cast<long long>(i0 + r) * ldi + j0 + tx] = -v;
  }
}

// H64[i][j] = (H[i][j] + H[j][i]) / 2
__global__ void k_sym_f64(const float* __restrict__ H, int ldh, int n, double* __restrict__ out) {
  const long long tot = static_cast<long long>(n) * n;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int i = static_cast<int>(e / n), j = static_cast<int>(e % n);
    out[e] = 0.5 * (static_cast<double>(H[static_cast<long long>(i) * ldh + j]) +
                    static_cast<double>(H[static_cast<long long>(j) * ldh + i]));
  }
}

// St[j][c] = Vt[sel[j]][c] (rows of the Ritz rotation, eigenvalue descending); theta[j] = mu[sel[j]]
__global__ void k_ritz_rows(const double* __restrict__ Vt, int n, const int* __restrict__ sel,
                            const double* __restrict__ mu, float* __restrict__ St, int lds,
                            float* __restrict__ theta) {
  const int j = blockIdx.x;
  const double* v = Vt + static_cast<long long>(sel[j]) * n;
  for (int c = threadIdx.x; c < n; c += blockDim.x) St[static_cast<long long>(j) * lds + c] = static_cast<float>(v[c]);
  if (threadIdx.x == 0) theta[j] = static_cast<float>(mu[sel[j]]);
}

// out[0] = max over j < k of ||CX[j] - theta_j X[j]|| / |theta_j| (float bits, atomicMax; out zeroed first)
__global__ void __launch_bounds__(256) k_ritz_resid(const float* __restrict__ X, const float* __restrict__ CX,
                                                    long long ld, int nn, const float* __restrict__ theta,
                                                    unsigned* __restrict__ out) {
  __shared__ double red[256];
  const int j = blockIdx.x;
  const float th = theta[j];
  double ss = 0.0;
  for (int c = threadIdx.x; c < nn; c += 256) {
    const double r = static_cast<double>(CX[j * ld + c]) - static_cast<double>(th) * X[j * ld + c];
    ss = fma(r, r, ss);
  }
  red[threadIdx.x] = ss;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) {
    float v = th != 0.f ? static_cast<float>(sqrt(red[0]) / fabs(static_cast<double>(th))) : 0.f;
    if (!(v == v)) v = 3.0e38f;  // NaN: never converged
    atomicMax(out, __float_as_uint(v));
  }
}

__global__ void k_copy_eig(const float* __restrict__ theta, int k, float* __restrict__ eig) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r < k) eig[r] = theta[r];
}

// ---------------------------------------------------------------- layouts
int pca_block(int k) { return rup(k + std::max(64, k / 4), 32); }

bool use_subspace(int nn, int k) { return nn > 1024 && pca_block(k) < nn; }

struct DenseLayout {
  size_t A, Vt, cs, mu, sel, red, Pr, total;
};

DenseLayout dense_layout(int n, int m, int k) {
  const size_t nn = static_cast<size_t>(std::min(n, m));
  DenseLayout L{};
  size_t o = 0;
  auto take = [&](size_t b) { const size_t at = o; o += al256(b); return at; };
  L.A = take(nn * nn * 8);
  L.Vt = take(nn * nn * 8);
  L.cs = take((nn / 2 + 1) * 2 * 8);
  L.mu = take(nn * 8);
  L.sel = take(nn * 4);
  L.red = take(4 * 8);
  L.Pr = n < m ? take(static_cast<size_t>(k) * m * 8) : 0;
  L.total = o;
  return L;
}

struct SubLayout {
  int nn, p, nn4, nn8, p4, p8, n8, m8;
  size_t Zh, Zl, ZTh, ZTl;       // Z [n][m8] (Gram route); Z^T [m][n8] (both routes with Z)
  size_t A32, Ah, Al;            // A [nn][nn8] fp32 / bf16 hi, lo
  size_t X32, CX32;              // X^T, (A X)^T [p][nn4] fp32
  size_t Yh, Yl;                 // row-normalised splits [p][nn8]
  size_t YTh, YTl, CTh, CTl;     // transposed splits [nn][p8]
  size_t G32, Li32, Sh, Sl;      // [p][p4] fp32, splits [p][p8]
  size_t rs, shift, theta, resid;
  size_t H64, V64, cs, mu, sel, red;
  size_t Pr;                     // Gram route: raw directions [k][m4] fp32
  size_t total;
};

SubLayout sub_layout(int n, int m, int k, bool with_z) {
  SubLayout L{};
  L.nn = std::min(n, m);
  L.p = pca_block(k);
  L.nn4 = rup(L.nn, 4);
  L.nn8 = rup(L.nn, 8);
  L.p4 = rup(L.p, 4);
  L.p8 = rup(L.p, 8);
  L.n8 = rup(n, 8);
  L.m8 = rup(m, 8);
  const size_t nn = L.nn, p = L.p;
  size_t o = 0;
  auto take = [&](size_t b) { const size_t at = o; o += al256(b); return at; };
  const bool gram = n < m;
  if (with_z) {
    if (gram) {
      L.Zh = take(static_cast<size_t>(n) * L.m8 * 2);
      L.Zl = take(static_cast<size_t>(n) * L.m8 * 2);
    }
    L.ZTh = take(static_cast<size_t>(m) * L.n8 * 2);
    L.ZTl = take(static_cast<size_t>(m) * L.n8 * 2);
  }
  L.A32 = take(nn * L.nn8 * 4);
  L.Ah = take(nn * L.nn8 * 2);
  L.Al = take(nn * L.nn8 * 2);
  L.X32 = take(p * L.nn4 * 4);
  L.CX32 = take(p * L.nn4 * 4);
  L.Yh = take(p * L.nn8 * 2);
  L.Yl = take(p * L.nn8 * 2);
  // transposed splits [nn][p8]; also used for row splits [p][nn8]
  const size_t ybig = std::max(nn * L.p8, p * L.nn8);
  L.YTh = take(ybig * 2);
  L.YTl = take(ybig * 2);
  L.CTh = take(nn * L.p8 * 2);
  L.CTl = take(nn * L.p8 * 2);
  L.G32 = take(p * L.p4 * 4);
  L.Li32 = take(p * L.p4 * 4);
  L.Sh = take(p * L.p8 * 2);
  L.Sl = take(p * L.p8 * 2);
  L.rs = take(p * 4);
  L.shift = take(16);
  L.theta = take(p * 4);
  L.resid = take(16);
  L.H64 = take(p * p * 8);
  L.V64 = take(p * p * 8);
  L.cs = take((p / 2 + 1) * 2 * 8);
  L.mu = take(p * 8);
  L.sel = take(p * 4);
  L.red = take(4 * 8);
  L.Pr = gram ? take(static_cast<size_t>(k) * rup(m, 4) * 4) : 0;
  L.total = o;
  return L;
}

}  // namespace

bool fit_pca_supported(int n, int m, int k) {
  const int nn = std::min(n, m);
  if (use_subspace(nn, k)) return pca_block(k) <= 12288 && nn <= 32768;
  return nn <= 12288;
}

size_t fit_pca_ws_bytes(int n, int m, int k) {
  const int nn = std::min(n, m);
  if (use_subspace(nn, k)) return sub_layout(n, m, k, true).total;
  return dense_layout(n, m, k).total;
}

#define PCA_TRY(x)                                                                         \
  do {                                                                                     \
    cudaError_t e_ = (x);                                                                  \
    if (e_ != cudaSuccess)                                                                 \
      return eogp::set_error(EOGP_ECUDA, "fit_pca: %s: %s", #x, cudaGetErrorString(e_));   \
  } while (0)

namespace {

unsigned grid_for(long long tot) {
  return static_cast<unsigned>(std::max<long long>(1, std::min<long long>((tot + 255) / 256, 152LL * 16)));
}

// Cyclic Jacobi on A (fp64, n x n, overwritten by its diagonal form); Vt = eigenvectors as rows.
int jacobi_eigen(double* A, double* Vt, int nn, double* cs, double* red, cudaStream_t st, int max_sweeps) {
  const int np = nn + (nn & 1);
  {
    const long long tot = static_cast<long long>(nn) * nn;
    k_eye<<<static_cast<unsigned>((tot + 255) / 256), 256, 0, st>>>(Vt, nn);
    PCA_TRY(cudaGetLastError());
  }
  const size_t apply_smem = 2 * static_cast<size_t>(nn) * sizeof(double);
  PCA_TRY(cudaFuncSetAttribute(k_jacobi_apply, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(apply_smem)));
  double prev_off = -1.0;
  for (int sweep = 0; sweep < max_sweeps && nn > 1; ++sweep) {
    for (int s = 0; s < np - 1; ++s) {
      k_jacobi_params<<<(np / 2 + 127) / 128, 128, 0, st>>>(A, nn, np, s, cs);
      k_jacobi_apply<<<np / 2, 256, apply_smem, st>>>(A, Vt, nn, np, s, cs);
    }
    PCA_TRY(cudaGetLastError());
    PCA_TRY(cudaMemsetAsync(red, 0, 2 * sizeof(double), st));
    k_offnorm<<<304, 256, 0, st>>>(A, nn, red);
    PCA_TRY(cudaGetLastError());
    double h[2];
    PCA_TRY(cudaMemcpyAsync(h, red, sizeof(h), cudaMemcpyDeviceToHost, st));
    PCA_TRY(cudaStreamSynchronize(st));
    const double off = std::sqrt(h[0]), tot = std::sqrt(h[1]);
    if (!(off > 1e-11 * tot)) break;
    if (prev_off >= 0.0 && sweep >= 4 && off > 0.5 * prev_off) break;  // rounding floor
    prev_off = off;
  }
  return EOGP_OK;
}

int fit_dense(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype, float* eig,
              char* ws, cudaStream_t st, const double* C_in, int ldc) {
  const DenseLayout L = dense_layout(C_in ? m : n, m, k);
  double* A = reinterpret_cast<double*>(ws + L.A);
  double* Vt = reinterpret_cast<double*>(ws + L.Vt);
  double* cs = reinterpret_cast<double*>(ws + L.cs);
  double* mu = reinterpret_cast<double*>(ws + L.mu);
  int* sel = reinterpret_cast<int*>(ws + L.sel);
  double* red = reinterpret_cast<double*>(ws + L.red);
  const bool gram = !C_in && n < m;
  const int nn = gram ? n : m;
  if (gram) {
    // A = Z Z^T (n x n)
    PCA_TRY(gemm_f64acc<float>(n, n, m, 1.0, Z, ldz, 1, Z, ldz, 1, A, n, st));
  } else if (C_in) {
    // A = C / n from a second moment summed elsewhere (e.g. over shards)
    k_scale_copy<<<static_cast<unsigned>((static_cast<long long>(m) * m + 255) / 256), 256, 0, st>>>(
        C_in, ldc, m, 1.0 / n, A);
    PCA_TRY(cudaGetLastError());
  } else {
    // A = Z^T Z / n (m x m): A(i,j) = sum_r Z[r][i] Z[r][j]
    PCA_TRY(gemm_f64acc<float>(m, m, n, 1.0 / n, Z, 1, ldz, Z, 1, ldz, A, m, st));
  }
  if (int rc = jacobi_eigen(A, Vt, nn, cs, red, st, 40)) return rc;
  k_rank<<<(nn + 255) / 256, 256, 0, st>>>(A, nn, k, mu, sel);
  PCA_TRY(cudaGetLastError());
  const int bf = pt_dtype == EOGP_BF16 ? 1 : 0;
  if (!gram) {
    k_emit<double><<<k, 256, 0, st>>>(Vt, nn, sel, m, Pt, ld_pt, bf, mu, 1.0, eig);
    PCA_TRY(cudaGetLastError());
  } else {
    double* Pr = reinterpret_cast<double*>(ws + L.Pr);
    // U_k rows (eigenvectors of Z Z^T) -> A's storage, then Pr = U_k Z (k x m).
    k_gather_f64_rows<<<k, 256, 0, st>>>(Vt, nn, sel, nn, A);
    PCA_TRY(cudaGetLastError());
    // Pr[r][c] = sum_x U[r][x] Z[x][c]
    PCA_TRY(gemm_f64acc<double>(k, m, n, 1.0, A, n, 1, Z, 1, ldz, Pr, m, st));
    k_emit<double><<<k, 256, 0, st>>>(Pr, m, nullptr, m, Pt, ld_pt, bf, mu, 1.0 / n, nullptr);
    PCA_TRY(cudaGetLastError());
    // eigenvalues of Z^T Z / n: mu[sel[r]] / n
    k_eig_out<<<(k + 255) / 256, 256, 0, st>>>(mu, sel, k, 1.0 / n, eig);
    PCA_TRY(cudaGetLastError());
  }
  return EOGP_OK;
}

// One Cholesky-QR pass: X32 (rows of X^T, p x nn4) <- orthonormal basis of the rows of Y32
// (which may be the same buffer): rows normalised, G = Y Y^T (tensor cores),
// L = chol(G + rel * mean(diag G) I), X^T = L^-1 Y^T.
int chol_qr_pass(const SubLayout& L, char* w, const float* Y32, float* X32, float rel, unsigned* status,
                 cudaStream_t st) {
  const int p = L.p, nn = L.nn;
  float* rs = reinterpret_cast<float*>(w + L.rs);
  bf16* Yh = reinterpret_cast<bf16*>(w + L.Yh);
  bf16* Yl = reinterpret_cast<bf16*>(w + L.Yl);
  bf16* YTh = reinterpret_cast<bf16*>(w + L.YTh);
  bf16* YTl = reinterpret_cast<bf16*>(w + L.YTl);
  float* G = reinterpret_cast<float*>(w + L.G32);
  float* Li = reinterpret_cast<float*>(w + L.Li32);
  bf16* Sh = reinterpret_cast<bf16*>(w + L.Sh);
  bf16* Sl = reinterpret_cast<bf16*>(w + L.Sl);
  float* shift = reinterpret_cast<float*>(w + L.shift);
  k_row_invnorm<<<p, 256, 0, st>>>(Y32, L.nn4, nn, rs);
  k_split_rows<<<grid_for(static_cast<long long>(p) * L.nn8), 256, 0, st>>>(Y32, L.nn4, p, nn, rs, Yh, Yl, L.nn8);
  k_split_T<<<dim3((nn + 31) / 32, (L.p8 + 31) / 32), dim3(32, 8), 0, st>>>(Y32, L.nn4, p, nn, rs, YTh, YTl, L.p8);
  PCA_TRY(cudaGetLastError());
  PCA_TRY(launch_tc_gemm_hl(p, p, nn, Yh, Yl, L.nn8, Yh, Yl, L.nn8, G, L.p4, 1.0f, status, st));
  k_diag_shift<<<1, 256, 0, st>>>(G, L.p4, p, rel, shift);
  k_add_diag<<<(p + 255) / 256, 256, 0, st>>>(G, L.p4, p, shift);
  PCA_TRY(cudaGetLastError());
  for (int j0 = 0; j0 < p; j0 += 32) {
    k_chol_diag<<<1, dim3(32, 32), 0, st>>>(G, L.p4, p, j0, status);
    const int below = p - (j0 + 32);
    if (below > 0) {
      k_chol_panel<<<(below + 127) / 128, 128, 0, st>>>(G, L.p4, p, j0);
      const int nt = (below + 63) / 64;
      k_chol_update<<<nt * (nt + 1) / 2, 256, 0, st>>>(G, L.p4, p, j0);
    }
  }
  PCA_TRY(cudaGetLastError());
  PCA_TRY(cudaMemsetAsync(Li, 0, static_cast<size_t>(p) * L.p4 * 4, st));
  const int nblk = (p + 31) / 32;
  k_trinv_diag<<<nblk, 32, 0, st>>>(G, L.p4, Li, L.p4, p);
  for (int d = 1; d < nblk; ++d) k_trinv_off<<<nblk - d, 256, 0, st>>>(G, L.p4, Li, L.p4, p, d);
  PCA_TRY(cudaGetLastError());
  k_split_rows<<<grid_for(static_cast<long long>(p) * L.p8), 256, 0, st>>>(Li, L.p4, p, p, nullptr, Sh, Sl, L.p8);
  PCA_TRY(cudaGetLastError());
  // X^T[j][l] = sum_i Li[j][i] Y^T[i][l]: A operand Li (K = p), B operand Y [nn][p8]
  PCA_TRY(launch_tc_gemm_hl(p, nn, p, Sh, Sl, L.p8, YTh, YTl, L.p8, X32, L.nn4, 1.0f, status, st));
  return EOGP_OK;
}

int orthonormalise(const SubLayout& L, char* w, const float* Y32, float* X32, unsigned* status, cudaStream_t st) {
  if (int rc = chol_qr_pass(L, w, Y32, X32, 1e-2f, status, st)) return rc;
  if (int rc = chol_qr_pass(L, w, X32, X32, 1e-4f, status, st)) return rc;
  return chol_qr_pass(L, w, X32, X32, 0.0f, status, st);
}

// CX32 = (A X)^T = X^T A: rows of X^T split, times the symmetric A (hi/lo).
int apply_A(const SubLayout& L, char* w, const float* X32, float* CX32, unsigned* status, cudaStream_t st) {
  bf16* Yh = reinterpret_cast<bf16*>(w + L.Yh);
  bf16* Yl = reinterpret_cast<bf16*>(w + L.Yl);
  k_split_rows<<<grid_for(static_cast<long long>(L.p) * L.nn8), 256, 0, st>>>(X32, L.nn4, L.p, L.nn, nullptr, Yh,
                                                                             Yl, L.nn8);
  PCA_TRY(cudaGetLastError());
  PCA_TRY(launch_tc_gemm_hl(L.p, L.nn, L.nn, Yh, Yl, L.nn8, w + L.Ah, w + L.Al, L.nn8, CX32, L.nn4, 1.0f, status,
                            st));
  return EOGP_OK;
}

// Rayleigh-Ritz: H = X^T (A X), eigenpairs, X and A X rotated onto the Ritz
// vectors (descending); returns the largest relative residual of the top k.
int rayleigh_ritz(const SubLayout& L, char* w, int k, unsigned* status, cudaStream_t st, float* max_res) {
  const int p = L.p, nn = L.nn;
  float* X32 = reinterpret_cast<float*>(w + L.X32);
  float* CX32 = reinterpret_cast<float*>(w + L.CX32);
  bf16* Yh = reinterpret_cast<bf16*>(w + L.Yh);
  bf16* Yl = reinterpret_cast<bf16*>(w + L.Yl);
  bf16* YTh = reinterpret_cast<bf16*>(w + L.YTh);
  bf16* YTl = reinterpret_cast<bf16*>(w + L.YTl);
  bf16* CTh = reinterpret_cast<bf16*>(w + L.CTh);
  bf16* CTl = reinterpret_cast<bf16*>(w + L.CTl);
  float* H = reinterpret_cast<float*>(w + L.G32);
  float* S32 = reinterpret_cast<float*>(w + L.Li32);
  bf16* Sh = reinterpret_cast<bf16*>(w + L.Sh);
  bf16* Sl = reinterpret_cast<bf16*>(w + L.Sl);
  double* H64 = reinterpret_cast<double*>(w + L.H64);
  double* V64 = reinterpret_cast<double*>(w + L.V64);
  double* mu = reinterpret_cast<double*>(w + L.mu);
  int* sel = reinterpret_cast<int*>(w + L.sel);
  float* theta = reinterpret_cast<float*>(w + L.theta);
  unsigned* resid = reinterpret_cast<unsigned*>(w + L.resid);
  // H = X^T (A X): rows of X^T and rows of (A X)^T, K = nn
  k_split_rows<<<grid_for(static_cast<long long>(p) * L.nn8), 256, 0, st>>>(X32, L.nn4, p, nn, nullptr, Yh, Yl,
                                                                          L.nn8);
  k_split_rows<<<grid_for(static_cast<long long>(p) * L.nn8), 256, 0, st>>>(CX32, L.nn4, p, nn, nullptr, YTh,
                                                                          YTl, L.nn8);
  PCA_TRY(cudaGetLastError());
  PCA_TRY(launch_tc_gemm_hl(p, p, nn, Yh, Yl, L.nn8, YTh, YTl, L.nn8, H, L.p4, 1.0f, status, st));
  k_sym_f64<<<grid_for(static_cast<long long>(p) * p), 256, 0, st>>>(H, L.p4, p, H64);
  PCA_TRY(cudaGetLastError());
  if (int rc = jacobi_eigen(H64, V64, p, reinterpret_cast<double*>(w + L.cs), reinterpret_cast<double*>(w + L.red),
                            st, 40))
    return rc;
  k_rank<<<(p + 255) / 256, 256, 0, st>>>(H64, p, p, mu, sel);
  k_ritz_rows<<<p, 256, 0, st>>>(V64, p, sel, mu, S32, L.p4, theta);
  k_split_rows<<<grid_for(static_cast<long long>(p) * L.p8), 256, 0, st>>>(S32, L.p4, p, p, nullptr, Sh, Sl, L.p8);
  // X and A X as K-major operands [nn][p8] (transposed splits)
  k_split_T<<<dim3((nn + 31) / 32, (L.p8 + 31) / 32), dim3(32, 8), 0, st>>>(X32, L.nn4, p, nn, nullptr, YTh, YTl,
                                                                           L.p8);
  k_split_T<<<dim3((nn + 31) / 32, (L.p8 + 31) / 32), dim3(32, 8), 0, st>>>(CX32, L.nn4, p, nn, nullptr, CTh, CTl,
                                                                           L.p8);
  PCA_TRY(cudaGetLastError());
  PCA_TRY(launch_tc_gemm_hl(p, nn, p, Sh, Sl, L.p8, YTh, YTl, L.p8, X32, L.nn4, 1.0f, status, st));
  PCA_TRY(launch_tc_gemm_hl(p, nn, p, Sh, Sl, L.p8, CTh, CTl, L.p8, CX32, L.nn4, 1.0f, status, st));
  PCA_TRY(cudaMemsetAsync(resid, 0, 4, st));
  k_ritz_resid<<<k, 256, 0, st>>>(X32, CX32, L.nn4, nn, theta, resid);
  PCA_TRY(cudaGetLastError());
  unsigned hbits = 0;
  PCA_TRY(cudaMemcpyAsync(&hbits, resid, 4, cudaMemcpyDeviceToHost, st));
  PCA_TRY(cudaStreamSynchronize(st));
  float v;
  std::memcpy(&v, &hbits, 4);
  *max_res = v;
  return EOGP_OK;
}

int fit_subspace(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype, float* eig,
                 char* w, unsigned* status, cudaStream_t st, const double* C_in, int ldc) {
  const bool gram = !C_in && n < m;
  const SubLayout L = sub_layout(C_in ? m : n, m, k, !C_in);
  const int nn = L.nn, p = L.p;
  float* A32 = reinterpret_cast<float*>(w + L.A32);
  // 1. A = Z^T Z / n or Z Z^T / n (tensor cores), or C / n; symmetrised hi/lo pair
  if (C_in) {
    k_f64_to_f32<<<grid_for(static_cast<long long>(m) * m), 256, 0, st>>>(C_in, ldc, m, 1.0 / n, A32, L.nn8);
    PCA_TRY(cudaGetLastError());
  } else {
    bf16* ZTh = reinterpret_cast<bf16*>(w + L.ZTh);
    bf16* ZTl = reinterpret_cast<bf16*>(w + L.ZTl);
    k_split_T<<<dim3((m + 31) / 32, (L.n8 + 31) / 32), dim3(32, 8), 0, st>>>(Z, ldz, n, m, nullptr, ZTh, ZTl, L.n8);
    PCA_TRY(cudaGetLastError());
    if (gram) {
      bf16* Zh = reinterpret_cast<bf16*>(w + L.Zh);
      bf16* Zl = reinterpret_cast<bf16*>(w + L.Zl);
      k_split_rows<<<grid_for(static_cast<long long>(n) * L.m8), 256, 0, st>>>(Z, ldz, n, m, nullptr, Zh, Zl, L.m8);
      PCA_TRY(cudaGetLastError());
      PCA_TRY(launch_tc_gemm_hl(n, n, m, Zh, Zl, L.m8, Zh, Zl, L.m8, A32, L.nn8, 1.0f / n, status, st));
    } else {
      PCA_TRY(launch_tc_gemm_hl(m, m, n, ZTh, ZTl, L.n8, ZTh, ZTl, L.n8, A32, L.nn8, 1.0f / n, status, st));
    }
  }
  k_split_sym<<<dim3((L.nn8 + 31) / 32, (nn + 31) / 32), dim3(32, 8), 0, st>>>(
      A32, L.nn8, nn, reinterpret_cast<bf16*>(w + L.Ah), reinterpret_cast<bf16*>(w + L.Al), L.nn8);
  PCA_TRY(cudaGetLastError());
  // 2. start: orthonormal basis of p Gaussian rows
  float* X32 = reinterpret_cast<float*>(w + L.X32);
  float* CX32 = reinterpret_cast<float*>(w + L.CX32);
  PCA_TRY(cudaMemsetAsync(X32, 0, static_cast<size_t>(p) * L.nn4 * 4, st));
  PCA_TRY(cudaMemsetAsync(CX32, 0, static_cast<size_t>(p) * L.nn4 * 4, st));
  k_gauss<<<grid_for(static_cast<long long>(p) * nn), 256, 0, st>>>(X32, L.nn4, p, nn, 0x5eedull);
  PCA_TRY(cudaGetLastError());
  if (int rc = orthonormalise(L, w, X32, X32, status, st)) return rc;
  // 3. iterate: X <- orth(A X); Rayleigh-Ritz every 5 iterations
  const int kRR = 5, kMaxIt = 400;
  const float kTol = 1e-3f;
  bool converged = false;
  for (int it = 1; it <= kMaxIt; ++it) {
    if (int rc = apply_A(L, w, X32, CX32, status, st)) return rc;
    if (it % kRR == 0) {
      float res = 0.f;
      if (int rc = rayleigh_ritz(L, w, k, status, st, &res)) return rc;
      if (res <= kTol) {
        converged = true;
        break;
      }
    }
    if (int rc = orthonormalise(L, w, CX32, X32, status, st)) return rc;
  }
  if (!converged)
    return eogp::set_error(EOGP_EDEVICE, "fit_pca: subspace iteration did not reach the residual bound in %d "
                           "iterations", kMaxIt);
  // 4. outputs: the top k Ritz pairs
  const int bf = pt_dtype == EOGP_BF16 ? 1 : 0;
  const float* theta = reinterpret_cast<const float*>(w + L.theta);
  if (!gram) {
    k_emit<float><<<k, 256, 0, st>>>(X32, L.nn4, nullptr, m, Pt, ld_pt, bf, nullptr, 1.0, nullptr);
  } else {
    // P rows = U_k^T Z (normalised): A operand rows of U^T (K = n), B operand Z^T [m][n8]
    bf16* Yh = reinterpret_cast<bf16*>(w + L.Yh);
    bf16* Yl = reinterpret_cast<bf16*>(w + L.Yl);
    float* Pr = reinterpret_cast<float*>(w + L.Pr);
    k_split_rows<<<grid_for(static_cast<long long>(k) * L.nn8), 256, 0, st>>>(X32, L.nn4, k, nn, nullptr, Yh, Yl,
                                                                            L.nn8);
    PCA_TRY(cudaGetLastError());
    PCA_TRY(launch_tc_gemm_hl(k, m, n, Yh, Yl, L.nn8, w + L.ZTh, w + L.ZTl, L.n8, Pr, rup(m, 4), 1.0f, status, st));
    k_emit<float><<<k, 256, 0, st>>>(Pr, rup(m, 4), nullptr, m, Pt, ld_pt, bf, nullptr, 1.0, nullptr);
  }
  PCA_TRY(cudaGetLastError());
  k_copy_eig<<<(k + 255) / 256, 256, 0, st>>>(theta, k, eig);
  PCA_TRY(cudaGetLastError());
  return EOGP_OK;
}

}  // namespace

int fit_pca_device(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype,
                   float* eig, void* ws, unsigned* status, cudaStream_t st, const double* C_in, int ldc) {
  const int nn = C_in ? m : std::min(n, m);
  char* w = static_cast<char*>(ws);
  if (use_subspace(nn, k)) return fit_subspace(Z, n, m, ldz, k, Pt, ld_pt, pt_dtype, eig, w, status, st, C_in, ldc);
  return fit_dense(Z, n, m, ldz, k, Pt, ld_pt, pt_dtype, eig, w, st, C_in, ldc);
}

cudaError_t second_moment_device(const float* Z, int n, int m, int ldz, double* C, int ldc, int accumulate,
                                 cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  // C(i,j) (+)= sum_r Z[r][i] Z[r][j]
  return gemm_f64acc<float>(m, m, n, 1.0, Z, 1, ldz, Z, 1, ldz, C, ldc, st, accumulate);
}
