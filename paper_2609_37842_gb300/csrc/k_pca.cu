// PCA fit of the second stage (App. B.2 "PCA fitting"; Alg. 1 "fit P_u by
// uncentered PCA of {z_iu}"): the top-k eigenvectors of Z^T Z / n, obtained
// from the n x n Gram matrix Z Z^T when n < m (the route the paper describes).
//
// Steps, all on the device:
//  1. A = Z^T Z / n (or Z Z^T): CUDA-core GEMM on the fp32 Z with fp64
//     accumulation (accuracy over speed; the fit is a one-time cost).
//  2. Cyclic two-sided Jacobi (Golub & Van Loan, Sec. 8.5) in round-robin
//     ("circle") order: each step rotates n'/2 disjoint (p, q) pairs. One
//     kernel forms the rotations (in double) from the current A; a second
//     applies J^T A J to rows p, q of A (row rotation, then the column
//     rotations of every pair inside the two rows held in shared memory) and
//     J^T to rows p, q of V^T. Sweeps repeat until the off-diagonal mass stops
//     shrinking or falls below 1e-11 of ||A||_F. A and V^T are kept in fp64 so
//     that mid-spectrum eigenvalues keep ~1e-10 relative accuracy.
//  3. Rank the eigenvalues (descending, ties to the lower index), keep the top
//     k, map Gram-route vectors through Z^T u / ||Z^T u||, normalise, and fix
//     each vector's sign so its largest-magnitude entry is positive.
#include <cmath>
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
__global__ void __launch_bounds__(256) k_emit(const double* __restrict__ src, int ld_src,
                                              const int* __restrict__ sel, int m,
                                              void* __restrict__ Pt, int ld_pt, int bf16_out,
                                              const double* __restrict__ mu, double eig_scale,
                                              float* __restrict__ eig) {
  __shared__ double s_ss[256];
  __shared__ double s_mx[256];
  __shared__ int s_ix[256];
  const int r = blockIdx.x;
  const double* v = src + static_cast<size_t>(sel ? sel[r] : r) * ld_src;
  double ss = 0.0, mx = -1.0;
  int ix = 0x7fffffff;
  for (int c = threadIdx.x; c < m; c += blockDim.x) {
    const double x = v[c];
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
  const double sgn = v[s_ix[0]] < 0.0 ? -1.0 : 1.0;
  const double f = nrm > 0.0 ? sgn / nrm : 0.0;
  for (int c = threadIdx.x; c < m; c += blockDim.x) {
    const float o = static_cast<float>(v[c] * f);
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

}  // namespace

size_t fit_pca_ws_bytes(int n, int m, int k) {
  const size_t np = static_cast<size_t>(n < m ? n : m);
  size_t b = 0;
  b += al256(np * np * sizeof(double));           // A
  b += al256(np * np * sizeof(double));           // Vt
  b += al256((np / 2 + 1) * 2 * sizeof(double));  // cs
  b += al256(np * sizeof(double));                // mu
  b += al256(static_cast<size_t>(k) * sizeof(int));
  b += al256(4 * sizeof(double));
  if (n < m) b += al256(static_cast<size_t>(k) * m * sizeof(double));  // Pr
  return b;
}

int fit_pca_device(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype,
                   float* eig, PcaWs ws, unsigned* status, cudaStream_t st, const double* C_in,
                   int ldc) {
  (void)status;
  const bool gram = !C_in && n < m;
  const int nn = gram ? n : m;
  const int np = nn + (nn & 1);
  cudaError_t e;
#define PCA_TRY(x)                                                                         \
  do {                                                                                     \
    e = (x);                                                                               \
    if (e != cudaSuccess)                                                                  \
      return eogp::set_error(EOGP_ECUDA, "fit_pca: %s: %s", #x, cudaGetErrorString(e));    \
  } while (0)

  if (gram) {
    // A = Z Z^T (n x n)
    PCA_TRY(gemm_f64acc<float>(n, n, m, 1.0, Z, ldz, 1, Z, ldz, 1, ws.A, n, st));
  } else if (C_in) {
    // A = C / n from a second moment summed elsewhere (e.g. over shards)
    k_scale_copy<<<static_cast<unsigned>((static_cast<long long>(m) * m + 255) / 256), 256, 0, st>>>(
        C_in, ldc, m, 1.0 / n, ws.A);
    PCA_TRY(cudaGetLastError());
  } else {
    // A = Z^T Z / n (m x m): A(i,j) = sum_r Z[r][i] Z[r][j]
    PCA_TRY(gemm_f64acc<float>(m, m, n, 1.0 / n, Z, 1, ldz, Z, 1, ldz, ws.A, m, st));
  }
  {
    const long long tot = static_cast<long long>(nn) * nn;
    k_eye<<<static_cast<unsigned>((tot + 255) / 256), 256, 0, st>>>(ws.Vt, nn);
    PCA_TRY(cudaGetLastError());
  }
  const size_t apply_smem = 2 * static_cast<size_t>(nn) * sizeof(double);
  PCA_TRY(cudaFuncSetAttribute(k_jacobi_apply, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(apply_smem)));
  double prev_off = -1.0;
  const int max_sweeps = 40;
  for (int sweep = 0; sweep < max_sweeps && nn > 1; ++sweep) {
    for (int s = 0; s < np - 1; ++s) {
      k_jacobi_params<<<(np / 2 + 127) / 128, 128, 0, st>>>(ws.A, nn, np, s, ws.cs);
      k_jacobi_apply<<<np / 2, 256, apply_smem, st>>>(ws.A, ws.Vt, nn, np, s, ws.cs);
    }
    PCA_TRY(cudaGetLastError());
    PCA_TRY(cudaMemsetAsync(ws.red, 0, 2 * sizeof(double), st));
    k_offnorm<<<304, 256, 0, st>>>(ws.A, nn, ws.red);
    PCA_TRY(cudaGetLastError());
    double red[2];
    PCA_TRY(cudaMemcpyAsync(red, ws.red, sizeof(red), cudaMemcpyDeviceToHost, st));
    PCA_TRY(cudaStreamSynchronize(st));
    const double off = std::sqrt(red[0]), tot = std::sqrt(red[1]);
    if (!(off > 1e-11 * tot)) break;
    if (prev_off >= 0.0 && sweep >= 4 && off > 0.5 * prev_off) break;  // rounding floor
    prev_off = off;
  }
  k_rank<<<(nn + 255) / 256, 256, 0, st>>>(ws.A, nn, k, ws.mu, ws.sel);
  PCA_TRY(cudaGetLastError());
  const int bf = pt_dtype == EOGP_BF16 ? 1 : 0;
  if (!gram) {
    k_emit<<<k, 256, 0, st>>>(ws.Vt, nn, ws.sel, m, Pt, ld_pt, bf, ws.mu, 1.0, eig);
    PCA_TRY(cudaGetLastError());
  } else {
    // U_k rows (eigenvectors of Z Z^T) -> A's storage, then Pr = U_k Z (k x m).
    k_gather_f64_rows<<<k, 256, 0, st>>>(ws.Vt, nn, ws.sel, nn, ws.A);
    PCA_TRY(cudaGetLastError());
    // Pr[r][c] = sum_x U[r][x] Z[x][c]
    PCA_TRY(gemm_f64acc<double>(k, m, n, 1.0, ws.A, n, 1, Z, 1, ldz, ws.Pr, m, st));
    k_emit<<<k, 256, 0, st>>>(ws.Pr, m, nullptr, m, Pt, ld_pt, bf, ws.mu, 1.0 / n, nullptr);
    PCA_TRY(cudaGetLastError());
    // eigenvalues of Z^T Z / n: mu[sel[r]] / n
    k_eig_out<<<(k + 255) / 256, 256, 0, st>>>(ws.mu, ws.sel, k, 1.0 / n, eig);
    PCA_TRY(cudaGetLastError());
  }
#undef PCA_TRY
  return EOGP_OK;
}

cudaError_t second_moment_device(const float* Z, int n, int m, int ldz, double* C, int ldc, int accumulate,
                                 cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  // C(i,j) (+)= sum_r Z[r][i] Z[r][j]
  return gemm_f64acc<float>(m, m, n, 1.0, Z, 1, ldz, Z, 1, ldz, C, ldc, st, accumulate);
}
