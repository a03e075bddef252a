// fp32 CUDA-core kernels: the EOGP_F32 path of eogp_compress_layer, the FP
// score mode, the Gram / covariance matrices of the PCA fit, and the row
// gather used to lay out retained eigenvectors.
//
//  k_simt_gemm: C[i][j] = alpha * sum_k A(i,k) B(j,k) with arbitrary element
//    strides, 64 x 64 tile per block, 4 x 4 per thread, fp32 FMA accumulation.
//  k_contract_f32: one thread per (example, retained coordinate r):
//    z[b][r] = scale[r] * sum_t S~[b,t][posR[r]] * A~[b,t][posC[r]]
//    (Eq. first_stage through the Kronecker identity of Sec. 2.2).
#include <algorithm>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

namespace {

__global__ void __launch_bounds__(256) k_simt_gemm(int M, int N, int K, float alpha,
                                                   const float* __restrict__ A, long long sai,
                                                   long long sak, const float* __restrict__ B,
                                                   long long sbj, long long sbk,
                                                   float* __restrict__ C, long long ldc) {
  __shared__ float As[16][65];
  __shared__ float Bs[16][65];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int i0 = blockIdx.y * 64, j0 = blockIdx.x * 64;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;
  const bool a_k_fast = (sak == 1);
  const bool b_k_fast = (sbk == 1);
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int r = 0; r < 4; ++r) {
      const int e = tid + 256 * r;
      int ii, kk;
      if (a_k_fast) { ii = e >> 4; kk = e & 15; } else { kk = e >> 6; ii = e & 63; }
      float v = 0.f;
      if (i0 + ii < M && k0 + kk < K) v = A[(i0 + ii) * sai + (k0 + kk) * sak];
      As[kk][ii] = v;
      int jj, kb;
      if (b_k_fast) { jj = e >> 4; kb = e & 15; } else { kb = e >> 6; jj = e & 63; }
      float w = 0.f;
      if (j0 + jj < N && k0 + kb < K) w = B[(j0 + jj) * sbj + (k0 + kb) * sbk];
      Bs[kb][jj] = w;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int x = 0; x < 4; ++x) a[x] = As[kk][ty + 16 * x];
#pragma unroll
      for (int x = 0; x < 4; ++x) b[x] = Bs[kk][tx + 16 * x];
#pragma unroll
      for (int x = 0; x < 4; ++x)
#pragma unroll
        for (int y = 0; y < 4; ++y) acc[x][y] = fmaf(a[x], b[y], acc[x][y]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int x = 0; x < 4; ++x) {
    const int i = i0 + ty + 16 * x;
    if (i >= M) continue;
#pragma unroll
    for (int y = 0; y < 4; ++y) {
      const int j = j0 + tx + 16 * y;
      if (j < N) C[i * ldc + j] = alpha * acc[x][y];
    }
  }
}

__global__ void k_contract_f32(const float* __restrict__ At, int ldA, const float* __restrict__ St,
                               int ldS, int B, int T, int m, const int32_t* __restrict__ posR,
                               const int32_t* __restrict__ posC, const float* __restrict__ scale,
                               float* __restrict__ z, int ldz) {
  const long long idx = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x;
  if (idx >= static_cast<long long>(B) * m) return;
  const int b = static_cast<int>(idx / m), r = static_cast<int>(idx % m);
  const int pr = posR[r], pc = posC[r];
  const float* s = St + static_cast<size_t>(b) * T * ldS + pr;
  const float* a = At + static_cast<size_t>(b) * T * ldA + pc;
  float acc = 0.f;
  for (int t = 0; t < T; ++t) acc = fmaf(s[static_cast<size_t>(t) * ldS], a[static_cast<size_t>(t) * ldA], acc);
  z[static_cast<size_t>(b) * ldz + r] = scale[r] * acc;
}

template <typename E>
__global__ void k_gather_rows(const E* __restrict__ src, int ld_src, const int32_t* __restrict__ idx,
                              int row_len, E* __restrict__ dst) {
  const int r = blockIdx.x;
  const E* s = src + static_cast<size_t>(idx[r]) * ld_src;
  E* d = dst + static_cast<size_t>(r) * row_len;
  for (int c = threadIdx.x; c < row_len; c += blockDim.x) d[c] = s[c];
}

}  // namespace

cudaError_t launch_simt_gemm(int M, int N, int K, float alpha, const float* A, long long sai,
                             long long sak, const float* Bm, long long sbj, long long sbk,
                             float* C, long long ldc, cudaStream_t st) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  dim3 grid((N + 63) / 64, (M + 63) / 64);
  k_simt_gemm<<<grid, 256, 0, st>>>(M, N, K, alpha, A, sai, sak, Bm, sbj, sbk, C, ldc);
  return cudaGetLastError();
}

cudaError_t launch_contract_f32(const float* At, int ldA, const float* St, int ldS, int B, int T,
                                int m, const int32_t* posR, const int32_t* posC,
                                const float* scale, float* z, int ldz, cudaStream_t st) {
  const long long n = static_cast<long long>(B) * m;
  if (n <= 0) return cudaSuccess;
  k_contract_f32<<<static_cast<unsigned>((n + 255) / 256), 256, 0, st>>>(At, ldA, St, ldS, B, T, m,
                                                                        posR, posC, scale, z, ldz);
  return cudaGetLastError();
}

cudaError_t launch_gather_rows(const void* src, int ld_src, int elem_bytes, const int32_t* idx,
                               int n_rows, int row_len, void* dst, cudaStream_t st) {
  if (n_rows <= 0) return cudaSuccess;
  if (elem_bytes == 4)
    k_gather_rows<uint32_t><<<n_rows, 256, 0, st>>>(static_cast<const uint32_t*>(src), ld_src, idx,
                                                    row_len, static_cast<uint32_t*>(dst));
  else
    k_gather_rows<uint16_t><<<n_rows, 256, 0, st>>>(static_cast<const uint16_t*>(src), ld_src, idx,
                                                    row_len, static_cast<uint16_t*>(dst));
  return cudaGetLastError();
}

namespace {
// sumsq[j * ld + i] = (accumulate ? sumsq : 0) + G[j][i]^2 in fp64 (G dense [rows][cols]).
__global__ void k_sq_accum(const float* __restrict__ G, int rows, int cols, double* __restrict__ sumsq,
                           int ld, int accumulate) {
  const long long n = static_cast<long long>(rows) * cols;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const double g = static_cast<double>(G[e]);
    const size_t o = static_cast<size_t>(e / cols) * ld + e % cols;
    sumsq[o] = accumulate ? sumsq[o] + g * g : g * g;
  }
}
}  // namespace

cudaError_t launch_sq_accum(const float* G, int rows, int cols, double* sumsq, int ld, int accumulate,
                            cudaStream_t st) {
  const long long n = static_cast<long long>(rows) * cols;
  if (n <= 0) return cudaSuccess;
  const unsigned blocks = static_cast<unsigned>(std::min<long long>((n + 255) / 256, 4096));
  k_sq_accum<<<blocks, 256, 0, st>>>(G, rows, cols, sumsq, ld, accumulate);
  return cudaGetLastError();
}

namespace {
// Row fix-ups of a rotated token matrix X [M x n] (row = b * T + t): add the
// bias-channel term bias[c], or zero the rows of tokens t >= lengths[b].
__global__ void k_rows_fixup(float* __restrict__ X, int M, int n, int ld, int T, const float* __restrict__ bias,
                             const int32_t* __restrict__ lengths) {
  const long long tot = static_cast<long long>(M) * n;
  for (long long e = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; e < tot;
       e += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int row = static_cast<int>(e / n), c = static_cast<int>(e % n);
    float* p = X + static_cast<size_t>(row) * ld + c;
    if (lengths && row % T >= lengths[row / T]) {
      *p = 0.f;
    } else if (bias) {
      *p += bias[c];
    }
  }
}
}  // namespace

cudaError_t launch_rows_fixup(float* X, int M, int n, int ld, int T, const float* bias,
                              const int32_t* lengths, cudaStream_t st) {
  const long long tot = static_cast<long long>(M) * n;
  if (tot <= 0 || (!bias && !lengths)) return cudaSuccess;
  const unsigned blocks = static_cast<unsigned>(std::min<long long>((tot + 255) / 256, 8192));
  k_rows_fixup<<<blocks, 256, 0, st>>>(X, M, n, ld, T, bias, lengths);
  return cudaGetLastError();
}
