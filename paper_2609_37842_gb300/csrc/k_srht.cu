// EOGP-R second stage (Sec. 3.2 "A scalable alternative to PCA"; App. B.2
// Eq. app_srht_definition): x = sqrt(p/k) R H_p D J z for each first-stage row
// z in R^m, p = 2^ceil(log2 m), H_p the orthonormal Walsh-Hadamard matrix in
// Sylvester order (H_p[r][c] = (-1)^popcount(r & c) / sqrt(p)).
//
// One CTA per row: the signed, zero-padded row is staged in shared memory and
// transformed in place by log2(p) butterfly passes (the unnormalised transform
// W = sqrt(p) H_p), then the kept rows are read out scaled by 1/sqrt(k)
// (sqrt(p/k) / sqrt(p)). The same CTA emits x, and/or the sign codes and
// ||x||_1 / k of Eq. onebit (fixed-order sums: bitwise reproducible).
// O(p log p) work on p floats of shared memory; HBM traffic is the z row in and
// x / codes out, so the kernel is bandwidth- or latency-bound.
#include <cuda_bf16.h>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

namespace {

constexpr int kThreads = 512;

template <bool HILO>
__global__ void __launch_bounds__(kThreads) k_srht(const void* __restrict__ z0, const void* __restrict__ z1,
                                                   int ldz, int m, int p, const int8_t* __restrict__ signs,
                                                   const int32_t* __restrict__ rows, int k, float scale,
                                                   float* __restrict__ x, int ldx, uint32_t* __restrict__ codes,
                                                   int ld_codes, float* __restrict__ scales, int ld_scales,
                                                   unsigned* status) {
  extern __shared__ float v[];
  __shared__ float wsum[kThreads / 32];
  const int b = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // J and D: signed row, zero-padded to p.
  for (int c = tid; c < p; c += kThreads) {
    float zc = 0.f;
    if (c < m) {
      if (HILO) {
        const size_t o = static_cast<size_t>(b) * ldz + c;
        zc = __bfloat162float(static_cast<const __nv_bfloat16*>(z0)[o]) +
             __bfloat162float(static_cast<const __nv_bfloat16*>(z1)[o]);
      } else {
        zc = static_cast<const float*>(z0)[static_cast<size_t>(b) * ldz + c];
      }
      if (signs[c] < 0) zc = -zc;
    }
    v[c] = zc;
  }
  __syncthreads();
  // Butterflies: pass h pairs (i, i + h) inside blocks of 2h.
  for (int lh = 0; (1 << lh) < p; ++lh) {
    const int h = 1 << lh;
    for (int t = tid; t < (p >> 1); t += kThreads) {
      const int i = ((t >> lh) << (lh + 1)) | (t & (h - 1));
      const float a0 = v[i], a1 = v[i + h];
      v[i] = a0 + a1;
      v[i + h] = a0 - a1;
    }
    __syncthreads();
  }
  // R and the normalisation; codes and the scale from the same values.
  float acc = 0.f;
  bool bad = false;
  for (int base = warp * 32; base < k; base += kThreads) {
    const int r = base + lane;
    float xr = 0.f;
    if (r < k) {
      const int row = rows[r];
      if (row < 0 || row >= p) {
        bad = true;
      } else {
        xr = v[row] * scale;
      }
      if (x) x[static_cast<size_t>(b) * ldx + r] = xr;
      bad |= isnan(xr);
      acc += fabsf(xr);
    }
    const uint32_t word = __ballot_sync(0xffffffffu, r < k && xr >= 0.f);
    if (codes && lane == 0) codes[static_cast<size_t>(b) * ld_codes + (base >> 5)] = word;
  }
  if (__any_sync(0xffffffffu, bad) && lane == 0) eogp::flag_status(status, EOGP_ST_DEVICE);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (lane == 0) wsum[warp] = acc;
  __syncthreads();
  if (tid == 0 && scales) {
    float t = 0.f;
    for (int w = 0; w < kThreads / 32; ++w) t += wsum[w];
    scales[static_cast<size_t>(b) * ld_scales] = t / static_cast<float>(k);
  }
}

}  // namespace

int srht_width(int m) {
  int p = 1;
  while (p < m) p <<= 1;
  return p;
}

size_t srht_smem_bytes(int m) { return static_cast<size_t>(srht_width(m)) * 4; }

cudaError_t launch_srht(const void* z0, const void* z1, bool hilo, int ldz, int B, int m,
                        const int8_t* signs, const int32_t* rows, int k, float* x, int ldx,
                        uint32_t* codes, int ld_codes, float* scales, int ld_scales, unsigned* status,
                        cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  const int p = srht_width(m);
  const size_t smem = srht_smem_bytes(m);
  const float scale = 1.0f / sqrtf(static_cast<float>(k));
  if (hilo) {
    cudaError_t e = cudaFuncSetAttribute(k_srht<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    k_srht<true><<<B, kThreads, smem, st>>>(z0, z1, ldz, m, p, signs, rows, k, scale, x, ldx, codes,
                                            ld_codes, scales, ld_scales, status);
  } else {
    cudaError_t e = cudaFuncSetAttribute(k_srht<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    k_srht<false><<<B, kThreads, smem, st>>>(z0, z1, ldz, m, p, signs, rows, k, scale, x, ldx, codes,
                                             ld_codes, scales, ld_scales, status);
  }
  return cudaGetLastError();
}
