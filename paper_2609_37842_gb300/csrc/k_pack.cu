// One-bit encoding (Sec. 3.3, Eq. onebit): per row x in R^k, sign bits packed
// LSB-first into 32-bit words (bit c % 32 of word c / 32 is [x_c >= 0]; the
// per-module byte packing of App. E.1 read as little-endian words) and the
// scale ||x||_1 / k. The same kernel finalises the split-K projection: x is
// the fixed-order sum of `splits` partial slabs.
//
// Full 128-column chunks use float4 loads: each lane holds 4 columns, forms a
// 4-bit nibble, and 8 lanes OR their nibbles into one word. The remainder uses
// one column per lane and a warp ballot. HBM-bound: it reads 4k bytes per row
// (times `splits`) and writes k/8 + 4.
#include <algorithm>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

namespace {

__device__ __forceinline__ float4 ld_stream4(const float* p) {
  return __ldcs(reinterpret_cast<const float4*>(p));
}

// ROW_WARPS = 8: one block (8 warps) per row, for small batches: 128-column
// chunks go to warps round-robin, each warp sums |x| over its chunks in column
// order and the 8 warp totals are added in warp order.
// ROW_WARPS = 1: one warp per row, rows strided over the grid, for large
// batches (more rows in flight, no block-level reduction).
// Either way the scale is bitwise reproducible.
template <int ROW_WARPS>
__device__ __forceinline__ void pack_row(const float* __restrict__ part, int splits, size_t slab,
                                         int ldp, int k, float* __restrict__ x_out, int ldx,
                                         uint32_t* __restrict__ codes, int ld_codes,
                                         float* __restrict__ scales, int ld_scales,
                                         unsigned* status, int row, int warp, int lane,
                                         float* wsum) {
  const float* src = part + static_cast<size_t>(row) * ldp;
  float* xo = x_out ? x_out + static_cast<size_t>(row) * ldx : nullptr;
  uint32_t* co = codes ? codes + static_cast<size_t>(row) * ld_codes : nullptr;
  float acc = 0.f;
  bool bad = false;

  const bool vec = ((ldp & 3) == 0) && ((reinterpret_cast<uintptr_t>(part) & 15) == 0) &&
                   ((slab & 3) == 0) &&
                   (x_out == nullptr ||
                    (((ldx & 3) == 0) && ((reinterpret_cast<uintptr_t>(x_out) & 15) == 0)));
  const int nfull = vec ? (k >> 7) : 0;
  // Up to 8 chunks per batch: all loads of a batch are issued before any is used.
  for (int it0 = warp; it0 < nfull; it0 += 8 * ROW_WARPS) {
    float4 vb[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int it = it0 + j * ROW_WARPS;
      if (it < nfull) {
        const int c = (it << 7) + (lane << 2);
        vb[j] = ld_stream4(src + c);
        for (int s = 1; s < splits; ++s) {
          const float4 w = ld_stream4(src + static_cast<size_t>(s) * slab + c);
          vb[j].x += w.x;
          vb[j].y += w.y;
          vb[j].z += w.z;
          vb[j].w += w.w;
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
    const int it = it0 + j * ROW_WARPS;
    if (it >= nfull) break;
    const int c = (it << 7) + (lane << 2);
    const float4 v = vb[j];
    if (xo) *reinterpret_cast<float4*>(xo + c) = v;
    bad |= isnan(v.x) | isnan(v.y) | isnan(v.z) | isnan(v.w);
    acc += fabsf(v.x);
    acc += fabsf(v.y);
    acc += fabsf(v.z);
    acc += fabsf(v.w);
    const uint32_t nib = (v.x >= 0.f ? 1u : 0u) | (v.y >= 0.f ? 2u : 0u) |
                         (v.z >= 0.f ? 4u : 0u) | (v.w >= 0.f ? 8u : 0u);
    uint32_t word = nib << (4 * (lane & 7));
    word |= __shfl_xor_sync(0xffffffffu, word, 1);
    word |= __shfl_xor_sync(0xffffffffu, word, 2);
    word |= __shfl_xor_sync(0xffffffffu, word, 4);
    if (co && (lane & 7) == 0) co[(it << 2) + (lane >> 3)] = word;
    }
  }
  // Remainder (or everything, when unaligned): 32-column words, one column per lane.
  const int c0 = nfull << 7;
  for (int base = c0 + 32 * warp; base < k; base += 32 * ROW_WARPS) {
    const int c = base + lane;
    const bool in = c < k;
    float v = 0.f;
    if (in) {
      v = src[c];
      for (int s = 1; s < splits; ++s) v += src[static_cast<size_t>(s) * slab + c];
      if (xo) xo[c] = v;
      bad |= isnan(v);
      acc += fabsf(v);
    }
    const uint32_t word = __ballot_sync(0xffffffffu, in && v >= 0.f);
    if (co && lane == 0) co[base >> 5] = word;
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if (__any_sync(0xffffffffu, bad) && lane == 0) eogp::flag_status(status, EOGP_ST_DEVICE);
  if (ROW_WARPS == 1) {
    if (lane == 0 && scales) scales[static_cast<size_t>(row) * ld_scales] = acc / static_cast<float>(k);
    return;
  }
  if (lane == 0) wsum[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0 && scales) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += wsum[w];
    scales[static_cast<size_t>(row) * ld_scales] = t / static_cast<float>(k);
  }
}

__global__ void __launch_bounds__(256) k_pack_block_row(const float* __restrict__ part, int splits,
                                                         size_t slab, int ldp, int B, int k,
                                                         float* __restrict__ x_out, int ldx,
                                                         uint32_t* __restrict__ codes, int ld_codes,
                                                         float* __restrict__ scales, int ld_scales,
                                                         unsigned* status) {
  __shared__ float wsum[8];
  pack_row<8>(part, splits, slab, ldp, k, x_out, ldx, codes, ld_codes, scales, ld_scales, status,
              blockIdx.x, threadIdx.x >> 5, threadIdx.x & 31, wsum);
}

__global__ void __launch_bounds__(256) k_pack_warp_row(const float* __restrict__ part, int splits,
                                                        size_t slab, int ldp, int B, int k,
                                                        float* __restrict__ x_out, int ldx,
                                                        uint32_t* __restrict__ codes, int ld_codes,
                                                        float* __restrict__ scales, int ld_scales,
                                                        unsigned* status) {
  const int lane = threadIdx.x & 31;
  const int w0 = blockIdx.x * 8 + (threadIdx.x >> 5);
  for (int row = w0; row < B; row += gridDim.x * 8)
    pack_row<1>(part, splits, slab, ldp, k, x_out, ldx, codes, ld_codes, scales, ld_scales, status,
                row, 0, lane, nullptr);
}

}  // namespace

cudaError_t launch_pack(const float* part, int splits, size_t slab, int ldp, int B, int k,
                        float* x_out, int ldx, uint32_t* codes, int ld_codes, float* scales,
                        int ld_scales, unsigned* status, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  if (B < 4096) {
    k_pack_block_row<<<static_cast<unsigned>(B), 256, 0, st>>>(part, splits, slab, ldp, B, k, x_out,
                                                               ldx, codes, ld_codes, scales,
                                                               ld_scales, status);
  } else {
    const int blocks = std::min((B + 7) / 8, 152 * 16);
    k_pack_warp_row<<<static_cast<unsigned>(blocks), 256, 0, st>>>(part, splits, slab, ldp, B, k,
                                                                   x_out, ldx, codes, ld_codes,
                                                                   scales, ld_scales, status);
  }
  return cudaGetLastError();
}
