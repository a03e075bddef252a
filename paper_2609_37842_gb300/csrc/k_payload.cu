// Store records (App. E.1, Eq. app_payload): per example, for each module in
// order, ceil(k_u / 8) bytes of signs (coordinate c at bit c % 8 of byte
// c / 8: the first bytes of the module's little-endian code words) followed by
// the module's scale as an IEEE half (round to nearest even, little-endian).
// One block per example; byte copies between the word-aligned code rows and the
// byte-packed records. HBM-bound.
#include <cuda_fp16.h>

#include <algorithm>

#include "eogp_internal.h"

namespace {

constexpr int kMaxMods = 1024;

struct PayloadArgs {
  int U;
  int k[kMaxMods];
  int woff[kMaxMods];  // word offset of module u in a code row
  int boff[kMaxMods];  // byte offset of module u's record
};

__global__ void k_payload_pack(const uint32_t* __restrict__ codes, int ld_codes, const float* __restrict__ scales,
                               int ld_scales, uint8_t* __restrict__ out, size_t ld_out,
                               const __grid_constant__ PayloadArgs g) {
  const size_t i = blockIdx.x;
  const uint8_t* crow = reinterpret_cast<const uint8_t*>(codes + i * ld_codes);
  uint8_t* orow = out + i * ld_out;
  for (int u = 0; u < g.U; ++u) {
    const int nb = (g.k[u] + 7) >> 3;
    const uint8_t* src = crow + static_cast<size_t>(g.woff[u]) * 4;
    uint8_t* dst = orow + g.boff[u];
    for (int c = threadIdx.x; c < nb + 2; c += blockDim.x) {
      uint8_t v;
      if (c < nb) {
        v = src[c];
        if (c == nb - 1 && (g.k[u] & 7)) v &= static_cast<uint8_t>((1u << (g.k[u] & 7)) - 1u);
      } else {
        const unsigned short h = __half_as_ushort(__float2half_rn(scales[i * ld_scales + u]));
        v = static_cast<uint8_t>(c == nb ? (h & 0xFF) : (h >> 8));
      }
      dst[c] = v;
    }
  }
}

__global__ void k_payload_unpack(const uint8_t* __restrict__ in, size_t ld_in, uint32_t* __restrict__ codes,
                                 int ld_codes, float* __restrict__ scales, int ld_scales,
                                 const __grid_constant__ PayloadArgs g) {
  const size_t i = blockIdx.x;
  const uint8_t* irow = in + i * ld_in;
  uint8_t* crow = reinterpret_cast<uint8_t*>(codes + i * ld_codes);
  for (int u = 0; u < g.U; ++u) {
    const int nb = (g.k[u] + 7) >> 3;
    const int nwb = ((g.k[u] + 31) >> 5) * 4;  // bytes of the module's code words
    const uint8_t* src = irow + g.boff[u];
    uint8_t* dst = crow + static_cast<size_t>(g.woff[u]) * 4;
    for (int c = threadIdx.x; c < nwb; c += blockDim.x) {
      uint8_t v = c < nb ? src[c] : 0;
      if (c == nb - 1 && (g.k[u] & 7)) v &= static_cast<uint8_t>((1u << (g.k[u] & 7)) - 1u);
      dst[c] = v;
    }
    if (threadIdx.x == 0) {
      const unsigned short h = static_cast<unsigned short>(src[nb] | (src[nb + 1] << 8));
      scales[i * ld_scales + u] = __half2float(__ushort_as_half(h));
    }
  }
}

void fill_args(PayloadArgs* g, const int* ks, int U) {
  g->U = U;
  int wo = 0, bo = 0;
  for (int u = 0; u < U; ++u) {
    g->k[u] = ks[u];
    g->woff[u] = wo;
    g->boff[u] = bo;
    wo += (ks[u] + 31) / 32;
    bo += (ks[u] + 7) / 8 + 2;
  }
}

}  // namespace

size_t payload_row_bytes(const int* ks, int U) {
  size_t b = 0;
  for (int u = 0; u < U; ++u) b += (ks[u] + 7) / 8 + 2;
  return b;
}

cudaError_t launch_payload_pack(const uint32_t* codes, int ld_codes, const float* scales, int ld_scales, int N,
                                const int* ks, int U, uint8_t* out, size_t ld_out, cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  PayloadArgs g;
  fill_args(&g, ks, U);
  k_payload_pack<<<N, 128, 0, st>>>(codes, ld_codes, scales, ld_scales, out, ld_out, g);
  return cudaGetLastError();
}

cudaError_t launch_payload_unpack(const uint8_t* in, size_t ld_in, int N, const int* ks, int U, uint32_t* codes,
                                  int ld_codes, float* scales, int ld_scales, cudaStream_t st) {
  if (N <= 0) return cudaSuccess;
  PayloadArgs g;
  fill_args(&g, ks, U);
  k_payload_unpack<<<N, 128, 0, st>>>(in, ld_in, codes, ld_codes, scales, ld_scales, g);
  return cudaGetLastError();
}
