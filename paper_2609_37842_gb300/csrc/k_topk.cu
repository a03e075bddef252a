// Per-query top-K of influence scores (App. C ranks the stored examples of
// each query by score, descending, and reads the first 20 for NDCG@20).
// Order: score descending, equal scores by lower stored index; NaN scores
// never rank; missing places are (-inf, -1).
//
// Two kernels:
// * k_topk_dense ranks a dense [Q, N] score matrix: block (slot s, query tile)
//   owns stored rows [s R, (s+1) R) of 32 queries; 128-row chunks are staged
//   transposed in shared memory and the warp offers each query's column to
//   that query's list.
// * k_topk_merge merges per-slot lists [S][Q][K] (written by k_topk_dense or by
//   the fused tensor-core scoring epilogue) into the final [Q, K]. Every slot
//   list is sorted, so the largest K-th entry over the slots is a lower bound
//   on the final K-th entry; only candidates at or above it are sorted.
#include <algorithm>
#include <cmath>

#include "eogp_internal.h"
#include "topk_dev.cuh"

namespace {

constexpr int kChunk = 128;
constexpr int kTs = kChunk + 1;  // staged row stride (floats)
constexpr int kMaxSlots = 512;
constexpr int kMergeCap = 4096;  // keys sorted at once by the merge

// Order-preserving 64-bit key: larger key = larger score, then lower index.
__device__ __forceinline__ unsigned long long make_key(float s, int idx) {
  const uint32_t b = __float_as_uint(s);
  const uint32_t o = (b & 0x80000000u) ? ~b : (b | 0x80000000u);
  return (static_cast<unsigned long long>(o) << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(idx));
}

__device__ __forceinline__ float key_score(unsigned long long key) {
  const uint32_t o = static_cast<uint32_t>(key >> 32);
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

__device__ __forceinline__ int key_index(unsigned long long key) {
  return static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(key));
}

template <int E>
__global__ void __launch_bounds__(32) k_topk_dense(const float* __restrict__ sc, int ld, int Q, int N,
                                                   int K, int rows_per_slot, float* __restrict__ lst,
                                                   int* __restrict__ lsi) {
  constexpr int kCap = 32 * E;
  extern __shared__ float sm[];
  float* tb = sm;                                     // [32 queries][kTs]
  float* ls = sm + 32 * kTs;                          // [32][kCap]
  int* li = reinterpret_cast<int*>(ls + 32 * kCap);   // [32][kCap]
  int* cnt = li + 32 * kCap;                          // [32]
  float* tau = reinterpret_cast<float*>(cnt + 32);    // [32]
  const int lane = threadIdx.x;
  const int slot = blockIdx.x, q0 = blockIdx.y * 32;
  const int nq = min(32, Q - q0);
  const int r_beg = slot * rows_per_slot, r_end = min(N, r_beg + rows_per_slot);
  const bool vec = (ld & 3) == 0 && (reinterpret_cast<uintptr_t>(sc) & 15) == 0;
  auto list_of = [&](int j) {
    return eogp::WarpTopk{ls + static_cast<size_t>(j) * kCap, li + static_cast<size_t>(j) * kCap, cnt + j, tau + j,
                          K, nullptr};
  };
  for (int j = 0; j < nq; ++j) eogp::topk_warp_reset(list_of(j), lane);
  for (int r0 = r_beg; r0 < r_end; r0 += kChunk) {
    const int nr = min(kChunk, r_end - r0);
    for (int j = 0; j < nq; ++j) {
      const float* src = sc + static_cast<size_t>(q0 + j) * ld + r0;
      if (vec && nr == kChunk) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(src) + lane);
        float* d = tb + j * kTs + 4 * lane;
        d[0] = v.x;
        d[1] = v.y;
        d[2] = v.z;
        d[3] = v.w;
      } else {
        for (int c = lane; c < nr; c += 32) tb[j * kTs + c] = src[c];
      }
    }
    __syncwarp();
    for (int j = 0; j < nq; ++j) eogp::topk_warp_offer<E>(tb + j * kTs, nr, r0, list_of(j), lane);
    __syncwarp();
  }
  for (int j = 0; j < nq; ++j) {
    const size_t o = (static_cast<size_t>(slot) * Q + q0 + j) * K;
    eogp::topk_warp_write<E>(list_of(j), lane, lst + o, lsi + o);
  }
}

__global__ void __launch_bounds__(256) k_topk_merge(const float* __restrict__ lst,
                                                    const int* __restrict__ lsi, int S, int Q, int K,
                                                    float* __restrict__ out_s, int ld_os,
                                                    int* __restrict__ out_i, int ld_oi) {
  __shared__ unsigned long long keys[kMergeCap];
  __shared__ unsigned long long red[8];
  __shared__ int fill;
  const int q = blockIdx.x, tid = threadIdx.x;
  // Lower bound: the largest K-th entry over the slots.
  unsigned long long lb = 0;
  for (int s = tid; s < S; s += blockDim.x) {
    const size_t o = (static_cast<size_t>(s) * Q + q) * K + (K - 1);
    const int ix = lsi[o];
    if (ix >= 0) lb = max(lb, make_key(lst[o], ix));
  }
  for (int off = 16; off > 0; off >>= 1) lb = max(lb, __shfl_xor_sync(0xffffffffu, lb, off));
  if ((tid & 31) == 0) red[tid >> 5] = lb;
  for (int i = tid; i < K; i += blockDim.x) keys[i] = 0;  // kept best K (0 = empty)
  __syncthreads();
  lb = red[0];
  for (int w = 1; w < (blockDim.x >> 5); ++w) lb = max(lb, red[w]);
  const long long C = static_cast<long long>(S) * K;
  const int W = kMergeCap - K;
  for (long long base = 0; base < C; base += W) {
    if (tid == 0) fill = 0;
    __syncthreads();
    const long long end = min(C, base + W);
    for (long long c = base + tid; c < end; c += blockDim.x) {
      const int s = static_cast<int>(c / K), p = static_cast<int>(c % K);
      const size_t o = (static_cast<size_t>(s) * Q + q) * K + p;
      const int ix = lsi[o];
      if (ix >= 0) {
        const unsigned long long key = make_key(lst[o], ix);
        if (key >= lb) keys[K + atomicAdd(&fill, 1)] = key;
      }
    }
    __syncthreads();
    const int n = K + fill;
    if (fill > 0) {
      int P = 2;
      while (P < n) P <<= 1;
      for (int i = n + tid; i < P; i += blockDim.x) keys[i] = 0;
      __syncthreads();
      // bitonic sort, descending
      for (int k2 = 2; k2 <= P; k2 <<= 1) {
        for (int j = k2 >> 1; j > 0; j >>= 1) {
          for (int i = tid; i < P; i += blockDim.x) {
            const int ixj = i ^ j;
            if (ixj > i) {
              const unsigned long long a = keys[i], b = keys[ixj];
              const bool desc = (i & k2) == 0;
              if (desc ? (a < b) : (a > b)) {
                keys[i] = b;
                keys[ixj] = a;
              }
            }
          }
          __syncthreads();
        }
      }
    }
    __syncthreads();
  }
  for (int p = tid; p < K; p += blockDim.x) {
    const unsigned long long key = keys[p];
    out_s[static_cast<size_t>(q) * ld_os + p] = key ? key_score(key) : -INFINITY;
    out_i[static_cast<size_t>(q) * ld_oi + p] = key ? key_index(key) : -1;
  }
}

int rows_per_slot(int N) {
  const int nch = (N + kChunk - 1) / kChunk;
  const int per = (nch + kMaxSlots - 1) / kMaxSlots;
  return std::max(1, per) * kChunk;
}

}  // namespace

int topk_dense_slots(int N) {
  const int R = rows_per_slot(N);
  return std::max(1, (N + R - 1) / R);
}

template <int E>
cudaError_t launch_topk_dense_e(const float* scores, int ld, int Q, int N, int K, float* lst, int* lsi,
                                cudaStream_t st) {
  const int S = topk_dense_slots(N);
  const size_t smem = (32 * kTs + 32 * static_cast<size_t>(32 * E) * 2 + 64) * 4;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(k_topk_dense<E>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  dim3 grid(S, (Q + 31) / 32);
  k_topk_dense<E><<<grid, 32, smem, st>>>(scores, ld, Q, N, K, rows_per_slot(N), lst, lsi);
  return cudaGetLastError();
}

cudaError_t launch_topk_dense(const float* scores, int ld, int Q, int N, int K, float* lst, int* lsi,
                              cudaStream_t st) {
  if (Q <= 0) return cudaSuccess;
  switch (eogp::topk_entries_per_lane(K)) {
    case 2: return launch_topk_dense_e<2>(scores, ld, Q, N, K, lst, lsi, st);
    case 4: return launch_topk_dense_e<4>(scores, ld, Q, N, K, lst, lsi, st);
    case 8: return launch_topk_dense_e<8>(scores, ld, Q, N, K, lst, lsi, st);
    default: return launch_topk_dense_e<16>(scores, ld, Q, N, K, lst, lsi, st);
  }
}

cudaError_t launch_topk_merge(const float* lst, const int* lsi, int S, int Q, int K, float* out_s,
                              int ld_os, int* out_i, int ld_oi, cudaStream_t st) {
  if (Q <= 0) return cudaSuccess;
  k_topk_merge<<<Q, 256, 0, st>>>(lst, lsi, S, Q, K, out_s, ld_os, out_i, ld_oi);
  return cudaGetLastError();
}
