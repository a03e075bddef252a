// Per-query top-K of influence scores (App. C ranks the stored examples of
// each query by score, descending, and reads the first 20 for NDCG@20).
// Order: score descending, equal scores by lower stored index; NaN scores
// never rank; missing places are (-inf, -1).
//
// Three kernels:
// * k_topk_select ranks one row of a dense [Q, N] score matrix per block when
//   the row fits in shared memory (N <= kSelectMaxN): the K-th largest score
//   is found exactly as the largest order-preserving 32-bit key t with at
//   least K keys >= t, built bit by bit from the top (block-wide counting
//   passes over the row held in shared memory, no atomics); the K winners are
//   gathered (the equal-to-threshold ones in index order, so the lowest indices
//   win ties) and sorted.
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
constexpr int kSelectMaxN = 49152;  // rows k_topk_select holds in shared memory (192 KB)

// Order-preserving 64-bit key: larger key = larger score, then lower index
// (-0 and +0 are the same score).
__device__ __forceinline__ unsigned long long make_key(float s, int idx) {
  const uint32_t b = __float_as_uint(s == 0.f ? 0.f : s);
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

constexpr int kSelThreads = 512;
constexpr int kSelWarps = kSelThreads / 32;

// 32-bit order key of a score: larger score, larger key; -0 and +0 equal; NaN
// maps to 0, below every score (no non-NaN float maps to 0).
__device__ __forceinline__ uint32_t sel_key(float s) {
  if (s != s) return 0u;
  const uint32_t b = __float_as_uint(s == 0.f ? 0.f : s);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Number of keys of this block's row that are >= t (block-uniform result).
// red is double-buffered by `parity` so consecutive calls need one barrier.
__device__ __forceinline__ uint32_t count_ge(const uint32_t* skey, int N, uint32_t t, uint32_t* red,
                                             int parity) {
  uint32_t c = 0;
  for (int i = threadIdx.x; i < N; i += kSelThreads) c += skey[i] >= t ? 1u : 0u;
  c = __reduce_add_sync(0xffffffffu, c);
  if ((threadIdx.x & 31) == 0) red[parity * kSelWarps + (threadIdx.x >> 5)] = c;
  __syncthreads();
  uint32_t tot = 0;
#pragma unroll
  for (int w = 0; w < kSelWarps; ++w) tot += red[parity * kSelWarps + w];
  return tot;
}

__global__ void __launch_bounds__(kSelThreads) k_topk_select(const float* __restrict__ sc, int ld, int N,
                                                             int K, float* __restrict__ out_s, int ld_os,
                                                             int* __restrict__ out_i, int ld_oi) {
  extern __shared__ uint32_t skey[];  // [N] keys of this query's row
  __shared__ uint32_t red[2 * kSelWarps];
  __shared__ uint32_t weq[kSelWarps];
  __shared__ unsigned long long cand[EOGP_TOPK_MAX];
  __shared__ uint32_t s_ngt;
  const int q = blockIdx.x, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const float* row = sc + static_cast<size_t>(q) * ld;
  for (int i = tid; i < N; i += kSelThreads) skey[i] = sel_key(row[i]);
  if (tid == 0) s_ngt = 0;
  __syncthreads();
  // Valid (non-NaN) scores are the keys >= 1.
  int parity = 0;
  const uint32_t nv = count_ge(skey, N, 1u, red, parity);
  parity ^= 1;
  const int Kv = static_cast<int>(min(static_cast<uint32_t>(K), nv));
  if (Kv > 0) {
    // T = the Kv-th largest key: the largest t with at least Kv keys >= t, built
    // bit by bit from the top.
    uint32_t T = 0;
    for (int bit = 31; bit >= 0; --bit) {
      const uint32_t c = T | (1u << bit);
      if (count_ge(skey, N, c, red, parity) >= static_cast<uint32_t>(Kv)) T = c;
      parity ^= 1;
    }
    const uint32_t ngt = T == 0xFFFFFFFFu ? 0u : count_ge(skey, N, T + 1u, red, parity);
    parity ^= 1;
    const uint32_t rem = static_cast<uint32_t>(Kv) - ngt;  // keys equal to T that rank, >= 1
    // Gather. Keys above T (ngt of them) in any order; keys equal to T in index
    // order, so that the rem lowest indices win: warp w scans the contiguous
    // segment [w seg, (w+1) seg) twice (count, then place).
    const int seg = ((N + kSelWarps - 1) / kSelWarps + 31) & ~31;
    const int b0 = warp * seg, b1 = min(N, b0 + seg);
    uint32_t mine = 0;
    for (int base = b0; base < b1; base += 32) {
      const int i = base + lane;
      mine += __popc(__ballot_sync(0xffffffffu, i < b1 && skey[i] == T));
    }
    if (lane == 0) weq[warp] = mine;
    __syncthreads();
    uint32_t before = 0;
    for (int w = 0; w < warp; ++w) before += weq[w];
    for (int base = b0; base < b1; base += 32) {
      const int i = base + lane;
      const uint32_t k = i < b1 ? skey[i] : 0u;
      const unsigned long long ck =
          (static_cast<unsigned long long>(k) << 32) | (0xFFFFFFFFu - static_cast<uint32_t>(i));
      if (k > T) cand[atomicAdd(&s_ngt, 1u)] = ck;
      const unsigned b = __ballot_sync(0xffffffffu, i < b1 && k == T);
      const uint32_t pos = before + static_cast<uint32_t>(__popc(b & ((1u << lane) - 1u)));
      if (((b >> lane) & 1u) && pos < rem) cand[ngt + pos] = ck;
      before += static_cast<uint32_t>(__popc(b));
    }
    __syncthreads();
    // Sort the Kv winners: descending key = score descending, then lower index.
    int P = 1;
    while (P < Kv) P <<= 1;
    for (int i = Kv + tid; i < P; i += kSelThreads) cand[i] = 0ull;
    __syncthreads();
    for (int k2 = 2; k2 <= P; k2 <<= 1) {
      for (int j = k2 >> 1; j > 0; j >>= 1) {
        for (int i = tid; i < P; i += kSelThreads) {
          const int ixj = i ^ j;
          if (ixj > i) {
            const unsigned long long a = cand[i], b2 = cand[ixj];
            const bool desc = (i & k2) == 0;
            if (desc ? (a < b2) : (a > b2)) {
              cand[i] = b2;
              cand[ixj] = a;
            }
          }
        }
        __syncthreads();
      }
    }
  }
  for (int p = tid; p < K; p += kSelThreads) {
    float v = -INFINITY;
    int ix = -1;
    if (p < Kv) {
      ix = static_cast<int>(0xFFFFFFFFu - static_cast<uint32_t>(cand[p]));
      v = row[ix];  // the stored score itself (keys merge -0 into +0)
    }
    out_s[static_cast<size_t>(q) * ld_os + p] = v;
    out_i[static_cast<size_t>(q) * ld_oi + p] = ix;
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

int topk_select_max_n() { return kSelectMaxN; }

cudaError_t launch_topk_select(const float* scores, int ld, int Q, int N, int K, float* out_s, int ld_os,
                               int* out_i, int ld_oi, cudaStream_t st) {
  if (Q <= 0) return cudaSuccess;
  if (N > kSelectMaxN || K > EOGP_TOPK_MAX) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(std::max(N, 1)) * 4;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(k_topk_select, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(smem));
    if (e != cudaSuccess) return e;
  }
  k_topk_select<<<Q, kSelThreads, smem, st>>>(scores, ld, N, K, out_s, ld_os, out_i, ld_oi);
  return cudaGetLastError();
}

cudaError_t launch_topk_merge(const float* lst, const int* lsi, int S, int Q, int K, float* out_s,
                              int ld_os, int* out_i, int ld_oi, cudaStream_t st) {
  if (Q <= 0) return cudaSuccess;
  k_topk_merge<<<Q, 256, 0, st>>>(lst, lsi, S, Q, K, out_s, ld_os, out_i, ld_oi);
  return cudaGetLastError();
}
