// Running per-query top-K lists, kept by one warp per query column (device
// helpers shared by the fused scoring epilogue and the dense ranking kernel).
//
// A column's list is a buffer of 32 E (score, stored index) entries in shared
// memory, its fill count and a threshold tau. Candidates (scores above tau) are
// appended a ballot at a time; when a batch would not fit, the buffer is
// pruned: sorted in registers across the warp (bitonic, E entries per lane) and
// cut to its best K, tau becoming the K-th best score (until then every non-NaN
// score is a candidate). Order is score descending, equal scores by lower index
// (rows arrive in increasing index, so a score equal to tau never belongs to the
// list once it is full). NaN scores never enter. K <= 32 (E - 1).
#pragma once

#include <climits>
#include <cmath>

namespace eogp {

// Entries per lane of a list that must hold K: the buffer takes K plus one ballot.
__host__ __device__ constexpr int topk_entries_per_lane(int K) {
  return K <= 32 ? 2 : K <= 96 ? 4 : K <= 224 ? 8 : 16;
}

struct WarpTopk {
  float* ls;   // [32 E] scores
  int* li;     // [32 E] stored indices
  int* cnt;    // entries held
  float* tau;  // NaN until a prune leaves K entries, then the K-th best score
  int K;
  unsigned* shared_tau;  // or null: order key of the best threshold any list of this query reached
};

// Order-preserving 32-bit key of a score (larger score, larger key; 0 = none).
__device__ __forceinline__ unsigned topk_key32(float s) {
  const unsigned b = __float_as_uint(s);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float topk_unkey32(unsigned k) {
  if (k == 0u) return -INFINITY;
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// a ranks before b: higher score, or equal score and lower index
__device__ __forceinline__ bool topk_before(float sa, int ia, float sb, int ib) {
  return sa > sb || (sa == sb && ia < ib);
}

// Sorts the held entries into rank order in registers: lane holds positions
// lane + 32 j, j < E; empty places are (-inf, INT_MAX), after every real entry.
template <int E>
__device__ __forceinline__ void topk_sorted(const WarpTopk& w, int lane, float (&s)[E], int (&ix)[E]) {
  const int cnt = *w.cnt;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const int p = lane + 32 * j;
    s[j] = p < cnt ? w.ls[p] : -INFINITY;
    ix[j] = p < cnt ? w.li[p] : INT_MAX;
  }
  // bitonic sort of 32 E elements, element e = 32 j + lane, rank order ascending in e
#pragma unroll
  for (int k2 = 2; k2 <= 32 * E; k2 <<= 1) {
#pragma unroll
    for (int d = k2 >> 1; d > 0; d >>= 1) {
      if (d >= 32) {
        const int dj = d >> 5;  // partner in the same lane, register j ^ dj
#pragma unroll
        for (int j = 0; j < E; ++j) {
          if (j & dj) continue;
          const int jj = j | dj;
          const bool up = ((32 * j + lane) & k2) == 0;
          const bool sw = up ? topk_before(s[jj], ix[jj], s[j], ix[j]) : topk_before(s[j], ix[j], s[jj], ix[jj]);
          if (sw) {
            const float ts = s[j];
            const int ti = ix[j];
            s[j] = s[jj];
            ix[j] = ix[jj];
            s[jj] = ts;
            ix[jj] = ti;
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < E; ++j) {
          const int e = 32 * j + lane;
          const float os = __shfl_xor_sync(0xffffffffu, s[j], d);
          const int oi = __shfl_xor_sync(0xffffffffu, ix[j], d);
          const bool lower = (e & d) == 0;  // this element is the lower of the pair
          const bool up = (e & k2) == 0;    // block sorted into rank order (else reversed)
          // the lower element of an "up" pair keeps the earlier-ranked value, and so on
          const bool take = (lower == up) ? topk_before(os, oi, s[j], ix[j]) : topk_before(s[j], ix[j], os, oi);
          if (take) {
            s[j] = os;
            ix[j] = oi;
          }
        }
      }
    }
  }
}

// Cuts the buffer to its best K entries and sets tau.
template <int E>
__device__ __forceinline__ void topk_prune(const WarpTopk& w, int lane) {
  float s[E];
  int ix[E];
  topk_sorted<E>(w, lane, s, ix);
  const int cnt = *w.cnt;
  const int keep = cnt < w.K ? cnt : w.K;
  __syncwarp();
  float kv = 0.f;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const int p = lane + 32 * j;
    if (p < keep) {
      w.ls[p] = s[j];
      w.li[p] = ix[j];
    }
    if (j == ((w.K - 1) >> 5)) kv = s[j];
  }
  const float kth = __shfl_sync(0xffffffffu, kv, (w.K - 1) & 31);
  __syncwarp();
  if (lane == 0) {
    *w.cnt = keep;
    *w.tau = keep == w.K ? kth : NAN;
    // Another list of the same query may skip scores below this one: this list
    // alone holds K stored rows scoring at least kth.
    if (keep == w.K && w.shared_tau) atomicMax(w.shared_tau, topk_key32(kth));
  }
  __syncwarp();
}

__device__ __forceinline__ void topk_warp_reset(const WarpTopk& w, int lane) {
  if (lane == 0) {
    *w.cnt = 0;
    *w.tau = NAN;
  }
  __syncwarp();
}

// Offers the nr (<= 128) staged scores col[0..nr) of one query column, stored
// indices base + r. Scores below tg (a threshold some list of this query has
// reached: the final K-th best is at least tg) are skipped. The whole warp calls
// this with the same column.
template <int E>
__device__ __forceinline__ void topk_warp_offer(const float* col, int nr, int base, const WarpTopk& w, int lane,
                                                float tg = -INFINITY) {
  float v[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = lane + 32 * i;
    v[i] = r < nr ? col[r] : NAN;
  }
  float tau = *w.tau;
  // candidate: above tau, or any non-NaN score while tau is NaN (not yet full)
  auto cand = [&](float x) { return x >= tg && (tau != tau ? x == x : x > tau); };
  bool any = false;
#pragma unroll
  for (int i = 0; i < 4; ++i) any |= cand(v[i]);
  if (!__any_sync(0xffffffffu, any)) return;  // the common case once the list has filled
  int cnt = *w.cnt;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    unsigned m = __ballot_sync(0xffffffffu, cand(v[i]));
    if (!m) continue;
    if (cnt + __popc(m) > 32 * E) {
      __syncwarp();
      if (lane == 0) *w.cnt = cnt;
      __syncwarp();
      topk_prune<E>(w, lane);
      cnt = *w.cnt;
      tau = *w.tau;
      m = __ballot_sync(0xffffffffu, cand(v[i]));
    }
    if (cand(v[i])) {
      const int pos = cnt + __popc(m & ((1u << lane) - 1u));
      w.ls[pos] = v[i];
      w.li[pos] = base + lane + 32 * i;
    }
    cnt += __popc(m);
  }
  __syncwarp();
  if (lane == 0) *w.cnt = cnt;
  __syncwarp();
}

// Writes the K places of a list to global memory in rank order; (-inf, -1)
// past the held entries.
template <int E>
__device__ __forceinline__ void topk_warp_write(const WarpTopk& w, int lane, float* gs, int* gi) {
  float s[E];
  int ix[E];
  topk_sorted<E>(w, lane, s, ix);
  const int cnt = *w.cnt;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const int p = lane + 32 * j;
    if (p < w.K) {
      gs[p] = p < cnt ? s[j] : -INFINITY;
      gi[p] = p < cnt ? ix[j] : -1;
    }
  }
  __syncwarp();
}

}  // namespace eogp
