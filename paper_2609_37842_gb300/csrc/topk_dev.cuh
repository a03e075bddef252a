// Per-query running top-K list kept by one thread (device helpers shared by the
// fused scoring epilogue and the dense ranking kernel).
//
// The list holds up to K (score, stored index) pairs in shared memory, unsorted,
// with the weakest entry tracked: once full, a new score replaces the weakest
// only if it is strictly larger (rows arrive in increasing index, so an equal
// score never displaces an earlier row). Order is established once, when the
// list is written out: score descending, equal scores by lower index.
#pragma once

#include <cmath>

namespace eogp {

struct TopkState {
  int cnt;    // entries held
  int wpos;   // position of the weakest entry (valid when cnt == K)
  float tau;  // its score; -inf while the list is not full
};

__device__ __forceinline__ void topk_reset(TopkState& t) {
  t.cnt = 0;
  t.wpos = 0;
  t.tau = -INFINITY;
}

// Weakest entry: lowest score, among equal scores the highest index.
__device__ __forceinline__ void topk_find_weakest(const float* ls, const int* li, int K, TopkState& t) {
  float ws = ls[0];
  int wi = li[0], wp = 0;
  for (int p = 1; p < K; ++p) {
    const float s = ls[p];
    const int i = li[p];
    if (s < ws || (s == ws && i > wi)) {
      ws = s;
      wi = i;
      wp = p;
    }
  }
  t.wpos = wp;
  t.tau = ws;
}

__device__ __forceinline__ void topk_offer(float v, int idx, float* ls, int* li, int K, TopkState& t) {
  if (t.cnt < K) {
    if (v == v) {  // NaN never ranks
      ls[t.cnt] = v;
      li[t.cnt] = idx;
      if (++t.cnt == K) topk_find_weakest(ls, li, K, t);
    }
  } else if (v > t.tau) {
    ls[t.wpos] = v;
    li[t.wpos] = idx;
    topk_find_weakest(ls, li, K, t);
  }
}

// Offers col[0..nr) with stored indices base + r; loads four rows ahead of the tests.
__device__ __forceinline__ void topk_scan(const float* col, int nr, int base, float* ls, int* li, int K,
                                          TopkState& t) {
  int r = 0;
  for (; r + 4 <= nr; r += 4) {
    const float v0 = col[r], v1 = col[r + 1], v2 = col[r + 2], v3 = col[r + 3];
    if (t.cnt < K || v0 > t.tau || v1 > t.tau || v2 > t.tau || v3 > t.tau) {
      topk_offer(v0, base + r, ls, li, K, t);
      topk_offer(v1, base + r + 1, ls, li, K, t);
      topk_offer(v2, base + r + 2, ls, li, K, t);
      topk_offer(v3, base + r + 3, ls, li, K, t);
    }
  }
  for (; r < nr; ++r) topk_offer(col[r], base + r, ls, li, K, t);
}

// Sorts the held entries (score descending, equal scores by lower index) and
// writes K places to global memory, (-inf, -1) past the held ones.
__device__ __forceinline__ void topk_write(float* ls, int* li, int K, const TopkState& t, float* gs, int* gi) {
  for (int a = 1; a < t.cnt; ++a) {  // insertion sort, once per list
    const float s = ls[a];
    const int i = li[a];
    int b = a;
    while (b > 0 && (ls[b - 1] < s || (ls[b - 1] == s && li[b - 1] > i))) {
      ls[b] = ls[b - 1];
      li[b] = li[b - 1];
      --b;
    }
    ls[b] = s;
    li[b] = i;
  }
  for (int p = 0; p < K; ++p) {
    gs[p] = p < t.cnt ? ls[p] : -INFINITY;
    gi[p] = p < t.cnt ? li[p] : -1;
  }
}

}  // namespace eogp
