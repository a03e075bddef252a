// Device code shared by the tensor-core scoring kernels (Sec. 3.3 Eq.
// onebit_influence; App. B.3): the kernels' argument block, the e2m1 expansion
// of stored code bits, the tile iteration, and the dequantise role, which folds
// each module's exact inner product d_u into the score in the fixed fp32 order
// acc = fl(acc + fl(fl(s_qu s_iu) d_u)) (CODES) or fl(acc + fl(s_iu d_u))
// (PAPER), module by module. k_score_tc.cu holds the one-CTA kernel (e4m3 and
// bf16 operands) and the dispatch; k_score_pair.cu the CTA-pair kernel (e2m1).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cmath>

#include "eogp_dev.cuh"
#include "eogp_internal.h"
#include "topk_dev.cuh"

namespace eogp {
namespace sc {

constexpr int kMaxMods = 1024;
constexpr int kExpWarps = 8;          // expander warps
constexpr int kDqWarp0 = kExpWarps;   // first of the four dequantise warps
constexpr int kMmaWarp = kExpWarps + 4;
constexpr int kFusedCap = kTopKBuf;   // list buffer per query column (K <= 32, 2 per lane)
constexpr int kAccLd = 132;           // row stride (floats) of a running score kept in shared memory

struct ScoreTcArgs {
  int N, Q, U, D, BNq, n_it, n_tiles, ldt, ldts, ldqs, ldo, K;
  int kuni;  // bits of every module when all modules are equal, else 0
  const uint32_t* train;
  const float* ts;
  const float* qs;
  float* out;
  float* lst;  // TOPK: per-CTA lists [gridDim.x][Q][K]
  int* lsi;
  float* bufs;  // TOPK: running list buffers [gridDim.x][BNq][kFusedCap] (global, L2-resident)
  int* bufi;
  unsigned* gtau;  // TOPK: per query, order key of the best threshold any CTA's list reached
  float* scr;      // TOPK: per-CTA scratch of one tile's scores [gridDim.x][BN][128] (L2-resident)
  unsigned* status;
  int k[kMaxMods];  // bits per module
};

// Shared-memory carve-up (byte offsets after 1024-byte alignment) of the parts
// the dequantise role uses: running score, query scales, barriers, ranking state.
struct TcSmem {
  uint32_t acc, sq, bars, lists, total;
};

// e2m1 (fp4) one-bit operands. Word c of 32 code bits -> four 32-bit columns
// of eight e2m1 values (+1 = 0x2 if the bit is set, -1 = 0xA if clear):
// column j holds bits j, j + 4, ..., j + 28 in its nibbles 0..7, so each column
// is one shift and one masked XOR. This permutes the K index within the word;
// the query operand is expanded with the same permutation (k_expand_queries_f4),
// and an inner product is unchanged by a permutation applied to both sides.
__device__ __forceinline__ uint32_t e2m1x8(uint32_t c, int j) {
  return ((c << (3 - j)) & 0x88888888u) ^ 0xAAAAAAAAu;
}

// Half a stage of one stored row (128 code bits) -> 16 TMEM columns of e2m1:
// word q of the half gives columns 4q .. 4q + 3, stored without waiting.
__device__ __forceinline__ void expand_half_tmem(uint32_t taddr, uint4 bits) {
  const uint32_t w[4] = {bits.x, bits.y, bits.z, bits.w};
  uint32_t v[16];
#pragma unroll
  for (int q = 0; q < 4; ++q)
#pragma unroll
    for (int j = 0; j < 4; ++j) v[4 * q + j] = e2m1x8(w[q], j);
  tmem_st16_issue(taddr, v);
}

// Tiles of a CTA (or of a CTA pair, which works on 256 stored rows at a time,
// each CTA on its own 128). Dense output: strided over the grid, so all CTAs
// work on the same query tile at a time. Ranking: a contiguous run of tiles, so
// a CTA ranks long runs of stored rows of one query tile (fewer fresh lists).
template <bool PAIR>
__device__ __forceinline__ int tile_unit() {
  return PAIR ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
}
template <bool PAIR>
__device__ __forceinline__ int tile_units() {
  return PAIR ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
}
template <bool TOPK, bool PAIR = false>
__device__ __forceinline__ int tile_begin(const ScoreTcArgs& g) {
  return TOPK ? static_cast<int>(static_cast<long long>(g.n_tiles) * tile_unit<PAIR>() / tile_units<PAIR>())
              : tile_unit<PAIR>();
}
template <bool TOPK, bool PAIR = false>
__device__ __forceinline__ int tile_end(const ScoreTcArgs& g) {
  return TOPK ? static_cast<int>(static_cast<long long>(g.n_tiles) * (tile_unit<PAIR>() + 1) / tile_units<PAIR>())
              : g.n_tiles;
}
template <bool TOPK, bool PAIR = false>
__device__ __forceinline__ int tile_step() {
  return TOPK ? 1 : tile_units<PAIR>();
}
// First stored row of this CTA's part of row tile ib.
template <bool PAIR>
__device__ __forceinline__ int tile_row0(int ib) {
  return PAIR ? ib * 256 + static_cast<int>(cluster_ctarank()) * 128 : ib * 128;
}

// The dequantise role (warps DQ0 .. DQ0 + NDW - 1; warp w reads TMEM
// lane quarter w % 4, TMEM lane = stored row of the CTA's tile; with eight
// warps the two of a lane quarter take half of the query columns each). Per module u of a tile: wait
// for the MMAs of d_u, fold acc = fl(acc + term(d_u)) into the running score
// (TMEM columns after the ND accumulators; with ACCS registers in a pair, else
// shared memory), release
// the accumulator; after the last module write the scores (dense) or screen and
// rank them (TOPK). In a CTA pair (PAIR) each CTA drains its own 128 rows and
// releases the accumulator on the leader CTA's barrier.
template <int MODE, bool TOPK, int BN, int ND, bool ACCS, bool PAIR, int NDW = 4, int DQ0 = kDqWarp0>
__device__ __forceinline__ void dequant_role(const ScoreTcArgs& g, uint8_t* smem, const TcSmem& L, uint32_t tmem,
                                             float* sq, uint64_t* dfull, uint64_t* dempty) {
  static_assert(NDW == 4 || NDW == 8, "four or eight dequantise warps");
  static_assert(DQ0 % 4 == 0, "warp w reads TMEM lane quarter w % 4");
  constexpr uint32_t kAcc = static_cast<uint32_t>(ND * BN);
  constexpr bool kAccS = ACCS;
  // The running score of several modules (ACCS): in registers in the pair
  // kernel, whose eight warps hold 64 columns of one row a thread (measured on
  // GPT-2 query scoring, the shared-memory running score cost more than the
  // MMAs it waits for), else in shared memory (the one-CTA kernel's four warps
  // would need 128 registers for it). Without ACCS, in the TMEM columns after
  // the accumulators, which only the one-CTA kernel's 128-query tiles have (the
  // pair kernel's other tile widths serve one module).
  constexpr bool kAccR = ACCS && PAIR && NDW == 8;
  constexpr bool kAccT = !ACCS && BN == 128 && !PAIR;
  static_assert(!kAccR || MODE == EOGP_SCORE_CODES, "the pair kernel scores one-bit queries");
  constexpr int kThr = NDW * 32;     // dequantise threads
  constexpr int CW = BN * 4 / NDW;   // query columns of a warp (all of them, or half)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q4 = warp & 3;
  const int wid = warp - DQ0;        // dequantise warp 0 .. NDW - 1
  const int ep = wid * 32 + lane;    // dequantise thread
  const int rr = q4 * 32 + lane;     // TMEM lane = stored row of the CTA's tile
  const int cbeg = (wid >> 2) * CW;  // this warp's first query column
  const int cend = min(g.BNq, cbeg + CW);
  const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
  float* lsb = g.bufs + static_cast<size_t>(blockIdx.x) * g.BNq * kFusedCap;
  int* lib = g.bufi + static_cast<size_t>(blockIdx.x) * g.BNq * kFusedCap;
  int* cntb = reinterpret_cast<int*>(smem + L.lists);
  float* taub = reinterpret_cast<float*>(cntb + BN);
  float* gtb = taub + BN;  // shared thresholds of this query tile, refreshed per tile
  uint32_t* cmask = reinterpret_cast<uint32_t*>(gtb + BN);  // [BN / 32][4] per-warp column masks
  int q0_cur = 0;
  auto list_of = [&](int col) {
    return WarpTopk{lsb + static_cast<size_t>(col) * kFusedCap, lib + static_cast<size_t>(col) * kFusedCap,
                    cntb + col, taub + col, g.K, g.gtau + q0_cur + col};
  };
  int seg_qt = -1;
  // Lists of the finished query tile to global memory; warp wid writes columns wid, wid + NDW, ...
  auto flush = [&]() {
    for (int col = wid; col < g.BNq; col += NDW) {
      const int q = seg_qt * g.BNq + col;
      if (q < g.Q) {
        const size_t off = (static_cast<size_t>(blockIdx.x) * g.Q + q) * g.K;
        topk_warp_write<2>(list_of(col), lane, g.lst + off, g.lsi + off);
      }
    }
  };
  // Last module of a tile, per chunk of 32 query columns: keep the scores in this
  // CTA's scratch (column-major) and note which columns hold a row that can
  // enter the column's list (one bit per column, per lane quarter); a column no
  // row of which beats its threshold (the usual case once the lists have
  // filled) is not offered.
  float* scr = g.scr + static_cast<size_t>(blockIdx.x) * BN * 128;
  // One 16-column half of a 32-column chunk: candidates' bits into `bits` (bit
  // c0 % 32 + j), the scores into the scratch.
  auto screen16 = [&](int c0, int q0, int row, const float (&a)[16], uint32_t& bits) {
    if (row < g.N) {
      const float4* t4 = reinterpret_cast<const float4*>(taub + c0);
      const float4* g4 = reinterpret_cast<const float4*>(gtb + c0);
#pragma unroll
      for (int j4 = 0; j4 < 4; ++j4) {
        const float4 t = t4[j4], u = g4[j4];
        const float tj[4] = {t.x, t.y, t.z, t.w}, uj[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float x = a[4 * j4 + e];
          const bool live = q0 + c0 + 4 * j4 + e < g.Q;
          if (live && x >= uj[e] && (tj[e] != tj[e] ? x == x : x > tj[e])) bits |= 1u << ((c0 & 31) + 4 * j4 + e);
        }
      }
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) scr[static_cast<size_t>(c0 + j) * 128 + rr] = a[j];
  };
  // After the D buffer is released: the flagged columns, dealt round-robin to
  // the warps, offered to their lists from the scratch.
  auto rank_tile = [&](int q0, int i0) {
    named_bar_sync(3, kThr);  // scratch and masks of every warp visible
    const int nr = min(128, g.N - i0);
    int n = 0;
    for (int c0 = 0; c0 < g.BNq; c0 += 32) {
      const uint32_t* cm = cmask + (c0 >> 5) * 4;
      uint32_t colmask = cm[0] | cm[1] | cm[2] | cm[3];
      for (; colmask; ++n) {
        const int cc = __ffs(colmask) - 1;
        colmask &= colmask - 1;
        if (n % NDW == wid)
          topk_warp_offer<2>(scr + static_cast<size_t>(c0 + cc) * 128, nr, i0, list_of(c0 + cc), lane,
                             gtb[c0 + cc]);
      }
    }
    named_bar_sync(3, kThr);  // lists settled before the next tile screens or flushes
  };
  uint32_t gm = 0;
  bool ok = true;
  for (int tile = tile_begin<TOPK, PAIR>(g), tstep = tile_step<TOPK, PAIR>(), tend = tile_end<TOPK, PAIR>(g);
       tile < tend && ok; tile += tstep) {
    const int qt = tile / g.n_it, ib = tile % g.n_it;
    const int i0 = tile_row0<PAIR>(ib), q0 = qt * g.BNq;
    const int row = i0 + rr;
    if (TOPK && qt != seg_qt) {
      if (seg_qt >= 0) {
        flush();
        named_bar_sync(3, kThr);  // every list written before any is reset
      }
      seg_qt = qt;
      q0_cur = q0;
      for (int col = ep; col < BN; col += kThr) {
        cntb[col] = 0;
        taub[col] = NAN;
      }
      named_bar_sync(3, kThr);
    }
    if (TOPK) {
      // Thresholds other CTAs' lists of these queries have reached (read before the
      // last module's ranking, after the barriers of the module loop).
      for (int col = ep; col < BN; col += kThr)
        gtb[col] = q0 + col < g.Q ? topk_unkey32(__ldcg(g.gtau + q0 + col)) : INFINITY;
    }
    // Scales: the query scales of module u go through shared memory (buffer
    // gm & 1), written after the drain of module u - 1 (at the tile's start for
    // the first module) and published by the barrier that ends it, so that
    // barrier is off the path from the MMAs' commit to the accumulator's
    // release. Buffer gm & 1 was last read in module gm - 2, which every thread
    // finished before the barrier that ended it. The scales of module u + 1
    // are loaded from global memory while module u is drained.
    constexpr int kSqPer = (BN + kThr - 1) / kThr;  // query columns of a tile per dequantise thread
    auto load_scales = [&](int u, float& si_u, float (&sq_u)[kSqPer]) {
      si_u = row < g.N ? g.ts[static_cast<size_t>(row) * g.ldts + u] : 0.f;
#pragma unroll
      for (int e = 0; e < kSqPer; ++e) {
        const int c = ep + kThr * e;
        sq_u[e] = (MODE == EOGP_SCORE_CODES && c < g.BNq && q0 + c < g.Q)
                      ? g.qs[static_cast<size_t>(q0 + c) * g.ldqs + u] : 0.f;
      }
    };
    auto store_sq = [&](uint32_t gmod, const float (&sq_u)[kSqPer]) {
      if (MODE == EOGP_SCORE_CODES) {
        float* b = sq + (gmod & 1u) * BN;
#pragma unroll
        for (int e = 0; e < kSqPer; ++e)
          if (ep + kThr * e < BN) b[ep + kThr * e] = sq_u[e];
      }
    };
    float si_next, sq_next[kSqPer];
    load_scales(0, si_next, sq_next);
    store_sq(gm, sq_next);
    float si_cur = si_next;
    if (g.U > 1) load_scales(1, si_next, sq_next);
    named_bar_sync(2, kThr);  // module 0's query scales (and TOPK thresholds) visible
    float accr[kAccR ? CW : 1];  // kAccR: this thread's running score, from +0
#pragma unroll
    for (int i = 0; i < (kAccR ? CW : 1); ++i) accr[i] = 0.f;
    for (int u = 0; u < g.U; ++u, ++gm) {
      const int buf = static_cast<int>(gm % ND);
      const uint32_t dph = (gm / ND) & 1u;
      const float si = si_cur;
      const float* sqb = sq + (gm & 1u) * BN;
      uint32_t w_ok = 1;
      if (lane == 0) w_ok = mbar_wait(&dfull[buf], dph, g.status) ? 1u : 0u;
      w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
      __syncwarp();
      tc_fence_after();
      const bool last = u + 1 == g.U;
      if (w_ok) {
      const uint32_t dcol = tmem + lane_base + buf * static_cast<uint32_t>(BN);
      const uint32_t acol = tmem + lane_base + kAcc;
      float* accrow = reinterpret_cast<float*>(smem + L.acc) + rr * kAccLd;  // kAccS: this row's running score
      auto acc_load = [&](int c0, uint32_t* ar, int n) {  // n floats from the shared running score
        for (int j = 0; j < n; j += 4) {
          const float4 v = *reinterpret_cast<const float4*>(accrow + c0 + j);
          ar[j] = __float_as_uint(v.x);
          ar[j + 1] = __float_as_uint(v.y);
          ar[j + 2] = __float_as_uint(v.z);
          ar[j + 3] = __float_as_uint(v.w);
        }
      };
      // the module's term: fl(fl(s_q s_i) d) (CODES) or fl(s_i d) (PAPER)
      auto term = [&](int c, uint32_t dv) {
        return MODE == EOGP_SCORE_CODES ? __fmul_rn(__fmul_rn(sqb[c], si), __uint_as_float(dv))
                                        : __fmul_rn(si, __uint_as_float(dv));
      };
      if constexpr (kAccR) {
        // Running score in registers (from +0: fl(0 + t) for the first
        // module); d_u 16 columns at a time (one TMEM wait a batch), the query
        // scales four at a time from shared memory.
        constexpr int RB = 16;
        uint32_t bits = 0;  // TOPK: candidates of the current 32-column chunk
#pragma unroll
        for (int b = 0; b < CW / RB; ++b) {
          const int cb = cbeg + RB * b;
          if (cb < cend) {
            uint32_t d0[RB];
            tmem_ld_issue(dcol + cb, d0);
            tmem_wait_ld(d0);
#pragma unroll
            for (int h = 0; h < RB / 16; ++h) {  // 16-column parts of the batch
              const int c0 = cb + 16 * h;
              float a[16];
#pragma unroll
              for (int j4 = 0; j4 < 4; ++j4) {
                const float4 s4 = *reinterpret_cast<const float4*>(sqb + c0 + 4 * j4);
                const float sv[4] = {s4.x, s4.y, s4.z, s4.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  const int j = 4 * j4 + e, ai = RB * b + 16 * h + j;
                  a[j] = accr[ai] =
                      __fadd_rn(accr[ai], __fmul_rn(__fmul_rn(sv[e], si), __uint_as_float(d0[16 * h + j])));
                }
              }
              if (last) {
                if (!TOPK) {
                  if (row < g.N) {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                      if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
                  }
                } else {
                  screen16(c0, q0, row, a, bits);
                  if ((c0 & 31) == 16) {  // the 32-column chunk is complete (BNq is a multiple of 32)
                    const uint32_t wbits = __reduce_or_sync(0xffffffffu, bits);
                    if (lane == 0) cmask[(c0 >> 5) * 4 + q4] = wbits;
                    bits = 0;
                  }
                }
              }
            }
          }
        }
      } else if constexpr (!kAccT) {
        // d_u in batches of 32 columns: the batch's TMEM loads are issued
        // before its one wait (tcgen05.wait::ld waits for all of the thread's
        // loads, so a load issued one 16-column chunk ahead is still waited for
        // before that chunk is done); the running score, when there is one, is
        // in shared memory.
        uint32_t bits = 0;  // TOPK: candidates of the current 32-column chunk
        for (int cb = cbeg; cb < cend; cb += 32) {
          uint32_t d0[32];
          tmem_ld32_issue(dcol + cb, d0);
          tmem_wait_ld(d0);
#pragma unroll
          for (int h = 0; h < 2; ++h) {  // 16-column halves of the batch
            const int c0 = cb + 16 * h;
            float a[16];
            if (u > 0) {
              uint32_t ar[16];
              acc_load(c0, ar, 16);
#pragma unroll
              for (int j = 0; j < 16; ++j) a[j] = __uint_as_float(ar[j]);
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) a[j] = 0.f;
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) a[j] = __fadd_rn(a[j], term(c0 + j, d0[16 * h + j]));
            if (!last) {
#pragma unroll
              for (int j = 0; j < 16; j += 4)
                *reinterpret_cast<float4*>(accrow + c0 + j) = make_float4(a[j], a[j + 1], a[j + 2], a[j + 3]);
            } else if (!TOPK) {
              if (row < g.N) {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
              }
            } else {
              screen16(c0, q0, row, a, bits);
              if (h == 1) {  // the 32-column chunk is complete (BNq is a multiple of 32)
                const uint32_t wbits = __reduce_or_sync(0xffffffffu, bits);
                if (lane == 0) cmask[(c0 >> 5) * 4 + q4] = wbits;  // a chunk's rows: the four lane quarters
                bits = 0;
              }
            }
          }
        }
      } else if (!last) {
        // Running score in TMEM (several modules, 128-query tiles of the bf16
        // kernel), 16 columns at a time: the TMEM loads of the next chunk are in
        // flight while this one is combined and stored back.
        uint32_t dr[16], ar[16];
        if (cbeg < cend) {
          tmem_ld16_issue(dcol + cbeg, dr);
          if (u > 0) tmem_ld16_issue(acol + cbeg, ar);
        }
        if (u == 0) {
#pragma unroll
          for (int j = 0; j < 16; ++j) ar[j] = 0u;
        }
#pragma unroll
        for (int ci = 0; ci < CW / 16; ++ci) {
          const int c0 = cbeg + 16 * ci;
          if (c0 < cend) {
            tmem_wait_ld(dr);
            if (u > 0) tmem_wait_ld(ar);
            uint32_t o[16];
#pragma unroll
            for (int j = 0; j < 16; ++j)
              o[j] = __float_as_uint(__fadd_rn(__uint_as_float(ar[j]), term(c0 + j, dr[j])));
            if (c0 + 16 < cend) {
              tmem_ld16_issue(dcol + c0 + 16, dr);
              if (u > 0) tmem_ld16_issue(acol + c0 + 16, ar);
            }
            tmem_st16_issue(acol + c0, o);
          }
        }
        tmem_wait_st();  // stored before the next module reads them
      } else {
        // Last module, running score in TMEM: 16 columns at a time.
        uint32_t dr[16], ar[16];
        if (cbeg < cend) {
          tmem_ld16_issue(dcol + cbeg, dr);
          if (u > 0) tmem_ld16_issue(acol + cbeg, ar);
        }
        if (u == 0) {
#pragma unroll
          for (int j = 0; j < 16; ++j) ar[j] = 0u;
        }
        uint32_t bits = 0;  // TOPK: candidates of the current 32-column chunk
#pragma unroll
        for (int ci = 0; ci < CW / 16; ++ci) {
          const int c0 = cbeg + 16 * ci;
          if (c0 < cend) {
            tmem_wait_ld(dr);
            if (u > 0) tmem_wait_ld(ar);
            float a[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) a[j] = __fadd_rn(__uint_as_float(ar[j]), term(c0 + j, dr[j]));
            if (c0 + 16 < cend) {
              tmem_ld16_issue(dcol + c0 + 16, dr);
              if (u > 0) tmem_ld16_issue(acol + c0 + 16, ar);
            }
            if (!TOPK) {
              if (row < g.N) {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                  if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
              }
            } else {
              screen16(c0, q0, row, a, bits);
              if ((c0 & 31) == 16) {
                const uint32_t wbits = __reduce_or_sync(0xffffffffu, bits);
                if (lane == 0) cmask[(c0 >> 5) * 4 + q4] = wbits;
                bits = 0;
              }
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {  // D buffer free: the MMAs run on
        if constexpr (PAIR)  // the pair's MMA issuer waits on the leader CTA's barrier
          mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(&dempty[buf]), 0));
        else
          mbar_arrive(&dempty[buf]);
      }
      }  // w_ok
      if (!last) {  // the next module's query scales into the other buffer
        store_sq(gm + 1, sq_next);
        si_cur = si_next;
        if (u + 2 < g.U) load_scales(u + 2, si_next, sq_next);
      }
      if (!named_bar_and(2, kThr, w_ok)) {  // every warp's ok; publishes the next scales
        ok = false;
        break;
      }
      if (TOPK && last) rank_tile(q0, i0);
    }
  }
  if (TOPK && seg_qt >= 0) flush();
}

// Waits with all lanes of the warp; true when every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned* status) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, status));
}

// Host side of the CTA-pair kernel (k_score_pair.cu): BN queries per tile (64,
// 128 or 256), G 256-bit stages per pipeline group (1 or 2; 4 with BN = 64),
// fused ranking or not.
size_t pair_smem_need(int BN, int G, bool topk);
// Clusters of two that can be resident at once on the current device.
int pair_cluster_cap(int num_sms);
// The two-issuer pair kernel (k_score_pair_ks.cu): one module, at most 64
// queries (one query tile), modules of a multiple of 1024 bits; tq and tc as
// for launch_pair (tc: the stored codes' map, boxes of 32 words x 128 rows).
size_t pair_ks_smem_need();
cudaError_t launch_pair_ks(const CUtensorMap& tq, const CUtensorMap& tc, const ScoreTcArgs& g, int grid,
                           cudaStream_t st);
// tq: the expanded queries' tensor map (boxes of 128 bytes x BNq / 2 rows); the
// stored codes' map is made here from g.train, g.ldt, g.D and g.N.
cudaError_t launch_pair(int BN, int G, bool topk, const CUtensorMap& tq, const ScoreTcArgs& g, int grid,
                        cudaStream_t st);

}  // namespace sc
}  // namespace eogp
