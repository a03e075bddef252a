// Scoring on the tensor cores (Sec. 3.3 Eq. onebit_influence; App. B.3 scan),
// in two modes and with two outputs.
//
// CODES: both sides one-bit. For module u the +-1 inner product d_u = <b_q, b_i>
//   is an integer with |d_u| <= k_u. Both sides are expanded to +-1 and
//   multiplied on the tensor cores into fp32 TMEM: as e2m1 values (+1 = 0x2,
//   -1 = 0xA) with tcgen05.mma kind::mxf4 and every block scale 1 when each
//   module is a multiple of 256 bits (twice the e4m3 rate), else as e4m3 bytes
//   (+1 = 0x38, -1 = 0xB8) with kind::f8f6f4. Both encodings are exact and
//   every partial sum is an integer far below 2^24, so d_u is exact. The epilogue dequantises in the same fixed fp32 order as the
//   popcount kernels, acc = fl(acc + fl(fl(s_qu * s_iu) * d_u)) in module order,
//   keeping acc in TMEM between modules, so scores are bitwise identical to the
//   popcount path and to the oracle's float32 evaluation.
// PAPER: the query stays unquantised (the paper's asymmetric score
//   sum_u s_iu <y_u, b_iu>). y is split into bf16 hi + lo (y - hi rounded again),
//   stored bits are expanded to bf16 +-1, and two kind::f16 MMAs (hi, lo) add
//   into one fp32 accumulator per module: products are exact, the split keeps
//   y to about 2^-17 relative, and the MMA sums in fp32. The epilogue forms
//   acc = fl(acc + fl(s_iu * d_u)) in module order.
//
// Output: either the dense [Q, N] score matrix, or (TOPK) only each query's K
// best stored rows. In the TOPK epilogue the last module's scores of a tile
// are compared, 32 query columns at a time, with each column's threshold;
// chunks holding a candidate are staged in shared memory and a warp per column
// appends the candidates to that query's list (topk_dev.cuh). A CTA's lists
// cover the stored rows of its tiles and are written out when the CTA moves to
// the next query tile; a separate kernel merges the per-CTA lists. The Q x N
// matrix never reaches HBM.
//
// Tiles: 128 stored rows (MMA M, operand A) x BNq queries (MMA N, operand B),
// BNq <= 256 for CODES with one module, else <= 128. Queries are prepared
// once per call in the workspace (e2m1 pairs or e4m3 bytes, or bf16 hi and lo
// rows) and fetched by TMA; stored rows are expanded from their bits by eight
// warps into tensor memory (CODES) or into 128-byte swizzled shared-memory rows
// (PAPER), so the store is read from HBM as bits. Dense output runs tiles query-tile-major: one query tile stays in L2
// while the stored codes stream past it.
//
// Warps: 0-7 expand stored rows, two threads per row (warp 0 lane 0 also
// issues the query TMA), 8-11 dequantise (TMEM lane quarters 0-3; in TOPK
// the four warps share the ranking), 12 owns TMEM and issues the MMAs. TMEM:
// with 128 queries per tile, three 128-column d_u buffers (modules u+1 and
// u+2 accumulate while module u is dequantised) and a 128-column running
// score; with 256, two 256-column buffers and no running score.
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <type_traits>
#include <cmath>
#include <cstdlib>

#include "eogp_dev.cuh"
#include "eogp_internal.h"
#include "topk_dev.cuh"

using namespace eogp;

namespace {

constexpr int kMaxMods = 1024;
constexpr int kExpWarps = 8;                        // expander warps (two per stored row)
constexpr int kThreadsTc = (kExpWarps + 4 + 1) * 32;  // + 4 dequantise warps + 1 MMA warp
constexpr int kDqWarp0 = kExpWarps;                 // first dequantise warp
constexpr int kMmaWarp = kExpWarps + 4;
constexpr uint32_t kAB = 16384u;                    // 128 rows x 128 bytes
constexpr int kFusedCap = kTopKBuf;                 // list buffer per query column (K <= 32, 2 per lane)

struct ScoreTcArgs {
  int N, Q, U, D, BNq, n_it, n_tiles, ldt, ldts, ldqs, ldo, K;
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

template <int MODE>
struct TcMode;
template <>
struct TcMode<EOGP_SCORE_CODES> {
  static constexpr int kBits = 128;  // code bits per pipeline stage
  static constexpr int kQBoxes = 1;  // query operand tiles per stage
  using HalfBits = uint2;            // one stage of half a stored row
};
template <>
struct TcMode<EOGP_SCORE_PAPER> {
  static constexpr int kBits = 64;
  static constexpr int kQBoxes = 2;  // hi, lo
  using HalfBits = uint32_t;
};

// BN: queries per tile (MMA N). 256 only for CODES with one module (no running
// score is needed, so the two accumulators take all 512 TMEM columns).
// AT: the expanded stored rows (operand A) go to tensor memory instead of
// shared memory (CODES): a pipeline stage is then only the query operand in
// shared memory plus a 32-column A slot in TMEM, and the tensor cores read A
// from TMEM (tcgen05.mma with [a-tmem]), taking the A writes and reads off the
// shared-memory bandwidth the query operand's TMA writes and MMA reads use.
template <int MODE, int BN, bool AT>
constexpr uint32_t tc_stage_bytes() {
  return (AT ? 0u : kAB) + static_cast<uint32_t>(BN) * 128u * TcMode<MODE>::kQBoxes;
}
template <bool AT>
constexpr uint32_t tc_b_offset() {
  return AT ? 0u : kAB;
}

// Pipeline stages. Shared-memory A: six when a stage is 32 KB (one-bit
// queries, 128 per tile), else four (48 KB stages). TMEM A: six 32 KB query
// stages with 256 queries per tile (A slots in TMEM columns 256-447), four with
// 128 (A slots in columns 384-511).
template <int MODE, bool TOPK, int BN, bool AT, bool F4 = false>
constexpr int tc_stages() {
  return AT ? (BN == 256 ? 6 : (F4 ? 7 : 8)) : ((MODE == EOGP_SCORE_CODES && BN == 128) ? 6 : 4);
}

// 128-query tiles with operand A in TMEM keep the running score in shared
// memory (row stride kAccLd floats: conflict-free float4 rows), leaving 256
// TMEM columns for eight A slots next to the two d_u accumulators.
template <int BN, bool AT>
constexpr bool tc_acc_smem() {
  return AT && BN == 128;
}
constexpr int kAccLd = 132;

// Stages the expanders fill per synchronisation round (one wait, fence and
// arrive round): two with six stages, so that the MMAs always have at least
// four stages to work on, else one.
template <int MODE, bool TOPK, int BN, bool AT, bool F4 = false>
constexpr int tc_group() {
  return tc_stages<MODE, TOPK, BN, AT, F4>() >= 6 ? 2 : 1;
}

// Accumulator buffers d_u in TMEM (BN columns each). Shared-memory A: three of
// 128 columns plus the 128-column running score, or two of 256 (one module, no
// running score). TMEM A: two of 128 plus the running score, or one of 256.
template <int BN, bool AT>
constexpr int tc_dbufs() {
  return AT ? (BN == 128 ? 2 : 1) : (BN == 128 ? 3 : 2);
}
constexpr int kMaxDbufs = 3;

// First TMEM column of A slot s (TMEM A), after the accumulators (one of 256
// columns, or two of 128).
template <int BN>
__device__ __forceinline__ uint32_t tc_acol(int s) {
  return static_cast<uint32_t>(256 + 32 * s);
}

// e2m1 path: the unit scale factors (ue8m0 0x7F = 1.0) of operands A and B,
// 16 TMEM columns each, after the S A slots (columns 448-479 with 256 queries
// per tile and six slots, 480-511 with 128 and seven).
template <int S>
constexpr uint32_t tc_sf_col() {
  return static_cast<uint32_t>(256 + 32 * S);
}

// Shared-memory carve-up (byte offsets after 1024-byte alignment).
struct TcSmem {
  uint32_t acc, sq, bars, lists, total;
};
template <int MODE, bool TOPK, int BN, bool AT, bool F4 = false>
__host__ __device__ inline TcSmem tc_smem_layout(int BNq, int K) {
  constexpr int S = tc_stages<MODE, TOPK, BN, AT, F4>();
  TcSmem l;
  l.acc = S * tc_stage_bytes<MODE, BN, AT>();
  l.sq = l.acc + (tc_acc_smem<BN, AT>() ? 128u * kAccLd * 4u : 0u);
  l.bars = l.sq + 2 * BN * 4;  // query scales, double-buffered by module
  l.lists = l.bars + (2 * S + 2 * kMaxDbufs) * 8 + 16;
  // per-column held count, own threshold and shared threshold (the list buffers
  // themselves are in global memory)
  l.total = l.lists + (TOPK ? BN * 12 + 8 * 4 * 4 : 0);
  return l;
}

// 4 code bits -> 4 e4m3 bytes (bit j -> byte j: +1 = 0x38 if set, -1 = 0xB8 if
// clear): the multiply places bit j at bit 8j + 7 (the four shifted copies of
// the nibble never overlap, so there are no carries).
__device__ __forceinline__ uint32_t e4m3x4(uint32_t nib) {
  return ((nib * 0x10204080u) & 0x80808080u) ^ 0xB8B8B8B8u;
}

// 8 code bits -> 8 e4m3 bytes (query expansion).
__device__ __forceinline__ uint64_t expand8(uint32_t v) {
  return static_cast<uint64_t>(e4m3x4(v & 0xFu)) | (static_cast<uint64_t>(e4m3x4((v >> 4) & 0xFu)) << 32);
}

// 4 code bits -> 4 bf16 values (bit j -> element j: +1 = 0x3F80 if set, -1 = 0xBF80 if
// clear). Each 16-bit lane isolates its bit at position j, then adding 0x8000 - 2^j
// carries into bit 15 exactly when the bit is set.
__device__ __forceinline__ uint64_t expand4_bf16(uint32_t v) {
  uint64_t x = (static_cast<uint64_t>(v & 0xFu) * 0x0001000100010001ull) & 0x0008000400020001ull;
  x = (x + 0x7FF87FFC7FFE7FFFull) & 0x8000800080008000ull;
  return 0xBF80BF80BF80BF80ull ^ x;
}

// Half a stage of one stored row -> 4 of its 8 swizzled 16-byte chunks
// (chunk c goes to position c ^ (row & 7)); `half` selects chunks 4 half .. +3.
__device__ __forceinline__ void expand_half(uint8_t* row, int sw, int half, uint32_t bits) {  // 32 bits -> bf16
#pragma unroll
  for (int cc = 0; cc < 4; ++cc) {
    const uint32_t h = bits >> (cc * 8);
    const uint64_t lo = expand4_bf16(h), hi = expand4_bf16(h >> 4);
    *reinterpret_cast<uint4*>(row + (((4 * half + cc) ^ sw) << 4)) =
        make_uint4(static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32), static_cast<uint32_t>(hi),
                   static_cast<uint32_t>(hi >> 32));
  }
}

// Half a stage of one stored row -> 16 TMEM columns of e4m3 (column n holds
// elements 4n..4n+3 of the half: bits 4n..4n+3), stored without waiting.
__device__ __forceinline__ void expand_half_tmem(uint32_t taddr, uint2 bits) {
  uint32_t v[16];
#pragma unroll
  for (int n = 0; n < 8; ++n) {
    v[n] = e4m3x4((bits.x >> (4 * n)) & 0xFu);
    v[8 + n] = e4m3x4((bits.y >> (4 * n)) & 0xFu);
  }
  tmem_st16_issue(taddr, v);
}

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

// The dequantise role (warps kDqWarp0 .. kDqWarp0 + 3, one TMEM lane quarter
// each; TMEM lane = stored row of the CTA's tile). Per module u of a tile: wait
// for the MMAs of d_u, fold acc = fl(acc + term(d_u)) into the running score
// (TMEM columns after the ND accumulators, or shared memory when ACCS), release
// the accumulator; after the last module write the scores (dense) or screen and
// rank them (TOPK). In a CTA pair (PAIR) each CTA drains its own 128 rows and
// releases the accumulator on the leader CTA's barrier.
template <int MODE, bool TOPK, int BN, int ND, bool ACCS, bool PAIR>
__device__ __forceinline__ void dequant_role(const ScoreTcArgs& g, uint8_t* smem, const TcSmem& L, uint32_t tmem,
                                             float* sq, uint64_t* dfull, uint64_t* dempty) {
  constexpr uint32_t kAcc = static_cast<uint32_t>(ND * BN);
  constexpr bool kAccS = ACCS;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q4 = warp & 3;
  const int ep = threadIdx.x - 32 * kDqWarp0;  // TMEM lane (stored row in the tile)
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
  const int dw = ep >> 5;  // dequantise warp 0..3
  int seg_qt = -1;
  // Lists of the finished query tile to global memory; warp dw writes columns dw, dw + 4, ...
  auto flush = [&]() {
    for (int col = dw; col < g.BNq; col += 4) {
      const int q = seg_qt * g.BNq + col;
      if (q < g.Q) {
        const size_t off = (static_cast<size_t>(blockIdx.x) * g.Q + q) * g.K;
        topk_warp_write<2>(list_of(col), lane, g.lst + off, g.lsi + off);
      }
    }
  };
  // Ranks one chunk of 32 query columns (values a[] of this thread's stored row):
  // if no value beats its column's threshold (the usual case once the lists
  // have filled), nothing is staged; otherwise the chunk is staged column-major
  // and warp dw offers 8 of the columns to their lists.
  // Last module of a tile, per chunk of 32 query columns: keep the scores in this
  // CTA's scratch (column-major) and note which columns hold a row that can
  // enter the column's list (one bit per column, per warp).
  float* scr = g.scr + static_cast<size_t>(blockIdx.x) * BN * 128;
  auto screen_chunk = [&](int c0, int q0, int row, const float (&a)[32]) {
    uint32_t bits = 0;
    if (row < g.N) {
      const float4* t4 = reinterpret_cast<const float4*>(taub + c0);
      const float4* g4 = reinterpret_cast<const float4*>(gtb + c0);
#pragma unroll
      for (int j4 = 0; j4 < 8; ++j4) {
        const float4 t = t4[j4], u = g4[j4];
        const float tj[4] = {t.x, t.y, t.z, t.w}, uj[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float x = a[4 * j4 + e];
          const bool live = q0 + c0 + 4 * j4 + e < g.Q;
          bits |= (live && x >= uj[e] && (tj[e] != tj[e] ? x == x : x > tj[e])) ? (1u << (4 * j4 + e)) : 0u;
        }
      }
    }
    const uint32_t wbits = __reduce_or_sync(0xffffffffu, bits);
    if (lane == 0) cmask[(c0 >> 5) * 4 + dw] = wbits;
#pragma unroll
    for (int j = 0; j < 32; ++j) scr[static_cast<size_t>(c0 + j) * 128 + ep] = a[j];
  };
  // After the D buffer is released: the flagged columns, dealt round-robin to
  // the four warps, offered to their lists from the scratch.
  auto rank_tile = [&](int q0, int i0) {
    named_bar_sync(3, 128);  // scratch and masks of every warp visible
    const int nr = min(128, g.N - i0);
    int n = 0;
    for (int c0 = 0; c0 < g.BNq; c0 += 32) {
      const uint32_t* cm = cmask + (c0 >> 5) * 4;
      uint32_t colmask = cm[0] | cm[1] | cm[2] | cm[3];
      for (; colmask; ++n) {
        const int cc = __ffs(colmask) - 1;
        colmask &= colmask - 1;
        if ((n & 3) == dw)
          topk_warp_offer<2>(scr + static_cast<size_t>(c0 + cc) * 128, nr, i0, list_of(c0 + cc), lane,
                             gtb[c0 + cc]);
      }
    }
    named_bar_sync(3, 128);  // lists settled before the next tile screens or flushes
  };
  uint32_t gm = 0;
  bool ok = true;
  for (int tile = tile_begin<TOPK, PAIR>(g), tstep = tile_step<TOPK, PAIR>(), tend = tile_end<TOPK, PAIR>(g);
       tile < tend && ok; tile += tstep) {
    const int qt = tile / g.n_it, ib = tile % g.n_it;
    const int i0 = tile_row0<PAIR>(ib), q0 = qt * g.BNq;
    const int row = i0 + ep;
    if (TOPK && qt != seg_qt) {
      if (seg_qt >= 0) {
        flush();
        named_bar_sync(3, 128);  // every list written before any is reset
      }
      seg_qt = qt;
      q0_cur = q0;
      for (int col = ep; col < BN; col += 128) {
        cntb[col] = 0;
        taub[col] = NAN;
      }
      named_bar_sync(3, 128);
    }
    if (TOPK) {
      // Thresholds other CTAs' lists of these queries have reached (read before the
      // last module's ranking, after the barriers of the module loop).
      for (int col = ep; col < BN; col += 128)
        gtb[col] = q0 + col < g.Q ? topk_unkey32(__ldcg(g.gtau + q0 + col)) : INFINITY;
    }
    // Scales of module u + 1 are loaded while module u is dequantised. The
    // query scales go through shared memory (buffer gm & 1): buffer gm & 1 was
    // last read in module gm - 2, which every thread finished before the
    // barrier of module gm - 1.
    constexpr int kSqPer = (BN + 127) / 128;  // query columns of a tile per dequantise thread
    float si_next = row < g.N ? g.ts[static_cast<size_t>(row) * g.ldts] : 0.f;
    float sq_next[kSqPer];
#pragma unroll
    for (int e = 0; e < kSqPer; ++e) {
      const int c = ep + 128 * e;
      sq_next[e] = (MODE == EOGP_SCORE_CODES && c < g.BNq && q0 + c < g.Q)
                       ? g.qs[static_cast<size_t>(q0 + c) * g.ldqs] : 0.f;
    }
    for (int u = 0; u < g.U; ++u, ++gm) {
      const int buf = static_cast<int>(gm % ND);
      const uint32_t dph = (gm / ND) & 1u;
      const float si = si_next;
      float* sqb = sq + (gm & 1u) * BN;
      if (MODE == EOGP_SCORE_CODES) {
#pragma unroll
        for (int e = 0; e < kSqPer; ++e)
          if (ep + 128 * e < BN) sqb[ep + 128 * e] = sq_next[e];
      }
      if (u + 1 < g.U) {
        si_next = row < g.N ? g.ts[static_cast<size_t>(row) * g.ldts + u + 1] : 0.f;
#pragma unroll
        for (int e = 0; e < kSqPer; ++e) {
          const int c = ep + 128 * e;
          sq_next[e] = (MODE == EOGP_SCORE_CODES && c < g.BNq && q0 + c < g.Q)
                           ? g.qs[static_cast<size_t>(q0 + c) * g.ldqs + u + 1] : 0.f;
        }
      }
      uint32_t w_ok = 1;
      if (lane == 0) w_ok = mbar_wait(&dfull[buf], dph, g.status) ? 1u : 0u;
      w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
      __syncwarp();
      tc_fence_after();
      if (!__syncthreads_and_named(w_ok)) {  // also publishes sqb
        ok = false;
        break;
      }
      const bool last = u + 1 == g.U;
      const uint32_t dcol = tmem + lane_base + buf * static_cast<uint32_t>(BN);
      const uint32_t acol = tmem + lane_base + kAcc;
      float* accrow = reinterpret_cast<float*>(smem + L.acc) + ep * kAccLd;  // kAccS: this row's running score
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
      if (!last) {
        // Running score, 16 columns at a time: the TMEM loads of the next chunk
        // are in flight while this one is combined and stored back.
        uint32_t dr[16], ar[16];
        tmem_ld16_issue(dcol, dr);
        if (!kAccS && u > 0) {
          tmem_ld16_issue(acol, ar);
        } else {
#pragma unroll
          for (int j = 0; j < 16; ++j) ar[j] = 0u;
        }
#pragma unroll
        for (int ci = 0; ci < BN / 16; ++ci) {
          const int c0 = 16 * ci;
          if (c0 < g.BNq) {
            tmem_wait_ld(dr);
            if constexpr (kAccS) {
              if (u > 0) acc_load(c0, ar, 16);
            } else {
              tmem_wait_ld(ar);
            }
            uint32_t o[16];
#pragma unroll
            for (int j = 0; j < 16; ++j)
              o[j] = __float_as_uint(__fadd_rn(__uint_as_float(ar[j]), term(c0 + j, dr[j])));
            if (c0 + 16 < g.BNq) {
              tmem_ld16_issue(dcol + c0 + 16, dr);
              if (!kAccS && u > 0) tmem_ld16_issue(acol + c0 + 16, ar);
            }
            if constexpr (kAccS) {
#pragma unroll
              for (int j = 0; j < 16; j += 4)
                *reinterpret_cast<float4*>(accrow + c0 + j) =
                    make_float4(__uint_as_float(o[j]), __uint_as_float(o[j + 1]), __uint_as_float(o[j + 2]),
                                __uint_as_float(o[j + 3]));
            } else {
              tmem_st16_issue(acol + c0, o);
            }
          }
        }
        if constexpr (!kAccS) tmem_wait_st();  // stored before the next module reads them
      } else {
        for (int c0 = 0; c0 < g.BNq; c0 += 32) {
          uint32_t dr[32], ar[32];
          tmem_ld32_issue(dcol + c0, dr);
          if (u > 0 && kAccS) {
            acc_load(c0, ar, 32);
          } else if (u > 0) {
            tmem_ld32_issue(acol + c0, ar);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) ar[j] = 0u;
          }
          tmem_wait_ld(dr);
          if constexpr (!kAccS) tmem_wait_ld(ar);
          float a[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) a[j] = __fadd_rn(__uint_as_float(ar[j]), term(c0 + j, dr[j]));
          if (!TOPK) {
            if (row < g.N) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
            }
          } else {
            screen_chunk(c0, q0, row, a);
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
      if (TOPK && last) rank_tile(q0, i0);
    }
  }
  if (TOPK && seg_qt >= 0) flush();
}

template <int MODE, bool TOPK, int BN, bool AT, bool F4 = false>
__global__ void __launch_bounds__(kThreadsTc, 1)
    k_score_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQlo,
               const __grid_constant__ ScoreTcArgs g) {
  static_assert(!AT || MODE == EOGP_SCORE_CODES, "operand A in TMEM is the one-bit path");
  static_assert(!F4 || AT, "e2m1 operands are read from TMEM");
  constexpr int S = tc_stages<MODE, TOPK, BN, AT, F4>();
  constexpr uint32_t kStage = tc_stage_bytes<MODE, BN, AT>();
  constexpr uint32_t kBOff = tc_b_offset<AT>();
  // code bits per pipeline stage, and the query operand's TMA x coordinate per
  // stage (elements of its tensor map: e4m3 / e2m1-pair bytes or bf16 values)
  constexpr int kBits = F4 ? 256 : TcMode<MODE>::kBits;
  constexpr int kQx = F4 ? 128 : kBits;
  constexpr uint32_t kSfa = tc_sf_col<S>(), kSfb = kSfa + 16u;
  constexpr int ND = tc_dbufs<BN, AT>();
  using HalfBits = std::conditional_t<F4, uint4, typename TcMode<MODE>::HalfBits>;
  constexpr int kG = 8;  // stages of code bits prefetched at a time
  constexpr int kP = tc_group<MODE, TOPK, BN, AT, F4>();
  constexpr bool kAccS = tc_acc_smem<BN, AT>();
  static_assert(kG % kP == 0, "prefetch groups hold whole expansion rounds");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const TcSmem L = tc_smem_layout<MODE, TOPK, BN, AT, F4>(g.BNq, g.K);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* sq = reinterpret_cast<float*>(smem + L.sq);  // [2][BN] query scales of module u (CODES)
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty = full + S;
  uint64_t* dfull = empty + S;
  uint64_t* dempty = dfull + ND;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(dempty + ND);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    if (MODE == EOGP_SCORE_PAPER) tma_prefetch_desc(&tmQlo);
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1 + kExpWarps);  // TMA transaction arrive + the expander warps
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < ND; ++b) {
      mbar_init(&dfull[b], 1);
      mbar_init(&dempty[b], 4);
    }
    fence_barrier_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tslot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp < kExpWarps) {
    // ---------------------------------------------------------- expanders
    // A stored row's modules are back to back, so pipeline stage j of a tile
    // reads bits [j kBits, (j+1) kBits) of the row and query columns from
    // j kBits on. Two threads share a row (a half stage each). The bits of the
    // next kG stages are loaded into registers while the current kG stages are
    // expanded, hiding the HBM latency. With six stages (one-bit queries, 128
    // per tile) two stages are filled per wait, proxy fence and arrive round.
    const int r = threadIdx.x & 127, half = threadIdx.x >> 7;  // stored row, half of its stage
    const uint32_t row_off = static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128);
    // TMEM A: this thread's row is TMEM lane r (warp w holds lanes 32 (w % 4) ..),
    // its half stage 16 columns of the stage's A slot.
    const uint32_t a_lane = tmem + (static_cast<uint32_t>(r & ~31) << 16) + 16u * static_cast<uint32_t>(half);
    if constexpr (F4) {
      // unit scale factors, once: warps 0-3 cover the four TMEM lane quarters
      if (half == 0) {
        uint32_t v[16];
#pragma unroll
        for (int e = 0; e < 16; ++e) v[e] = 0x7F7F7F7Fu;
        const uint32_t q_lane = tmem + (static_cast<uint32_t>(r & ~31) << 16);
        tmem_st16_issue(q_lane + kSfa, v);
        tmem_st16_issue(q_lane + kSfb, v);
        tmem_wait_st();  // ordered before this warp's first arrive on a full barrier
      }
    }
    auto put = [&](int s, uint8_t* st, HalfBits bits) {
      if constexpr (AT) {
        tc_fence_after();  // the MMAs that read the slot before (released through empty[s]) are done
        expand_half_tmem(a_lane + tc_acol<BN>(s), bits);
      } else {
        expand_half(st + row_off, r & 7, half, bits);
      }
    };
    // the half stages written so far become visible to the MMA issuer once the
    // warp's lane 0 arrives on the stage's barrier
    auto publish = [&]() {
      if constexpr (AT) {
        tmem_wait_st();
        tc_fence_before();
      } else {
        fence_proxy_async_smem();
      }
    };
    const int nst = g.D / kBits;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = tile_begin<TOPK>(g), tstep = tile_step<TOPK>(), tend = tile_end<TOPK>(g);
         tile < tend && ok; tile += tstep) {
      const int qt = tile / g.n_it, ib = tile % g.n_it;
      const int i0 = ib * 128, q0 = qt * g.BNq;
      const bool rv = i0 + r < g.N;
      const HalfBits* brow =
          reinterpret_cast<const HalfBits*>(g.train + static_cast<size_t>(rv ? i0 + r : 0) * g.ldt) + half;
      HalfBits cur[kG], nxt[kG];
#pragma unroll
      for (int jj = 0; jj < kG; ++jj) cur[jj] = (rv && jj < nst) ? __ldg(brow + 2 * jj) : HalfBits{};
      for (int j0 = 0; j0 < nst && ok; j0 += kG) {
#pragma unroll
        for (int jj = 0; jj < kG; ++jj)
          nxt[jj] = (rv && j0 + kG + jj < nst) ? __ldg(brow + 2 * (j0 + kG + jj)) : HalfBits{};
        if constexpr (kP == 1) {
#pragma unroll
          for (int jj = 0; jj < kG; ++jj) {
            const int j = j0 + jj;
            if (j < nst && ok) {
              const int s = static_cast<int>(it % S);
              const uint32_t ph = (it / S) & 1u;
              ++it;
              uint32_t w_ok = 1;
              if (lane == 0) w_ok = mbar_wait(&empty[s], ph ^ 1u, g.status) ? 1u : 0u;
              w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
              if (!w_ok) {
                ok = false;
              } else {
                uint8_t* st = smem + static_cast<size_t>(s) * kStage;
                if (warp == 0 && lane == 0) {
                  mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(g.BNq) * 128u * TcMode<MODE>::kQBoxes);
                  tma_load_2d(st + kBOff, &tmQ, j * kQx, q0, &full[s]);
                  if (MODE == EOGP_SCORE_PAPER)
                    tma_load_2d(st + kBOff + static_cast<uint32_t>(BN) * 128u, &tmQlo, j * kQx, q0, &full[s]);
                }
                put(s, st, cur[jj]);
                publish();
                __syncwarp();
                if (lane == 0) mbar_arrive(&full[s]);
              }
            }
          }
        } else {
          static_assert(MODE == EOGP_SCORE_CODES, "two-stage rounds load one query operand per stage");
#pragma unroll
          for (int jj = 0; jj < kG; jj += 2) {
            const int j = j0 + jj;
            if (j < nst && ok) {
              const bool two = j + 1 < nst;
              const int s0 = static_cast<int>(it % S), s1 = static_cast<int>((it + 1) % S);
              const uint32_t ph0 = (it / S) & 1u, ph1 = ((it + 1) / S) & 1u;
              it += two ? 2 : 1;
              uint32_t w_ok = 1;
              if (lane == 0) {
                w_ok = mbar_wait(&empty[s0], ph0 ^ 1u, g.status) ? 1u : 0u;
                if (w_ok && two) w_ok = mbar_wait(&empty[s1], ph1 ^ 1u, g.status) ? 1u : 0u;
              }
              w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
              if (!w_ok) {
                ok = false;
              } else {
                uint8_t* st0 = smem + static_cast<size_t>(s0) * kStage;
                uint8_t* st1 = smem + static_cast<size_t>(s1) * kStage;
                if (warp == 0 && lane == 0) {
                  const uint32_t qbytes = static_cast<uint32_t>(g.BNq) * 128u * TcMode<MODE>::kQBoxes;
                  mbar_arrive_expect_tx(&full[s0], qbytes);
                  tma_load_2d(st0 + kBOff, &tmQ, j * kQx, q0, &full[s0]);
                  if (two) {
                    mbar_arrive_expect_tx(&full[s1], qbytes);
                    tma_load_2d(st1 + kBOff, &tmQ, (j + 1) * kQx, q0, &full[s1]);
                  }
                }
                put(s0, st0, cur[jj]);
                if (two) put(s1, st1, cur[jj + 1]);
                publish();
                __syncwarp();
                if (lane == 0) {
                  mbar_arrive(&full[s0]);
                  if (two) mbar_arrive(&full[s1]);
                }
              }
            }
          }
        }
#pragma unroll
        for (int jj = 0; jj < kG; ++jj) cur[jj] = nxt[jj];
      }
    }
  } else if (warp < kMmaWarp) {
    dequant_role<MODE, TOPK, BN, ND, kAccS, false>(g, smem, L, tmem, sq, dfull, dempty);
  } else {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = F4 ? idesc_mxf4_f32(128, g.BNq)
                             : MODE == EOGP_SCORE_CODES ? idesc_e4m3_f32(128, g.BNq)
                                                        : idesc_bf16_f32(128, g.BNq, 0, 0);
      const uint32_t sfa = tmem + kSfa, sfb = tmem + kSfb;  // e2m1: unit scale factors
      // One lane issues every MMA, so its own work per stage is kept minimal:
      // ring slot, phase, A slot and descriptors advance incrementally (a
      // descriptor's address field is byte address >> 4: +2 steps 32 bytes).
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      uint64_t dst = dbase;  // descriptor of ring slot rs (its first operand tile)
      uint32_t acl = tmem + tc_acol<BN>(0);  // TMEM A slot of ring slot rs (AT)
      int rs = 0;
      uint32_t rph = 0, gm = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK>(g), tstep = tile_step<TOPK>(), tend = tile_end<TOPK>(g);
           tile < tend && ok; tile += tstep) {
        for (int u = 0; u < g.U && ok; ++u, ++gm) {
          const int buf = static_cast<int>(gm % ND);
          const uint32_t dph = (gm / ND) & 1u;
          if (!mbar_wait(&dempty[buf], dph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + buf * static_cast<uint32_t>(BN);
          const int nkb = g.k[u] / kBits;
          for (int kb = 0; kb < nkb; ++kb) {
            const int s = rs;
            const uint32_t ph = rph;
            const uint64_t a0 = dst;  // A (shared-memory A) or the query operand (TMEM A)
            const uint64_t b0 = dst + (kAB >> 4), b1 = b0 + ((static_cast<uint32_t>(BN) * 128u) >> 4);
            const uint32_t at0 = acl;
            if (++rs == S) {
              rs = 0;
              rph ^= 1u;
              dst = dbase;
              acl = tmem + tc_acol<BN>(0);
            } else {
              dst += kStage >> 4;
              acl += 32u;
            }
            if (!mbar_wait(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
              if constexpr (F4) {
                tc_mma_f4_ta(d, at0 + 8u * kk, a0 + 2 * kk, idesc, sfa, sfb, acc);
              } else if constexpr (AT) {
                tc_mma_f8_ta(d, at0 + 8u * kk, a0 + 2 * kk, idesc, acc);
              } else if (MODE == EOGP_SCORE_CODES) {
                tc_mma_f8(d, a0 + 2 * kk, b0 + 2 * kk, idesc, acc);
              } else {
                tc_mma_f16(d, a0 + 2 * kk, b0 + 2 * kk, idesc, acc);
                tc_mma_f16(d, a0 + 2 * kk, b1 + 2 * kk, idesc, 1u);
              }
            }
            tc_commit(&empty[s]);
          }
          tc_commit(&dfull[buf]);
        }
      }
    }
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == kMmaWarp) tmem_dealloc(tmem, 512);
}

// ------------------------------------------------------------------------
// k_score_pair -- one-bit (CODES) scoring with e2m1 operands on CTA pairs.
//
// A pair works on 256 stored rows (MMA M = 256, tcgen05 cta_group::2): each
// CTA expands its own 128 rows into its own TMEM (operand A) and loads its own
// half of the tile's queries (operand B, BNq / 2 rows per CTA, no multicast);
// the leader CTA (rank 0) issues the MMAs, whose accumulator rows land in each
// CTA's TMEM, so each CTA dequantises its own rows exactly as the one-CTA
// kernel does. Against one CTA per 128-row tile this halves the query
// operand's stream from L2 per stored row.
//
// Two rings:
//  * code boxes (shared memory, 4 or 8 x 16 KB): 128 rows x 1024 code bits,
//    128-byte swizzle, loaded by TMA so that HBM latency is hidden by the ring
//    rather than by registers;
//  * stages (S of them): a query stage in shared memory (BNq / 2 rows x 128
//    bytes of e2m1, loaded by TMA as soon as the MMAs release the stage) and an
//    A slot of 32 TMEM columns (the expanded stored rows), released together by
//    one MMA commit. (Separate rings for the two, with their own barriers,
//    commits and depths, measured 1.3x slower.)
// One producer thread per TMA stream runs ahead as far as its ring allows. Each expander
// warp takes whole stages of its 32 rows (warps 0-3 the even stages of a
// tile, 4-7 the odd ones): two 16-byte shared-memory loads, the e2m1 expansion
// (same K order as the one-CTA kernel and the query expansion), the TMEM
// stores, and one relaxed arrive on the leader's barrier of the A slot. That
// arrive orders enough: it is issued after tcgen05.wait::st, which returns only
// once the thread's TMEM stores have completed, and after the tcgen05 fence;
// the leader issues the MMAs only after observing it; and in the pair MMA each
// SM's tensor core reads operand A from its own CTA's TMEM, which no cache sits
// in front of. (The pair rotation kernel releases its accumulators the same
// way.) Measured on the scan at Q = 1024: 23.0 ms with relaxed arrives, 30.0 ms
// with CTA-scope release, 30.9 ms with cluster-scope release, and 44.8 ms when
// one thread of the peer forwards every stage with one cluster-scope release.
//
// Warps: 0-7 expand, 8-11 dequantise (dequant_role), 12 owns TMEM and, in the
// leader, issues the MMAs, 13 loads the code boxes, 14 the query stages.
// ------------------------------------------------------------------------
constexpr int kPairThreads = (kExpWarps + 4 + 1 + 2) * 32;
constexpr int kCodeWarp = kMmaWarp + 1;
constexpr int kQueryWarp = kMmaWarp + 2;
constexpr int kCodeBoxWords = 32;            // 1024 code bits of a row per box (4 stages)
constexpr uint32_t kCodeBox = 128u * 128u;   // 128 rows x 128 bytes

// TMEM: one accumulator of 256 columns (256 queries per tile, one module), else
// two of BN columns; then the A slots of 32 columns; then the unit scale
// factors (16 columns each for A and B).
template <int BN>
constexpr int pr_dbufs() {
  return BN == 256 ? 1 : 2;
}
template <int BN>
constexpr int pr_stages() {
  return (512 - pr_dbufs<BN>() * BN - 32) / 32;
}
// The running score of several modules lives in shared memory; only 128-query
// tiles serve several modules (64-query tiles have no room for it in TMEM
// either, so they serve one module, and 256-query tiles keep one accumulator).
template <int BN>
constexpr bool pr_acc_smem() {
  return BN == 128;
}
// Code boxes in flight: as many as the shared memory holds next to the query
// stages (and the running score of several modules).
template <int BN>
constexpr int pr_code_ring() {
  return BN == 64 ? 8 : BN == 256 ? 6 : 4;
}
template <int BN>
constexpr uint32_t pr_acol0() {
  return static_cast<uint32_t>(pr_dbufs<BN>() * BN);
}
template <int BN>
constexpr uint32_t pr_sf_col() {
  return pr_acol0<BN>() + 32u * static_cast<uint32_t>(pr_stages<BN>());
}

// Shared memory: query stages, the code ring, then the layout the dequantise
// role shares with the one-CTA kernel (running score, query scales, barriers,
// ranking state).
template <bool TOPK, int BN>
__host__ __device__ inline TcSmem pr_smem_layout(uint32_t* code_off) {
  constexpr int S = pr_stages<BN>(), kCodeRing = pr_code_ring<BN>();
  constexpr uint32_t kStage = static_cast<uint32_t>(BN / 2) * 128u;
  TcSmem l;
  *code_off = S * kStage;
  l.acc = *code_off + kCodeRing * kCodeBox;
  l.sq = l.acc + (pr_acc_smem<BN>() ? 128u * kAccLd * 4u : 0u);
  l.bars = l.sq + 2 * BN * 4;
  l.lists = l.bars + (2 * S + 2 * pr_dbufs<BN>() + 2 * kCodeRing) * 8 + 16;
  l.total = l.lists + (TOPK ? BN * 12 + 8 * 4 * 4 : 0);
  return l;
}

// Waits with all lanes of the warp; true when every lane saw the phase complete.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned* status) {
  return __all_sync(0xffffffffu, mbar_wait(bar, parity, status));
}

template <bool TOPK, int BN>
__global__ void __launch_bounds__(kPairThreads, 1)
    k_score_pair(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmC,
                 const __grid_constant__ ScoreTcArgs g) {
  constexpr int S = pr_stages<BN>(), ND = pr_dbufs<BN>();
  constexpr int kCodeRing = pr_code_ring<BN>();
  constexpr uint32_t kStage = static_cast<uint32_t>(BN / 2) * 128u;
  constexpr uint32_t kSfa = pr_sf_col<BN>(), kSfb = kSfa + 16u;
  static_assert(kSfb + 16u <= 512u, "TMEM budget");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint32_t code_off;
  const TcSmem L = pr_smem_layout<TOPK, BN>(&code_off);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  float* sq = reinterpret_cast<float*>(smem + L.sq);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty = full + S;
  uint64_t* dfull = empty + S;
  uint64_t* dempty = dfull + ND;
  uint64_t* cfull = dempty + ND;
  uint64_t* cempty = cfull + kCodeRing;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(cempty + kCodeRing);
  const int nst = g.D / 256;            // 256-bit stages per tile
  const int nbx = (nst + 3) / 4;        // code boxes per tile

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmC);
    for (int s = 0; s < S; ++s) {
      // leader's copy: per CTA the query producer's expect_tx arrive (+ its TMA
      // bytes) and the stage's four expander warps
      mbar_init(&full[s], 2 * (1 + kExpWarps / 2));
      mbar_init(&empty[s], 1);  // MMA completion, multicast to both CTAs
    }
    for (int b = 0; b < ND; ++b) {
      mbar_init(&dfull[b], 1);   // multicast to both CTAs
      mbar_init(&dempty[b], 8);  // 4 dequantise warps x 2 CTAs (leader's copy)
    }
    for (int b = 0; b < kCodeRing; ++b) {
      mbar_init(&cfull[b], 1);           // the producer's expect_tx arrive (+ TMA bytes)
      mbar_init(&cempty[b], kExpWarps);  // every expander warp, once per box
    }
    fence_barrier_init();
  }
  if (warp == kMmaWarp) tmem_alloc_pair(tslot, 512);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp < kExpWarps) {
    // ---------------------------------------------------------- expanders
    const int q4 = warp & 3, par = warp >> 2;  // lane quarter, stage parity
    const int r = q4 * 32 + lane;              // stored row in the CTA's tile = TMEM lane
    const uint32_t a_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    if (par == 0) {  // unit scale factors (ue8m0 0x7F = 1.0) of A and B, once
      uint32_t v[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) v[e] = 0x7F7F7F7Fu;
      tmem_st16_issue(a_lane + kSfa, v);
      tmem_st16_issue(a_lane + kSfb, v);
      tmem_wait_st();  // ordered before this warp's first arrive on a full barrier
    }
    const uint32_t row_sw = static_cast<uint32_t>(r & 7);
    uint32_t it = 0, bx = 0;  // stages and code boxes of earlier tiles
    bool ok = true;
    for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
         tile < tend && ok; tile += tstep) {
      for (int bt = 0; bt < nbx && ok; ++bt) {
        const uint32_t b = bx + bt;
        const int cs = static_cast<int>(b % kCodeRing);
        if (!warp_wait(&cfull[cs], (b / kCodeRing) & 1u, g.status)) {
          ok = false;
          break;
        }
        const uint8_t* crow = smem + code_off + cs * kCodeBox + r * 128;
        for (int sub = par; sub < 4; sub += 2) {
          const int jt = 4 * bt + sub;  // stage within the tile
          if (jt >= nst) break;
          const uint32_t j = it + jt;
          const int sa = static_cast<int>(j % S);
          if (!warp_wait(&empty[sa], ((j / S) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          const uint4 w0 = *reinterpret_cast<const uint4*>(crow + (((2 * sub) ^ row_sw) << 4));
          const uint4 w1 = *reinterpret_cast<const uint4*>(crow + (((2 * sub + 1) ^ row_sw) << 4));
          tc_fence_after();  // the MMAs that read the slot before (released through empty) are done
          const uint32_t acol = a_lane + pr_acol0<BN>() + 32u * sa;
          expand_half_tmem(acol, w0);
          expand_half_tmem(acol + 16u, w1);
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(&full[sa]), 0));
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&cempty[cs]);  // this warp is done reading box b
      }
      it += nst;
      bx += nbx;
    }
  } else if (warp < kMmaWarp) {
    dequant_role<EOGP_SCORE_CODES, TOPK, BN, ND, pr_acc_smem<BN>(), true>(g, smem, L, tmem, sq, dfull, dempty);
  } else if (warp == kMmaWarp) {
    if (lane == 0 && rank == 0) {
      // ---------------------------------------------------------- MMA issuer (leader)
      const uint32_t idesc = idesc_mxf4_f32(256, g.BNq);
      const uint32_t sfa = tmem + kSfa, sfb = tmem + kSfb;
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      uint64_t dq = dbase;                   // descriptor of query stage rs
      uint32_t acl = tmem + pr_acol0<BN>();  // A slot rs
      int rs = 0;
      uint32_t rph = 0, gm = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
           tile < tend && ok; tile += tstep) {
        for (int u = 0; u < g.U && ok; ++u, ++gm) {
          const int buf = static_cast<int>(gm % ND);
          if (!mbar_wait_cluster(&dempty[buf], ((gm / ND) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + buf * static_cast<uint32_t>(BN);
          const int nkb = g.k[u] / 256;
          for (int kb = 0; kb < nkb; ++kb) {
            const int s = rs;
            const uint32_t ph = rph;
            const uint64_t b0 = dq;
            const uint32_t at0 = acl;
            if (++rs == S) {
              rs = 0;
              rph ^= 1u;
              dq = dbase;
              acl = tmem + pr_acol0<BN>();
            } else {
              dq += kStage >> 4;
              acl += 32u;
            }
            // both CTAs' query bytes and expander warps
            if (!mbar_wait_cluster(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_f4_ta_pair(d, at0 + 8u * kk, b0 + 2 * kk, idesc, sfa, sfb, (kb | kk) != 0 ? 1u : 0u);
            tc_commit_pair_mc(&empty[s], 0x3);
          }
          tc_commit_pair_mc(&dfull[buf], 0x3);
        }
      }
    }
    __syncwarp();
  } else if (warp == kCodeWarp) {
    // ---------------------------------------------------------- code producer
    // This CTA's rows, one box of four stages at a time, as far ahead as the
    // code ring allows.
    if (lane == 0) {
      uint32_t bx = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
           tile < tend && ok; tile += tstep) {
        const int i0 = tile_row0<true>(tile % g.n_it);
        for (int bt = 0; bt < nbx; ++bt) {
          const uint32_t b = bx + bt;
          const int cs = static_cast<int>(b % kCodeRing);
          if (!mbar_wait(&cempty[cs], ((b / kCodeRing) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&cfull[cs], kCodeBox);
          tma_load_2d(smem + code_off + cs * kCodeBox, &tmC, bt * kCodeBoxWords, i0, &cfull[cs]);
        }
        bx += nbx;
      }
    }
    __syncwarp();
  } else if (warp == kQueryWarp) {
    // ---------------------------------------------------------- query producer
    // This CTA's half of each stage's query rows, as soon as the MMAs release
    // the stage; the bytes are counted on the leader's barrier.
    if (lane == 0) {
      const uint32_t qbytes = static_cast<uint32_t>(g.BNq / 2) * 128u;
      uint32_t it = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
           tile < tend && ok; tile += tstep) {
        const int qrow = (tile / g.n_it) * g.BNq + static_cast<int>(rank) * (g.BNq / 2);
        for (int jt = 0; jt < nst; ++jt) {
          const uint32_t j = it + jt;
          const int s = static_cast<int>(j % S);
          if (!mbar_wait(&empty[s], ((j / S) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          const uint32_t fl = mapa_shared(smem_u32(&full[s]), 0);
          mbar_arrive_expect_tx_cluster(fl, qbytes);
          tma_load_2d_pair(smem_u32(smem + s * kStage), &tmQ, jt * 128, qrow, fl);
        }
        it += nst;
      }
    }
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while its peer may still signal it
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc_pair(tmem, 512);
}

// Query codes -> e4m3 bytes: out[q][c] = +1 / -1 for bit c of the concatenated modules.
__global__ void k_expand_queries(const uint32_t* __restrict__ query, int ldq, int row_bytes,
                                 uint8_t* __restrict__ out) {
  const int q = blockIdx.y;
  const int wtot = (row_bytes >> 5);  // words per row (32 bits -> 32 bytes)
  for (int w = blockIdx.x * blockDim.x + threadIdx.x; w < wtot; w += gridDim.x * blockDim.x) {
    const uint32_t v = query[static_cast<size_t>(q) * ldq + w];
    uint4 a, b;
    const uint64_t e0 = expand8(v), e1 = expand8(v >> 8), e2 = expand8(v >> 16), e3 = expand8(v >> 24);
    a = make_uint4(static_cast<uint32_t>(e0), static_cast<uint32_t>(e0 >> 32), static_cast<uint32_t>(e1),
                   static_cast<uint32_t>(e1 >> 32));
    b = make_uint4(static_cast<uint32_t>(e2), static_cast<uint32_t>(e2 >> 32), static_cast<uint32_t>(e3),
                   static_cast<uint32_t>(e3 >> 32));
    uint4* o = reinterpret_cast<uint4*>(out + static_cast<size_t>(q) * row_bytes + w * 32);
    o[0] = a;
    o[1] = b;
  }
}

// Query codes -> e2m1 +-1 in the stored rows' TMEM order (e2m1x8): word w of a
// row gives output bytes 16 w .. 16 w + 15, column j of the word in bytes
// 16 w + 4 j .. + 3 (two values per byte, the lower K index in the low nibble).
__global__ void k_expand_queries_f4(const uint32_t* __restrict__ query, int ldq, int row_bytes,
                                    uint8_t* __restrict__ out) {
  const int q = blockIdx.y;
  const int wtot = row_bytes >> 4;  // words per row (32 bits -> 16 bytes)
  for (int w = blockIdx.x * blockDim.x + threadIdx.x; w < wtot; w += gridDim.x * blockDim.x) {
    const uint32_t v = query[static_cast<size_t>(q) * ldq + w];
    reinterpret_cast<uint4*>(out + static_cast<size_t>(q) * row_bytes)[w] =
        make_uint4(e2m1x8(v, 0), e2m1x8(v, 1), e2m1x8(v, 2), e2m1x8(v, 3));
  }
}

// Query coordinates y (fp32) -> bf16 hi = rn(y) and lo = rn(y - hi), dense rows of D.
__global__ void k_split_queries(const float* __restrict__ y, int ldq, int D,
                                __nv_bfloat16* __restrict__ hi, __nv_bfloat16* __restrict__ lo) {
  const int q = blockIdx.y;
  for (int c = blockIdx.x * blockDim.x + threadIdx.x; c < D; c += gridDim.x * blockDim.x) {
    const float v = y[static_cast<size_t>(q) * ldq + c];
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    hi[static_cast<size_t>(q) * D + c] = h;
    lo[static_cast<size_t>(q) * D + c] = __float2bfloat16_rn(v - __bfloat162float(h));
  }
}

template <int MODE, bool TOPK, int BN, bool AT = false, bool F4 = false>
size_t tc_smem_need(int BNq, int K) {
  return 1024 + tc_smem_layout<MODE, TOPK, BN, AT, F4>(BNq, K).total;
}

// Operand A of the one-bit (CODES) kernel is written to TMEM; the PAPER kernel
// keeps its bf16 +-1 operand in shared memory.
bool tc_a_in_tmem(int mode) { return mode == EOGP_SCORE_CODES; }

// e2m1 (fp4) operands for the one-bit kernel: the MMA (kind::mxf4 with unit
// scales, exact for +-1) runs at twice the e4m3 rate and a stage carries 256
// code bits. Needs every module a multiple of 256 bits (the 16-byte row
// alignment the TMA of the stored codes needs is a precondition of every
// tensor-core scoring call); EOGP_OPT_SCORE_OPERAND = 1 keeps e4m3.
bool tc_f4(int mode, const int* ks, int U) {
  if (!tc_a_in_tmem(mode)) return false;
  if (eogp::option(EOGP_OPT_SCORE_OPERAND) == 1) return false;
  for (int u = 0; u < U; ++u)
    if (ks[u] % 256) return false;
  return true;
}

// Queries per tile of the one-CTA kernel: 256 for CODES with one module and
// enough queries (when the shared memory allows), else 128. (Measured with
// operand A in TMEM on the 4.2M-code scan at Q = 1024: 48.0 ms with 256-query
// tiles and one accumulator, 63.2 ms with 192-query tiles and two: the
// expansion is repeated per query tile.)
int tc_bn(int mode, int U, int Q, int K) {
  if (mode == EOGP_SCORE_CODES && U == 1 && Q >= 256 &&
      (K == 0 || tc_smem_need<EOGP_SCORE_CODES, true, 256>(256, K) <= 232448))
    return 256;
  return 128;
}

// Queries per tile of the pair kernel. One module: 256 for more than 128
// queries (one accumulator), 64 for at most 64 (more A slots and code boxes;
// an N = 64 MMA takes as long as an N = 128 one), else 128. Several modules:
// 128 (the running score needs the shared memory the other widths use).
int pr_bn(int U, int Q) { return U > 1 ? 128 : Q > 128 ? 256 : Q <= 64 ? 64 : 128; }

int bnq_for(int Q, int BN) { return std::min(BN, (Q + 31) / 32 * 32); }

template <bool TOPK, int BN>
size_t pr_smem_need() {
  uint32_t code_off;
  return 1024 + pr_smem_layout<TOPK, BN>(&code_off).total;
}

// The kernel a call runs and its tiling.
struct TcCfg {
  bool pair;  // k_score_pair (one-bit, e2m1) or k_score_tc
  bool f4;    // e2m1 operands
  int BN, BNq, rows;  // queries per tile (template, actual), stored rows per tile
};
TcCfg tc_cfg(int mode, const int* ks, int U, int Q, int K) {
  TcCfg c;
  c.f4 = tc_f4(mode, ks, U);
  c.pair = c.f4;
  c.BN = c.pair ? pr_bn(U, Q) : tc_bn(mode, U, Q, K);
  c.BNq = bnq_for(Q, c.BN);
  c.rows = c.pair ? 256 : 128;
  return c;
}

// Clusters of two k_score_pair CTAs that can be resident at once on the
// current device, cached per device index (half the SMs when it cannot be read).
int pair_cluster_cap(int num_sms) {
  static std::atomic<int> cache[128];
  int dev = 0;
  const int fallback = std::max(1, num_sms / 2);
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return fallback;
  int v = cache[dev].load(std::memory_order_relaxed);
  if (v > 0) return v;
  const size_t smem = pr_smem_need<true, 128>();
  if (cudaFuncSetAttribute(k_score_pair<true, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(smem)) != cudaSuccess)
    return fallback;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * fallback);
  cfg.blockDim = dim3(kPairThreads);
  cfg.dynamicSmemBytes = smem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k_score_pair<true, 128>, &cfg) != cudaSuccess || n < 1) {
    cudaGetLastError();
    return fallback;
  }
  v = std::min(n, fallback);
  cache[dev].store(v, std::memory_order_relaxed);
  return v;
}

// CTAs of a call: one per SM at most (one CTA, or one pair per two SMs).
int tc_grid(const TcCfg& c, int N, int Q, int num_sms) {
  const long long tiles = static_cast<long long>((N + c.rows - 1) / c.rows) * ((Q + c.BNq - 1) / c.BNq);
  if (c.pair) return 2 * static_cast<int>(std::max<long long>(1, std::min<long long>(tiles, pair_cluster_cap(num_sms))));
  return static_cast<int>(std::max<long long>(1, std::min<long long>(tiles, std::max(1, num_sms))));
}

template <int MODE, bool TOPK, int BN, bool AT, bool F4 = false>
cudaError_t launch_tc_kernel(const CUtensorMap& t0, const CUtensorMap& t1, const ScoreTcArgs& g,
                             int grid, cudaStream_t st) {
  const size_t smem = tc_smem_need<MODE, TOPK, BN, AT, F4>(g.BNq, g.K);
  cudaError_t e = cudaFuncSetAttribute(k_score_tc<MODE, TOPK, BN, AT, F4>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  k_score_tc<MODE, TOPK, BN, AT, F4><<<grid, kThreadsTc, smem, st>>>(t0, t1, g);
  return cudaGetLastError();
}

template <bool TOPK, int BN>
cudaError_t launch_pair_kernel(const CUtensorMap& tq, const CUtensorMap& tc, const ScoreTcArgs& g, int grid,
                               cudaStream_t st) {
  const size_t smem = pr_smem_need<TOPK, BN>();
  cudaError_t e = cudaFuncSetAttribute(k_score_pair<TOPK, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kPairThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_score_pair<TOPK, BN>, tq, tc, g);
}

template <bool TOPK>
cudaError_t dispatch_tc(int mode, const TcCfg& c, const CUtensorMap& t0, const CUtensorMap& t1,
                        const ScoreTcArgs& g, int grid, cudaStream_t st) {
  if (c.BN == 256 && g.U != 1) return cudaErrorInvalidValue;  // 256-query tiles keep no running score
  if (mode == EOGP_SCORE_PAPER) return launch_tc_kernel<EOGP_SCORE_PAPER, TOPK, 128, false>(t0, t1, g, grid, st);
  if (c.pair) {
    if (c.BN == 64 && g.U != 1) return cudaErrorInvalidValue;  // 64-query tiles keep no running score
    if (c.BN == 256) return launch_pair_kernel<TOPK, 256>(t0, t1, g, grid, st);
    if (c.BN == 64) return launch_pair_kernel<TOPK, 64>(t0, t1, g, grid, st);
    return launch_pair_kernel<TOPK, 128>(t0, t1, g, grid, st);
  }
  if (c.BN == 256) return launch_tc_kernel<EOGP_SCORE_CODES, TOPK, 256, true>(t0, t1, g, grid, st);
  return launch_tc_kernel<EOGP_SCORE_CODES, TOPK, 128, true>(t0, t1, g, grid, st);
}

}  // namespace

bool score_tc_supported(int mode, const int* ks, int U, int Q) {
  if (U < 1 || U > kMaxMods || Q < 1 || Q > 65535) return false;
  if (mode == EOGP_SCORE_CODES) {
    if (Q < 64) return false;  // the popcount kernels are faster for a handful of queries
    for (int u = 0; u < U; ++u)
      if (ks[u] <= 0 || ks[u] % 128) return false;
    return true;
  }
  if (mode == EOGP_SCORE_PAPER) {
    for (int u = 0; u < U; ++u)
      if (ks[u] <= 0 || ks[u] % 64) return false;
    return true;
  }
  return false;
}

size_t score_tc_list_buf_bytes(int mode, const int* ks, int U, int Q, int K, int grid) {
  const TcCfg c = tc_cfg(mode, ks, U, Q, K);
  return static_cast<size_t>(grid) * c.BNq * kFusedCap * 4;  // each of scores and indices
}

size_t score_tc_scratch_bytes(int mode, const int* ks, int U, int Q, int K, int grid) {
  return static_cast<size_t>(grid) * tc_cfg(mode, ks, U, Q, K).BN * 128 * 4;
}

size_t score_tc_ws_bytes(int mode, const int* ks, int U, int Q) {
  long long D = 0;
  for (int u = 0; u < U; ++u) D += ks[u];
  const size_t per = mode == EOGP_SCORE_PAPER ? 4 : 1;  // bf16 hi + lo, or e4m3
  return (static_cast<size_t>(Q) * D * per + 255) & ~size_t(255);
}

int score_tc_grid(int mode, const int* ks, int U, int N, int Q, int K, int num_sms) {
  return tc_grid(tc_cfg(mode, ks, U, Q, K), N, Q, num_sms);
}

bool score_tc_topk_fits(int mode, const int* ks, int U, int Q, int K) {
  if (K < 1 || K > kTopKMax) return false;
  const TcCfg c = tc_cfg(mode, ks, U, Q, K);
  size_t need;
  if (mode == EOGP_SCORE_PAPER)
    need = tc_smem_need<EOGP_SCORE_PAPER, true, 128>(c.BNq, K);
  else if (c.pair)
    need = c.BN == 256 ? pr_smem_need<true, 256>() : c.BN == 64 ? pr_smem_need<true, 64>() : pr_smem_need<true, 128>();
  else
    need = c.BN == 256 ? tc_smem_need<EOGP_SCORE_CODES, true, 256, true>(c.BNq, K)
                       : tc_smem_need<EOGP_SCORE_CODES, true, 128, true>(c.BNq, K);
  return need <= 232448;
}

cudaError_t launch_score_tc(int mode, const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                            const int* ks, int U, const void* query, int ldq, const float* qs,
                            int ldqs, int Q, float* out, int ldo, const TcTopK* topk, void* ws,
                            int num_sms, unsigned* status, cudaStream_t st) {
  if (N <= 0 || Q <= 0) return cudaSuccess;
  const TcCfg c = tc_cfg(mode, ks, U, Q, topk ? topk->K : 0);
  ScoreTcArgs g;  // ~4 KB parameter block, copied at launch
  g.N = N;
  g.Q = Q;
  g.U = U;
  g.BNq = c.BNq;
  g.n_it = (N + c.rows - 1) / c.rows;
  g.n_tiles = g.n_it * ((Q + g.BNq - 1) / g.BNq);
  g.ldt = ldt;
  g.ldts = ldts;
  g.ldqs = ldqs;
  g.ldo = ldo;
  g.K = topk ? topk->K : 0;
  g.train = train;
  g.ts = ts;
  g.qs = qs;
  g.out = out;
  g.lst = topk ? topk->lst : nullptr;
  g.lsi = topk ? topk->lsi : nullptr;
  g.bufs = topk ? topk->bufs : nullptr;
  g.bufi = topk ? topk->bufi : nullptr;
  g.gtau = topk ? topk->gtau : nullptr;
  g.scr = topk ? topk->scr : nullptr;
  g.status = status;
  int D = 0;
  for (int u = 0; u < U; ++u) {
    g.k[u] = ks[u];
    D += ks[u];
  }
  g.D = D;
  const int grid = tc_grid(c, N, Q, num_sms);
  CUtensorMap t0, t1;
  if (mode == EOGP_SCORE_CODES) {
    // expanded query rows: D e4m3 bytes, or D / 2 bytes of e2m1 pairs
    uint8_t* qx = static_cast<uint8_t*>(ws);
    const int row_bytes = c.f4 ? D / 2 : D;
    dim3 eg(std::max(1, std::min((D / 32 + 255) / 256, 64)), Q);
    if (c.f4)
      k_expand_queries_f4<<<eg, 256, 0, st>>>(static_cast<const uint32_t*>(query), ldq, row_bytes, qx);
    else
      k_expand_queries<<<eg, 256, 0, st>>>(static_cast<const uint32_t*>(query), ldq, D, qx);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const uint64_t dims[2] = {static_cast<uint64_t>(row_bytes), static_cast<uint64_t>(Q)};
    const uint64_t strides[1] = {static_cast<uint64_t>(row_bytes)};
    // a pair CTA loads half of the tile's query rows
    const uint32_t box[2] = {128, static_cast<uint32_t>(c.pair ? g.BNq / 2 : g.BNq)};
    if (make_tmap(&t0, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, qx, dims, strides, box,
                  CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
    t1 = t0;
    if (c.pair) {
      // stored code rows: boxes of 32 words (1024 bits) x 128 rows, 128-byte swizzle
      const uint64_t cdims[2] = {static_cast<uint64_t>(D / 32), static_cast<uint64_t>(N)};
      const uint64_t cstr[1] = {static_cast<uint64_t>(ldt) * 4};
      const uint32_t cbox[2] = {static_cast<uint32_t>(kCodeBoxWords), 128};
      if (make_tmap(&t1, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, train, cdims, cstr, cbox, CU_TENSOR_MAP_SWIZZLE_128B))
        return cudaErrorInvalidValue;
    }
  } else {
    __nv_bfloat16* hi = static_cast<__nv_bfloat16*>(ws);
    __nv_bfloat16* lo = hi + static_cast<size_t>(Q) * D;
    dim3 eg(std::max(1, std::min((D + 255) / 256, 64)), Q);
    k_split_queries<<<eg, 256, 0, st>>>(static_cast<const float*>(query), ldq, D, hi, lo);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const uint64_t dims[2] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Q)};
    const uint64_t strides[1] = {static_cast<uint64_t>(D) * 2};
    const uint32_t box[2] = {64, static_cast<uint32_t>(g.BNq)};
    if (make_tmap(&t0, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, hi, dims, strides, box,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        make_tmap(&t1, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, lo, dims, strides, box,
                  CU_TENSOR_MAP_SWIZZLE_128B))
      return cudaErrorInvalidValue;
  }
  if (topk) {
    // List entries a CTA never fills keep index -1 and are skipped by the merge.
    cudaError_t e =
        cudaMemsetAsync(topk->lsi, 0xFF, static_cast<size_t>(grid) * Q * topk->K * sizeof(int), st);
    if (e != cudaSuccess) return e;
    e = cudaMemsetAsync(topk->gtau, 0, static_cast<size_t>(Q) * sizeof(unsigned), st);  // key 0: none yet
    if (e != cudaSuccess) return e;
    e = dispatch_tc<true>(mode, c, t0, t1, g, grid, st);
    if (e != cudaSuccess) return e;
    return launch_topk_merge(topk->lst, topk->lsi, grid, Q, topk->K, topk->out_s, topk->ld_os,
                             topk->out_i, topk->ld_oi, st);
  }
  return dispatch_tc<false>(mode, c, t0, t1, g, grid, st);
}
