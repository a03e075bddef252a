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

#include "score_tc.cuh"

using namespace eogp;
using namespace eogp::sc;

namespace {

constexpr int kThreadsTc = (kExpWarps + 4 + 1) * 32;  // + 4 dequantise warps + 1 MMA warp
constexpr uint32_t kAB = 16384u;                    // 128 rows x 128 bytes

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
template <int MODE, bool TOPK, int BN, bool AT>
constexpr int tc_stages() {
  return AT ? (BN == 256 ? 6 : 8) : ((MODE == EOGP_SCORE_CODES && BN == 128) ? 6 : 4);
}

// 128-query tiles with operand A in TMEM keep the running score in shared
// memory (row stride kAccLd floats: conflict-free float4 rows), leaving 256
// TMEM columns for eight A slots next to the two d_u accumulators.
template <int BN, bool AT>
constexpr bool tc_acc_smem() {
  return AT && BN == 128;
}

// Stages the expanders fill per synchronisation round (one wait, fence and
// arrive round): two with six stages, so that the MMAs always have at least
// four stages to work on, else one.
template <int MODE, bool TOPK, int BN, bool AT>
constexpr int tc_group() {
  return tc_stages<MODE, TOPK, BN, AT>() >= 6 ? 2 : 1;
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

// Shared-memory carve-up (byte offsets after 1024-byte alignment).
template <int MODE, bool TOPK, int BN, bool AT>
__host__ __device__ inline TcSmem tc_smem_layout(int BNq, int K) {
  constexpr int S = tc_stages<MODE, TOPK, BN, AT>();
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

template <int MODE, bool TOPK, int BN, bool AT>
__global__ void __launch_bounds__(kThreadsTc, 1)
    k_score_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQlo,
               const __grid_constant__ ScoreTcArgs g) {
  static_assert(!AT || MODE == EOGP_SCORE_CODES, "operand A in TMEM is the one-bit path");
  constexpr int S = tc_stages<MODE, TOPK, BN, AT>();
  constexpr uint32_t kStage = tc_stage_bytes<MODE, BN, AT>();
  constexpr uint32_t kBOff = tc_b_offset<AT>();
  // code bits per pipeline stage, and the query operand's TMA x coordinate per
  // stage (elements of its tensor map: e4m3 bytes or bf16 values)
  constexpr int kBits = TcMode<MODE>::kBits;
  constexpr int kQx = kBits;
  constexpr int ND = tc_dbufs<BN, AT>();
  using HalfBits = typename TcMode<MODE>::HalfBits;
  constexpr int kG = 8;  // stages of code bits prefetched at a time
  constexpr int kP = tc_group<MODE, TOPK, BN, AT>();
  constexpr bool kAccS = tc_acc_smem<BN, AT>();
  static_assert(kG % kP == 0, "prefetch groups hold whole expansion rounds");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const TcSmem L = tc_smem_layout<MODE, TOPK, BN, AT>(g.BNq, g.K);
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
      const uint32_t idesc =
          MODE == EOGP_SCORE_CODES ? idesc_e4m3_f32(128, g.BNq) : idesc_bf16_f32(128, g.BNq, 0, 0);
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
              if constexpr (AT) {
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

template <int MODE, bool TOPK, int BN, bool AT = false>
size_t tc_smem_need(int BNq, int K) {
  return 1024 + tc_smem_layout<MODE, TOPK, BN, AT>(BNq, K).total;
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

// The kernel a call runs and its tiling.
struct TcCfg {
  bool pair;  // k_score_pair (one-bit, e2m1) or k_score_tc
  bool f4;    // e2m1 operands
  int BN, BNq, rows;  // queries per tile (template, actual), stored rows per tile
  int G;      // pair kernel: 256-bit stages per pipeline group
};
TcCfg tc_cfg(int mode, const int* ks, int U, int Q, int K) {
  TcCfg c;
  c.f4 = tc_f4(mode, ks, U);
  c.pair = c.f4;
  c.BN = c.pair ? pr_bn(U, Q) : tc_bn(mode, U, Q, K);
  c.BNq = bnq_for(Q, c.BN);
  c.rows = c.pair ? 256 : 128;
  // stages per group of the pair kernel (groups never straddle modules): four
  // with 64-query tiles when every module is a multiple of 1024 bits, two when
  // a multiple of 512, else one
  c.G = c.BN == 64 ? 4 : 2;
  for (int u = 0; u < U && c.pair; ++u)
    while (c.G > 1 && ks[u] % (256 * c.G)) c.G /= 2;
  return c;
}

// CTAs of a call: one per SM at most (one CTA, or one pair per two SMs).
int tc_grid(const TcCfg& c, int N, int Q, int num_sms) {
  const long long tiles = static_cast<long long>((N + c.rows - 1) / c.rows) * ((Q + c.BNq - 1) / c.BNq);
  if (c.pair) return 2 * static_cast<int>(std::max<long long>(1, std::min<long long>(tiles, pair_cluster_cap(num_sms))));
  return static_cast<int>(std::max<long long>(1, std::min<long long>(tiles, std::max(1, num_sms))));
}

template <int MODE, bool TOPK, int BN, bool AT>
cudaError_t launch_tc_kernel(const CUtensorMap& t0, const CUtensorMap& t1, const ScoreTcArgs& g,
                             int grid, cudaStream_t st) {
  const size_t smem = tc_smem_need<MODE, TOPK, BN, AT>(g.BNq, g.K);
  cudaError_t e = cudaFuncSetAttribute(k_score_tc<MODE, TOPK, BN, AT>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  k_score_tc<MODE, TOPK, BN, AT><<<grid, kThreadsTc, smem, st>>>(t0, t1, g);
  return cudaGetLastError();
}

template <bool TOPK>
cudaError_t dispatch_tc(int mode, const TcCfg& c, const CUtensorMap& t0, const CUtensorMap& t1,
                        const ScoreTcArgs& g, int grid, cudaStream_t st) {
  if (c.BN == 256 && g.U != 1) return cudaErrorInvalidValue;  // 256-query tiles keep no running score
  if (mode == EOGP_SCORE_PAPER) return launch_tc_kernel<EOGP_SCORE_PAPER, TOPK, 128, false>(t0, t1, g, grid, st);
  if (c.pair) return launch_pair(c.BN, c.G, TOPK, t0, g, grid, st);
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
    need = pair_smem_need(c.BN, c.G, true);
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
  g.kuni = ks[0];
  for (int u = 1; u < U; ++u)
    if (ks[u] != ks[0]) g.kuni = 0;
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
