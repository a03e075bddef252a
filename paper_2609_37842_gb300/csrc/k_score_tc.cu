// Scoring on the tensor cores (Sec. 3.3 Eq. onebit_influence; App. B.3 scan),
// in two modes and with two outputs.
//
// CODES: both sides one-bit. For module u the +-1 inner product d_u = <b_q, b_i>
//   is an integer with |d_u| <= k_u. Both sides are expanded to e4m3 bytes
//   (+1 = 0x38, -1 = 0xB8, exact) and multiplied with tcgen05.mma kind::f8f6f4
//   into fp32 TMEM: every partial sum is an integer far below 2^24, so d_u is
//   exact. The epilogue dequantises in the same fixed fp32 order as the
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
// are staged 32 query columns at a time in shared memory and the thread that
// owns a query column merges them into that query's sorted list (score
// descending, equal scores by lower stored index). A CTA's lists cover the
// stored rows of its tiles and go to global memory when the CTA moves to the
// next query tile; a separate kernel merges the per-CTA lists. The Q x N
// matrix never reaches HBM.
//
// Tiles: 128 stored rows (MMA M, operand A) x BNq <= 128 queries (MMA N,
// operand B). Queries are prepared once per call in the workspace (e4m3 bytes,
// or bf16 hi and lo rows) and fetched by TMA; stored rows are expanded from
// their bits into shared memory (128-byte swizzled rows) by four warps, so the
// store is read from HBM as bits. Tiles run query-tile-major: one query tile
// stays in L2 while the stored codes stream past it.
//
// Warps: 0-3 expand stored rows (warp 0 lane 0 also issues the query TMA),
// 4-7 dequantise (TMEM lane quarters 0-3; in TOPK, thread t also owns query
// column t), 8 owns TMEM and issues the MMAs. TMEM: two 128-column d_u
// buffers (module u+1 accumulates while module u is dequantised) and a
// 128-column running score.
#include <cuda_bf16.h>

#include <algorithm>
#include <cmath>

#include "eogp_dev.cuh"
#include "eogp_internal.h"
#include "topk_dev.cuh"

using namespace eogp;

namespace {

constexpr int kMaxMods = 1024;
constexpr int kThreadsTc = 288;
constexpr uint32_t kAB = 16384u;  // 128 rows x 128 bytes
constexpr int kTbStride = 129;    // staged column stride (floats): conflict-free both ways

struct ScoreTcArgs {
  int N, Q, U, D, BNq, n_it, n_tiles, ldt, ldts, ldqs, ldo, K;
  const uint32_t* train;
  const float* ts;
  const float* qs;
  float* out;
  float* lst;  // TOPK: per-CTA lists [gridDim.x][Q][K]
  int* lsi;
  unsigned* status;
  int k[kMaxMods];     // bits per module
};

template <int MODE>
struct TcMode;
template <>
struct TcMode<EOGP_SCORE_CODES> {
  static constexpr int kBits = 128;  // code bits per pipeline stage
  static constexpr int kQBoxes = 1;  // query operand tiles per stage
  using Bits = uint4;                // one stage of one stored row
};
template <>
struct TcMode<EOGP_SCORE_PAPER> {
  static constexpr int kBits = 64;
  static constexpr int kQBoxes = 2;  // hi, lo
  using Bits = uint2;
};

template <int MODE, bool TOPK>
constexpr int tc_stages() {
  return (MODE == EOGP_SCORE_PAPER && TOPK) ? 3 : 4;
}

template <int MODE>
constexpr uint32_t tc_stage_bytes() {
  return kAB * (1 + TcMode<MODE>::kQBoxes);
}

// Shared-memory carve-up (byte offsets after 1024-byte alignment).
struct TcSmem {
  uint32_t sq, bars, tb, lists, total;
};
template <int MODE, bool TOPK>
__host__ __device__ inline TcSmem tc_smem_layout(int BNq, int K) {
  constexpr int S = tc_stages<MODE, TOPK>();
  TcSmem l;
  l.sq = S * tc_stage_bytes<MODE>();
  l.bars = l.sq + 128 * 4;
  l.tb = l.bars + (2 * S + 4) * 8 + 16;
  l.lists = l.tb + (TOPK ? 32 * kTbStride * 4 : 0);
  l.total = l.lists + (TOPK ? static_cast<uint32_t>(BNq) * K * 8 : 0);
  return l;
}

// 8 code bits -> 8 e4m3 bytes (bit j -> byte j: +1 if set, -1 if clear).
__device__ __forceinline__ uint64_t expand8(uint32_t v) {
  uint64_t x = (static_cast<uint64_t>(v & 0xFFu) * 0x0101010101010101ull) & 0x8040201008040201ull;
  x = (x + 0x7F7F7F7F7F7F7F7Full) & 0x8080808080808080ull;  // 0x80 where the bit is set
  return 0xB8B8B8B8B8B8B8B8ull ^ x;
}

// 4 code bits -> 4 bf16 values (bit j -> element j: +1 = 0x3F80 if set, -1 = 0xBF80 if
// clear). Each 16-bit lane isolates its bit at position j, then adding 0x8000 - 2^j
// carries into bit 15 exactly when the bit is set.
__device__ __forceinline__ uint64_t expand4_bf16(uint32_t v) {
  uint64_t x = (static_cast<uint64_t>(v & 0xFu) * 0x0001000100010001ull) & 0x0008000400020001ull;
  x = (x + 0x7FF87FFC7FFE7FFFull) & 0x8000800080008000ull;
  return 0xBF80BF80BF80BF80ull ^ x;
}

// One stage of one stored row -> its 128-byte swizzled shared-memory row
// (16-byte chunk c goes to position c ^ (row & 7)).
__device__ __forceinline__ void expand_stage(uint8_t* dst, int sw, uint4 bits) {  // 128 bits -> e4m3
  const uint32_t wv[4] = {bits.x, bits.y, bits.z, bits.w};
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const uint32_t h = wv[c >> 1] >> ((c & 1) * 16);
    const uint64_t lo = expand8(h), hi = expand8(h >> 8);
    *reinterpret_cast<uint4*>(dst + ((c ^ sw) << 4)) =
        make_uint4(static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32), static_cast<uint32_t>(hi),
                   static_cast<uint32_t>(hi >> 32));
  }
}
__device__ __forceinline__ void expand_stage(uint8_t* dst, int sw, uint2 bits) {  // 64 bits -> bf16
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    const uint32_t h = (c < 4 ? bits.x : bits.y) >> ((c & 3) * 8);
    const uint64_t lo = expand4_bf16(h), hi = expand4_bf16(h >> 4);
    *reinterpret_cast<uint4*>(dst + ((c ^ sw) << 4)) =
        make_uint4(static_cast<uint32_t>(lo), static_cast<uint32_t>(lo >> 32), static_cast<uint32_t>(hi),
                   static_cast<uint32_t>(hi >> 32));
  }
}

// Tiles of a CTA. Dense output: strided over the grid, so all CTAs work on the
// same query tile at a time. Ranking: a contiguous run of tiles, so a CTA
// ranks long runs of stored rows of one query tile (fewer fresh lists).
template <bool TOPK>
__device__ __forceinline__ int tile_begin(const ScoreTcArgs& g) {
  return TOPK ? static_cast<int>(static_cast<long long>(g.n_tiles) * blockIdx.x / gridDim.x) : blockIdx.x;
}
template <bool TOPK>
__device__ __forceinline__ int tile_end(const ScoreTcArgs& g) {
  return TOPK ? static_cast<int>(static_cast<long long>(g.n_tiles) * (blockIdx.x + 1) / gridDim.x) : g.n_tiles;
}
template <bool TOPK>
__device__ __forceinline__ int tile_step() {
  return TOPK ? 1 : gridDim.x;
}

template <int MODE, bool TOPK>
__global__ void __launch_bounds__(kThreadsTc, 1)
    k_score_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmQlo,
               const __grid_constant__ ScoreTcArgs g) {
  constexpr int S = tc_stages<MODE, TOPK>();
  constexpr uint32_t kStage = tc_stage_bytes<MODE>();
  constexpr int kBits = TcMode<MODE>::kBits;
  constexpr int kG = 8;  // stages of code bits prefetched at a time
  using StageBits = typename TcMode<MODE>::Bits;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const TcSmem L = tc_smem_layout<MODE, TOPK>(g.BNq, g.K);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* sq = reinterpret_cast<float*>(smem + L.sq);  // [128] query scales of module u (CODES)
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty = full + S;
  uint64_t* dfull = empty + S;
  uint64_t* dempty = dfull + 2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(dempty + 2);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    if (MODE == EOGP_SCORE_PAPER) tma_prefetch_desc(&tmQlo);
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 5);  // TMA transaction arrive + 4 expander warps
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&dfull[b], 1);
      mbar_init(&dempty[b], 4);
    }
    fence_barrier_init();
  }
  if (warp == 8) tmem_alloc(tslot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp < 4) {
    // ---------------------------------------------------------- expanders
    // A stored row's modules are back to back, so pipeline stage j of a tile
    // reads bits [j kBits, (j+1) kBits) of the row and query columns from
    // j kBits on. The bits of the next kG stages are loaded into registers
    // while the current kG stages are expanded, hiding the HBM latency.
    const int r = threadIdx.x;  // stored row within the tile
    const uint32_t row_off = static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128);
    const int nst = g.D / kBits;
    uint32_t it = 0;
    bool ok = true;
    for (int tile = tile_begin<TOPK>(g), tstep = tile_step<TOPK>(), tend = tile_end<TOPK>(g);
         tile < tend && ok; tile += tstep) {
      const int qt = tile / g.n_it, ib = tile % g.n_it;
      const int i0 = ib * 128, q0 = qt * g.BNq;
      const bool rv = i0 + r < g.N;
      const StageBits* brow =
          reinterpret_cast<const StageBits*>(g.train + static_cast<size_t>(rv ? i0 + r : 0) * g.ldt);
      StageBits cur[kG], nxt[kG];
#pragma unroll
      for (int jj = 0; jj < kG; ++jj) cur[jj] = (rv && jj < nst) ? __ldg(brow + jj) : StageBits{};
      for (int j0 = 0; j0 < nst && ok; j0 += kG) {
#pragma unroll
        for (int jj = 0; jj < kG; ++jj)
          nxt[jj] = (rv && j0 + kG + jj < nst) ? __ldg(brow + j0 + kG + jj) : StageBits{};
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
                tma_load_2d(st + kAB, &tmQ, j * kBits, q0, &full[s]);
                if (MODE == EOGP_SCORE_PAPER) tma_load_2d(st + 2 * kAB, &tmQlo, j * kBits, q0, &full[s]);
              }
              expand_stage(st + row_off, r & 7, cur[jj]);
              fence_proxy_async_smem();
              __syncwarp();
              if (lane == 0) mbar_arrive(&full[s]);
            }
          }
        }
#pragma unroll
        for (int jj = 0; jj < kG; ++jj) cur[jj] = nxt[jj];
      }
    }
  } else if (warp < 8) {
    // ---------------------------------------------------------- dequantise
    const int q4 = warp & 3;
    const int ep = threadIdx.x - 128;  // TMEM lane (stored row in the tile); TOPK: query column
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    float* tb = reinterpret_cast<float*>(smem + L.tb);
    float* ls = reinterpret_cast<float*>(smem + L.lists) + static_cast<size_t>(ep) * g.K;
    int* li = reinterpret_cast<int*>(smem + L.lists + static_cast<size_t>(g.BNq) * g.K * 4) +
              static_cast<size_t>(ep) * g.K;
    int seg_qt = -1;
    TopkState tk;
    topk_reset(tk);
    auto flush = [&]() {
      const int q = seg_qt * g.BNq + ep;
      if (ep < g.BNq && q < g.Q) {
        const size_t o = (static_cast<size_t>(blockIdx.x) * g.Q + q) * g.K;
        topk_write(ls, li, g.K, tk, g.lst + o, g.lsi + o);
      }
    };
    uint32_t gm = 0;
    bool ok = true;
    for (int tile = tile_begin<TOPK>(g), tstep = tile_step<TOPK>(), tend = tile_end<TOPK>(g);
         tile < tend && ok; tile += tstep) {
      const int qt = tile / g.n_it, ib = tile % g.n_it;
      const int i0 = ib * 128, q0 = qt * g.BNq;
      const int row = i0 + ep;
      if (TOPK && qt != seg_qt) {
        if (seg_qt >= 0) flush();
        seg_qt = qt;
        topk_reset(tk);
      }
      for (int u = 0; u < g.U; ++u, ++gm) {
        const int buf = static_cast<int>(gm & 1u);
        const uint32_t dph = (gm >> 1) & 1u;
        if (MODE == EOGP_SCORE_CODES) {
          named_bar_sync(1, 128);  // previous module's readers of sq are done
          if (ep < g.BNq) sq[ep] = q0 + ep < g.Q ? g.qs[static_cast<size_t>(q0 + ep) * g.ldqs + u] : 0.f;
          named_bar_sync(1, 128);
        }
        uint32_t w_ok = 1;
        if (lane == 0) w_ok = mbar_wait(&dfull[buf], dph, g.status) ? 1u : 0u;
        w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
        __syncwarp();
        tc_fence_after();
        if (!__syncthreads_and_named(w_ok)) {
          ok = false;
          break;
        }
        const float si = row < g.N ? g.ts[static_cast<size_t>(row) * g.ldts + u] : 0.f;
        const bool last = u + 1 == g.U;
        for (int c0 = 0; c0 < g.BNq; c0 += 32) {
          float d[32], a[32];
          tmem_ld32(tmem + lane_base + buf * 128u + c0, d);
          if (u == 0) {
#pragma unroll
            for (int j = 0; j < 32; ++j) a[j] = 0.f;
          } else {
            tmem_ld32(tmem + lane_base + 256u + c0, a);
          }
          if (MODE == EOGP_SCORE_CODES) {
#pragma unroll
            for (int j = 0; j < 32; ++j) a[j] = __fadd_rn(a[j], __fmul_rn(__fmul_rn(sq[c0 + j], si), d[j]));
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) a[j] = __fadd_rn(a[j], __fmul_rn(si, d[j]));
          }
          if (!last || TOPK) {
            tmem_st32(tmem + lane_base + 256u + c0, a);
          } else if (row < g.N) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dempty[buf]);  // D buffer free: the MMAs run on
        if (TOPK && last) {
          // Rank the finished tile from the running-score columns, 32 query columns at
          // a time: staged column-major, then the warp owning them offers them to its lists.
          for (int c0 = 0; c0 < g.BNq; c0 += 32) {
            float a[32];
            tmem_ld32(tmem + lane_base + 256u + c0, a);
#pragma unroll
            for (int j = 0; j < 32; ++j) tb[j * kTbStride + ep] = a[j];
            named_bar_sync(3, 128);
            if ((ep >> 5) == (c0 >> 5) && q0 + ep < g.Q)
              topk_scan(tb + lane * kTbStride, min(128, g.N - i0), i0, ls, li, g.K, tk);
            named_bar_sync(3, 128);
          }
        }
      }
    }
    if (TOPK && seg_qt >= 0) flush();
  } else {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc =
          MODE == EOGP_SCORE_CODES ? idesc_e4m3_f32(128, g.BNq) : idesc_bf16_f32(128, g.BNq, 0, 0);
      uint32_t it = 0, gm = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK>(g), tstep = tile_step<TOPK>(), tend = tile_end<TOPK>(g);
         tile < tend && ok; tile += tstep) {
        for (int u = 0; u < g.U && ok; ++u, ++gm) {
          const int buf = static_cast<int>(gm & 1u);
          const uint32_t dph = (gm >> 1) & 1u;
          if (!mbar_wait(&dempty[buf], dph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + buf * 128u;
          const int nkb = g.k[u] / kBits;
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const int s = static_cast<int>(it % S);
            const uint32_t ph = (it / S) & 1u;
            if (!mbar_wait(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + static_cast<size_t>(s) * kStage);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint64_t ad = sdesc_sw128(sa + kk * 32, 16, 1024);
              const uint32_t acc = (kb | kk) != 0 ? 1u : 0u;
              if (MODE == EOGP_SCORE_CODES) {
                tc_mma_f8(d, ad, sdesc_sw128(sa + kAB + kk * 32, 16, 1024), idesc, acc);
              } else {
                tc_mma_f16(d, ad, sdesc_sw128(sa + kAB + kk * 32, 16, 1024), idesc, acc);
                tc_mma_f16(d, ad, sdesc_sw128(sa + 2 * kAB + kk * 32, 16, 1024), idesc, 1u);
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
  if (warp == 8) tmem_dealloc(tmem, 512);
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

int bnq_for(int Q) { return std::min(128, (Q + 31) / 32 * 32); }

template <int MODE, bool TOPK>
cudaError_t launch_tc_kernel(const CUtensorMap& t0, const CUtensorMap& t1, const ScoreTcArgs& g,
                             int grid, cudaStream_t st) {
  const size_t smem = 1024 + tc_smem_layout<MODE, TOPK>(g.BNq, g.K).total;
  cudaError_t e = cudaFuncSetAttribute(k_score_tc<MODE, TOPK>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  k_score_tc<MODE, TOPK><<<grid, kThreadsTc, smem, st>>>(t0, t1, g);
  return cudaGetLastError();
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

size_t score_tc_ws_bytes(int mode, const int* ks, int U, int Q) {
  long long D = 0;
  for (int u = 0; u < U; ++u) D += ks[u];
  const size_t per = mode == EOGP_SCORE_PAPER ? 4 : 1;  // bf16 hi + lo, or e4m3
  return (static_cast<size_t>(Q) * D * per + 255) & ~size_t(255);
}

int score_tc_grid(int N, int Q, int num_sms) {
  const long long tiles =
      static_cast<long long>((N + 127) / 128) * ((Q + bnq_for(Q) - 1) / bnq_for(Q));
  return static_cast<int>(std::max<long long>(1, std::min<long long>(tiles, std::max(1, num_sms))));
}

bool score_tc_topk_fits(int mode, int Q, int K) {
  if (K < 1 || K > kTopKMax) return false;
  const size_t need = 1024 + (mode == EOGP_SCORE_PAPER
                                  ? tc_smem_layout<EOGP_SCORE_PAPER, true>(bnq_for(Q), K).total
                                  : tc_smem_layout<EOGP_SCORE_CODES, true>(bnq_for(Q), K).total);
  return need <= 232448;
}

cudaError_t launch_score_tc(int mode, const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                            const int* ks, int U, const void* query, int ldq, const float* qs,
                            int ldqs, int Q, float* out, int ldo, const TcTopK* topk, void* ws,
                            int num_sms, unsigned* status, cudaStream_t st) {
  if (N <= 0 || Q <= 0) return cudaSuccess;
  ScoreTcArgs g;  // ~4 KB parameter block, copied at launch
  g.N = N;
  g.Q = Q;
  g.U = U;
  g.BNq = bnq_for(Q);
  g.n_it = (N + 127) / 128;
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
  g.status = status;
  int D = 0;
  for (int u = 0; u < U; ++u) {
    g.k[u] = ks[u];
    D += ks[u];
  }
  g.D = D;
  const int grid = score_tc_grid(N, Q, num_sms);
  CUtensorMap t0, t1;
  if (mode == EOGP_SCORE_CODES) {
    uint8_t* qx = static_cast<uint8_t*>(ws);
    dim3 eg(std::max(1, std::min((D / 32 + 255) / 256, 64)), Q);
    k_expand_queries<<<eg, 256, 0, st>>>(static_cast<const uint32_t*>(query), ldq, D, qx);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    const uint64_t dims[2] = {static_cast<uint64_t>(D), static_cast<uint64_t>(Q)};
    const uint64_t strides[1] = {static_cast<uint64_t>(D)};
    const uint32_t box[2] = {128, static_cast<uint32_t>(g.BNq)};
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
    e = mode == EOGP_SCORE_CODES ? launch_tc_kernel<EOGP_SCORE_CODES, true>(t0, t1, g, grid, st)
                                 : launch_tc_kernel<EOGP_SCORE_PAPER, true>(t0, t1, g, grid, st);
    if (e != cudaSuccess) return e;
    return launch_topk_merge(topk->lst, topk->lsi, grid, Q, topk->K, topk->out_s, topk->ld_os,
                             topk->out_i, topk->ld_oi, st);
  }
  return mode == EOGP_SCORE_CODES ? launch_tc_kernel<EOGP_SCORE_CODES, false>(t0, t1, g, grid, st)
                                  : launch_tc_kernel<EOGP_SCORE_PAPER, false>(t0, t1, g, grid, st);
}
