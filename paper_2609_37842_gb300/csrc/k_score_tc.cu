// One-bit scoring on the tensor cores (CODES mode, Sec. 3.3 Eq. onebit_influence
// with both sides one-bit; App. B.3 scan).
//
// For module u the +-1 inner product d_u = <b_q, b_i> is an integer with
// |d_u| <= k_u. Both sides are expanded to e4m3 bytes (+1 = 0x38, -1 = 0xB8,
// exact) and multiplied with tcgen05.mma kind::f8f6f4 into fp32 TMEM: every
// partial sum is an integer far below 2^24, so d_u is exact. The epilogue then
// dequantises in the same fixed fp32 order as the popcount kernels,
//   acc = fl(acc + fl(fl(s_qu * s_iu) * d_u))   in module order,
// keeping acc in TMEM between modules, so scores are bitwise identical to the
// popcount path and to the oracle's float32 evaluation.
//
// Tiles: 128 stored rows (MMA M, operand A) x BNq <= 128 queries (MMA N,
// operand B), K = 128 code bits per pipeline stage. Queries are expanded once
// per call into the workspace and fetched by TMA; stored rows are expanded from
// their bits into shared memory (128-byte swizzled rows) by four warps, so the
// store is read from HBM as bits. Tiles run query-tile-major: one query tile
// stays in L2 while the stored codes stream past it.
//
// Warps: 0-3 expand stored rows (warp 0 lane 0 also issues the query TMA),
// 4-7 dequantise (TMEM lane quarters 0-3), 8 owns TMEM and issues the MMAs.
// TMEM: two 128-column d_u buffers (module u+1 accumulates while module u is
// dequantised) and a 128-column running score.
#include <algorithm>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

using namespace eogp;

namespace {

constexpr int kMaxMods = 1024;
constexpr int kThreadsTc = 288;
constexpr int kStages = 4;
constexpr uint32_t kAB = 16384u;  // 128 rows x 128 bytes

struct ScoreTcArgs {
  int N, Q, U, BNq, n_it, n_tiles, ldt, ldts, ldqs, ldo;
  const uint32_t* train;
  const float* ts;
  const float* qs;
  float* out;
  unsigned* status;
  int k[kMaxMods];     // bits per module (multiple of 128)
  int woff[kMaxMods];  // word offset of module u in a stored row
  int boff[kMaxMods];  // byte offset of module u in an expanded query row
};

// 8 code bits -> 8 e4m3 bytes (bit j -> byte j: +1 if set, -1 if clear).
__device__ __forceinline__ uint64_t expand8(uint32_t v) {
  uint64_t x = (static_cast<uint64_t>(v & 0xFFu) * 0x0101010101010101ull) & 0x8040201008040201ull;
  x = (x + 0x7F7F7F7F7F7F7F7Full) & 0x8080808080808080ull;  // 0x80 where the bit is set
  return 0xB8B8B8B8B8B8B8B8ull ^ x;
}

__global__ void __launch_bounds__(kThreadsTc, 1)
    k_score_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ ScoreTcArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr uint32_t kStage = 2 * kAB;
  float* sq = reinterpret_cast<float*>(smem + kStages * kStage);  // [128] query scales of module u
  uint64_t* full = reinterpret_cast<uint64_t*>(sq + 128);
  uint64_t* empty = full + kStages;
  uint64_t* dfull = empty + kStages;
  uint64_t* dempty = dfull + 2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(dempty + 2);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    for (int s = 0; s < kStages; ++s) {
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
    const int r = threadIdx.x;  // stored row within the tile
    const uint32_t row_off = static_cast<uint32_t>((r >> 3) * 1024 + (r & 7) * 128);
    uint32_t it = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < g.n_tiles && ok; tile += gridDim.x) {
      const int qt = tile / g.n_it, ib = tile % g.n_it;
      const int i0 = ib * 128, q0 = qt * g.BNq;
      const bool rv = i0 + r < g.N;
      const uint32_t* crow = g.train + static_cast<size_t>(rv ? i0 + r : 0) * g.ldt;
      for (int u = 0; u < g.U && ok; ++u) {
        const int nkb = g.k[u] >> 7;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = static_cast<int>(it % kStages);
          const uint32_t ph = (it / kStages) & 1u;
          uint32_t w_ok = 1;
          if (lane == 0) w_ok = mbar_wait(&empty[s], ph ^ 1u, g.status) ? 1u : 0u;
          w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
          if (!w_ok) {
            ok = false;
            break;
          }
          uint8_t* st = smem + static_cast<size_t>(s) * kStage;
          if (warp == 0 && lane == 0) {
            mbar_arrive_expect_tx(&full[s], static_cast<uint32_t>(g.BNq) * 128u);
            tma_load_2d(st + kAB, &tmQ, g.boff[u] + kb * 128, q0, &full[s]);
          }
          uint4 bits = make_uint4(0, 0, 0, 0);
          if (rv) bits = __ldg(reinterpret_cast<const uint4*>(crow + g.woff[u] + kb * 4));
          const uint32_t wv[4] = {bits.x, bits.y, bits.z, bits.w};
#pragma unroll
          for (int c = 0; c < 8; ++c) {  // 16 bits -> 16 bytes per swizzled 16-byte chunk
            const uint32_t h = wv[c >> 1] >> ((c & 1) * 16);
            const uint64_t lo = expand8(h), hi = expand8(h >> 8);
            uint4 v;
            v.x = static_cast<uint32_t>(lo);
            v.y = static_cast<uint32_t>(lo >> 32);
            v.z = static_cast<uint32_t>(hi);
            v.w = static_cast<uint32_t>(hi >> 32);
            *reinterpret_cast<uint4*>(st + row_off + ((c ^ (r & 7)) << 4)) = v;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(&full[s]);
        }
      }
    }
  } else if (warp < 8) {
    // ---------------------------------------------------------- dequantise
    const int q4 = warp & 3;
    const int ep = threadIdx.x - 128;
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    uint32_t gm = 0;
    bool ok = true;
    for (int tile = blockIdx.x; tile < g.n_tiles && ok; tile += gridDim.x) {
      const int qt = tile / g.n_it, ib = tile % g.n_it;
      const int i0 = ib * 128, q0 = qt * g.BNq;
      const int row = i0 + q4 * 32 + lane;
      for (int u = 0; u < g.U; ++u, ++gm) {
        const int buf = static_cast<int>(gm & 1u);
        const uint32_t dph = (gm >> 1) & 1u;
        named_bar_sync(1, 128);  // previous module's readers of sq are done
        if (ep < g.BNq) sq[ep] = q0 + ep < g.Q ? g.qs[static_cast<size_t>(q0 + ep) * g.ldqs + u] : 0.f;
        named_bar_sync(1, 128);
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
        for (int c0 = 0; c0 < g.BNq; c0 += 32) {
          float d[32], a[32];
          tmem_ld32(tmem + lane_base + buf * 128u + c0, d);
          if (u == 0) {
#pragma unroll
            for (int j = 0; j < 32; ++j) a[j] = 0.f;
          } else {
            tmem_ld32(tmem + lane_base + 256u + c0, a);
          }
#pragma unroll
          for (int j = 0; j < 32; ++j) a[j] = __fadd_rn(a[j], __fmul_rn(__fmul_rn(sq[c0 + j], si), d[j]));
          if (u + 1 < g.U) {
            tmem_st32(tmem + lane_base + 256u + c0, a);
          } else if (row < g.N) {
#pragma unroll 8
            for (int j = 0; j < 32; ++j)
              if (q0 + c0 + j < g.Q) g.out[static_cast<size_t>(q0 + c0 + j) * g.ldo + row] = a[j];
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dempty[buf]);
      }
    }
  } else {
    // ---------------------------------------------------------- MMA issuer
    if (lane == 0) {
      const uint32_t idesc = idesc_e4m3_f32(128, g.BNq);
      uint32_t it = 0, gm = 0;
      bool ok = true;
      for (int tile = blockIdx.x; tile < g.n_tiles && ok; tile += gridDim.x) {
        for (int u = 0; u < g.U && ok; ++u, ++gm) {
          const int buf = static_cast<int>(gm & 1u);
          const uint32_t dph = (gm >> 1) & 1u;
          if (!mbar_wait(&dempty[buf], dph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + buf * 128u;
          const int nkb = g.k[u] >> 7;
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const int s = static_cast<int>(it % kStages);
            const uint32_t ph = (it / kStages) & 1u;
            if (!mbar_wait(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + static_cast<size_t>(s) * kStage);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_f8(d, sdesc_sw128(sa + kk * 32, 16, 1024), sdesc_sw128(sa + kAB + kk * 32, 16, 1024),
                        idesc, (kb | kk) != 0 ? 1u : 0u);
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

// Query codes -> e4m3 bytes: out[q][boff_u + c] = +1 / -1 for bit c of module u.
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

size_t score_tc_smem() {
  return 1024 + kStages * 2 * kAB + 128 * 4 + (2 * kStages + 4) * 8 + 16;
}

}  // namespace

bool score_tc_supported(const int* ks, int U, int Q) {
  if (Q < 64 || Q > 65535 || U < 1 || U > kMaxMods) return false;
  for (int u = 0; u < U; ++u)
    if (ks[u] <= 0 || ks[u] % 128) return false;
  return true;
}

size_t score_tc_ws_bytes(const int* ks, int U, int Q) {
  long long D = 0;
  for (int u = 0; u < U; ++u) D += ks[u];
  return (static_cast<size_t>(Q) * D + 255) & ~size_t(255);
}

cudaError_t launch_score_tc(const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                            const int* ks, int U, const uint32_t* query, int ldq, const float* qs,
                            int ldqs, int Q, float* out, int ldo, void* ws, int num_sms,
                            unsigned* status, cudaStream_t st) {
  if (N <= 0 || Q <= 0) return cudaSuccess;
  ScoreTcArgs g;  // ~12 KB parameter block, copied at launch
  g.N = N;
  g.Q = Q;
  g.U = U;
  g.BNq = std::min(128, (Q + 31) / 32 * 32);
  g.n_it = (N + 127) / 128;
  g.n_tiles = g.n_it * ((Q + g.BNq - 1) / g.BNq);
  g.ldt = ldt;
  g.ldts = ldts;
  g.ldqs = ldqs;
  g.ldo = ldo;
  g.train = train;
  g.ts = ts;
  g.qs = qs;
  g.out = out;
  g.status = status;
  int wo = 0, bo = 0;
  for (int u = 0; u < U; ++u) {
    g.k[u] = ks[u];
    g.woff[u] = wo;
    g.boff[u] = bo;
    wo += ks[u] / 32;
    bo += ks[u];
  }
  const int row_bytes = bo;
  uint8_t* qx = static_cast<uint8_t*>(ws);
  {
    dim3 grid(std::max(1, std::min((row_bytes / 32 + 255) / 256, 64)), Q);
    k_expand_queries<<<grid, 256, 0, st>>>(query, ldq, row_bytes, qx);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  CUtensorMap tq;
  const uint64_t dims[2] = {static_cast<uint64_t>(row_bytes), static_cast<uint64_t>(Q)};
  const uint64_t strides[1] = {static_cast<uint64_t>(row_bytes)};
  const uint32_t box[2] = {128, static_cast<uint32_t>(g.BNq)};
  if (make_tmap(&tq, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, qx, dims, strides, box,
                CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  const size_t smem = score_tc_smem();
  cudaError_t e = cudaFuncSetAttribute(k_score_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int grid = std::min(g.n_tiles, std::max(1, num_sms));
  k_score_tc<<<grid, kThreadsTc, smem, st>>>(tq, g);
  return cudaGetLastError();
}
