// tcgen05 tensor-core kernels (bf16 in, fp32 accumulate in TMEM), fed by TMA.
//
// k_tc_gemm -- D[M x N] = sum_a X_a[M x K] W[N x K]^T, both operands K-major.
//   Used twice per module for the Kronecker rotations of Sec. 2.2
//   (A~ = A V_A[C]^T over the retained columns, S~ = S V_S[R]^T over the
//   retained rows; M = B*T tokens) and once for the second-stage projection
//   x = P^T z (Eq. second_stage; M = B examples, N = k, K = m) where z enters as
//   a bf16 hi + lo pair (two A operands into the same accumulator).
//   Epilogue 0 writes D as a bf16 hi/lo pair (hi = rn(D), lo = rn(D - hi)), so
//   the next contraction sees D to ~16 significant bits; epilogue 1 writes an
//   fp32 partial slab per K split.
//
// k_tc_contract -- for example b and one active 128 x 128 tile (R block rt,
//   C block ct) of the retained block: G~_b[tile] = sum_t S~_b[t, rows]^T
//   A~_b[t, cols] with K = tokens, both operands MN-major (token rows).
//   hi*hi + hi*lo + lo*hi: three MMAs per K step. The epilogue stages the fp32
//   tile in shared memory and gathers the retained entries of the tile,
//   scaled by (Lambda + lambda)^{-1/2} (Eq. first_stage), into z.
//
// Warp roles (192 threads): warp 0 issues TMA, warp 1 owns TMEM and issues
// MMAs (one lane), warps 2-5 run the epilogue (warp w reads TMEM lanes
// 32*(w%4)..+31). Every mbarrier wait is bounded (eogp_dev.cuh); after a
// timeout every role falls through to the common exit, which frees TMEM.
#include <algorithm>
#include <cstdlib>
#include <mutex>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

using namespace eogp;

namespace {

constexpr int kThreads = 192;
constexpr uint32_t kABytes = 128u * 64u * 2u;  // 128 rows x 64 bf16 (one 128-byte swizzle row each)

struct GemmArgs {
  int M, N, K, BN, stages, nA, nW, kbps, epi, ldo;
  float alpha;  // epilogue 1: output scale
  void* out0;
  void* out1;
  size_t slab;
  unsigned* status;
};

__device__ __forceinline__ uint32_t pack_bf16x2(__nv_bfloat16 a, __nv_bfloat16 b) {
  return static_cast<uint32_t>(__bfloat16_as_ushort(a)) |
         (static_cast<uint32_t>(__bfloat16_as_ushort(b)) << 16);
}

__device__ __forceinline__ uint32_t tmem_cols_for(int n) {
  return n <= 32 ? 32u : n <= 64 ? 64u : n <= 128 ? 128u : 256u;
}

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmX0, const __grid_constant__ CUtensorMap tmX1,
              const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmW1,
              const GemmArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t b_bytes = static_cast<uint32_t>(g.BN) * 128u;
  const uint32_t stage_bytes = static_cast<uint32_t>(g.nA) * kABytes + static_cast<uint32_t>(g.nW) * b_bytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(g.stages) * stage_bytes);
  uint64_t* empty = full + g.stages;
  uint64_t* done = empty + g.stages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  const uint32_t tmem_cols = tmem_cols_for(g.BN);

  const int n0 = blockIdx.x * g.BN, m0 = blockIdx.y * 128;
  const int nkb_total = (g.K + 63) / 64;
  const int kb0 = blockIdx.z * g.kbps;
  const int nkb = max(0, min(g.kbps, nkb_total - kb0));

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmX0);
    if (g.nA > 1) tma_prefetch_desc(&tmX1);
    tma_prefetch_desc(&tmW);
    if (g.nW > 1) tma_prefetch_desc(&tmW1);
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, tmem_cols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      int rs = 0;
      uint32_t rph = 0;
      for (int i = 0; i < nkb; ++i) {
        const int s = rs;
        const uint32_t ph = rph;
        if (++rs == g.stages) {
          rs = 0;
          rph ^= 1u;
        }
        if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) break;
        uint8_t* st = smem + static_cast<size_t>(s) * stage_bytes;
        mbar_arrive_expect_tx(&full[s], stage_bytes);
        const int kx = (kb0 + i) * 64;
        tma_load_2d(st, &tmX0, kx, m0, &full[s]);
        if (g.nA > 1) tma_load_2d(st + kABytes, &tmX1, kx, m0, &full[s]);
        tma_load_2d(st + g.nA * kABytes, &tmW, kx, n0, &full[s]);
        if (g.nW > 1) tma_load_2d(st + g.nA * kABytes + b_bytes, &tmW1, kx, n0, &full[s]);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, g.BN, 0, 0);
      int rs = 0;
      uint32_t rph = 0;
      for (int i = 0; i < nkb; ++i) {
        const int s = rs;
        const uint32_t ph = rph;
        if (++rs == g.stages) {
          rs = 0;
          rph ^= 1u;
        }
        if (!mbar_wait(&full[s], ph, g.status)) break;
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
        const uint32_t sb = sa + g.nA * kABytes;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
          for (int w = 0; w < g.nW; ++w) {
            const uint64_t bd = sdesc_sw128(sb + w * b_bytes + kk * 32, 16, 1024);
            for (int a = 0; a < g.nA; ++a) {
              if (a == 1 && w == 1) continue;  // lo x lo: below the hi/lo pair's precision
              const uint64_t ad = sdesc_sw128(sa + a * kABytes + kk * 32, 16, 1024);
              tc_mma_f16(tmem, ad, bd, idesc, (i | kk | a | w) != 0 ? 1u : 0u);
            }
          }
        }
        tc_commit(&empty[s]);
      }
      tc_commit(done);
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    uint32_t ok = 1;
    if (lane == 0) ok = mbar_wait(done, 0, g.status) ? 1u : 0u;
    ok = __shfl_sync(0xffffffffu, ok, 0);
    __syncwarp();
    tc_fence_after();
    if (ok && nkb > 0) {
      const int row = m0 + q * 32 + lane;
      const uint32_t tbase = tmem + (static_cast<uint32_t>(q * 32) << 16);
      if (g.epi == 0) {
        __nv_bfloat16* hi = static_cast<__nv_bfloat16*>(g.out0);
        __nv_bfloat16* lo = static_cast<__nv_bfloat16*>(g.out1);
        for (int c = 0; c < g.BN; c += 16) {
          float v[16];
          tmem_ld16(tbase + c, v);
          const int col = n0 + c;
          if (row < g.M && col < g.ldo) {
            uint32_t h[8], l[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * e]);
              const __nv_bfloat16 h1 = __float2bfloat16_rn(v[2 * e + 1]);
              const __nv_bfloat16 l0 = __float2bfloat16_rn(v[2 * e] - __bfloat162float(h0));
              const __nv_bfloat16 l1 = __float2bfloat16_rn(v[2 * e + 1] - __bfloat162float(h1));
              h[e] = pack_bf16x2(h0, h1);
              l[e] = pack_bf16x2(l0, l1);
            }
            const size_t off = static_cast<size_t>(row) * g.ldo + col;
            uint4* ph = reinterpret_cast<uint4*>(hi + off);
            uint4* pl = reinterpret_cast<uint4*>(lo + off);
            ph[0] = make_uint4(h[0], h[1], h[2], h[3]);
            ph[1] = make_uint4(h[4], h[5], h[6], h[7]);
            pl[0] = make_uint4(l[0], l[1], l[2], l[3]);
            pl[1] = make_uint4(l[4], l[5], l[6], l[7]);
          }
        }
      } else {
        float* out = static_cast<float*>(g.out0) + static_cast<size_t>(blockIdx.z) * g.slab;
        for (int c = 0; c < g.BN; c += 16) {
          float v[16];
          tmem_ld16(tbase + c, v);
          const int col = n0 + c;
          if (row < g.M && col < g.N) {
            float* o = out + static_cast<size_t>(row) * g.ldo + col;
            if (g.alpha != 1.0f) {
#pragma unroll
              for (int e = 0; e < 16; ++e) v[e] *= g.alpha;
            }
            if (col + 16 <= g.N) {
#pragma unroll
              for (int e = 0; e < 4; ++e)
                reinterpret_cast<float4*>(o)[e] =
                    make_float4(v[4 * e], v[4 * e + 1], v[4 * e + 2], v[4 * e + 3]);
            } else {
              for (int e = 0; e < 16; ++e)
                if (col + e < g.N) o[e] = v[e];
            }
          }
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, tmem_cols);
}

struct ContractArgs {
  int T, stages, n_tiles, n_items, nblkS, nblkA;
  const int32_t* tile_rc;
  const int32_t* grp_start;  // [n_tiles * 4 + 1]: entries per (tile, 32-column chunk)
  const int4* ent;           // {r, (ro << 8) | co, bits of the fp32 scale, 0}
  float* z;
  int ldz;
  __nv_bfloat16* zhi;
  __nv_bfloat16* zlo;
  int ldzb;
  unsigned* status;
};

constexpr uint32_t kOpBytes = 16384u;          // one 128-wide operand tile, 64 tokens
constexpr uint32_t kCStage = 4u * kOpBytes;    // S hi, S lo, A hi, A lo
constexpr uint32_t kCStageBuf = 128u * 33u * 4u;  // 128 x 32 (+1 pad) epilogue staging

// Persistent: one CTA per SM walks items (example b, active tile) with
// b = item / n_tiles, so the tiles of one example run together and share
// operands through L2. Two TMEM accumulators let the gather epilogue of one
// item overlap the loads and MMAs of the next.
__global__ void __launch_bounds__(kThreads, 1)
    k_tc_contract(const __grid_constant__ CUtensorMap tmShi, const __grid_constant__ CUtensorMap tmSlo,
                  const __grid_constant__ CUtensorMap tmAhi, const __grid_constant__ CUtensorMap tmAlo,
                  const ContractArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float* stage_buf = reinterpret_cast<float*>(smem + static_cast<size_t>(g.stages) * kCStage);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(stage_buf) + kCStageBuf);
  uint64_t* empty = full + g.stages;
  uint64_t* tfull = empty + g.stages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  const int nkb = (g.T + 63) / 64;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmShi);
    tma_prefetch_desc(&tmSlo);
    tma_prefetch_desc(&tmAhi);
    tma_prefetch_desc(&tmAlo);
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      bool ok = true;
      for (int item = blockIdx.x; item < g.n_items && ok; item += gridDim.x) {
        const int b = item / g.n_tiles, tile = item % g.n_tiles;
        const int rc = g.tile_rc[tile];
        const int zs = b * g.nblkS + (rc >> 16), za = b * g.nblkA + (rc & 0xFFFF);
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = rs;
          const uint32_t ph = rph;
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
          }
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + static_cast<size_t>(s) * kCStage;
          mbar_arrive_expect_tx(&full[s], kCStage);
          const int t0 = kb * 64;
          tma_load_3d(st + 0 * kOpBytes, &tmShi, 0, t0, zs, &full[s]);
          tma_load_3d(st + 0 * kOpBytes + 8192, &tmShi, 64, t0, zs, &full[s]);
          tma_load_3d(st + 1 * kOpBytes, &tmSlo, 0, t0, zs, &full[s]);
          tma_load_3d(st + 1 * kOpBytes + 8192, &tmSlo, 64, t0, zs, &full[s]);
          tma_load_3d(st + 2 * kOpBytes, &tmAhi, 0, t0, za, &full[s]);
          tma_load_3d(st + 2 * kOpBytes + 8192, &tmAhi, 64, t0, za, &full[s]);
          tma_load_3d(st + 3 * kOpBytes, &tmAlo, 0, t0, za, &full[s]);
          tma_load_3d(st + 3 * kOpBytes + 8192, &tmAlo, 64, t0, za, &full[s]);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, 128, 1, 1);
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      int i = 0;
      bool ok = true;
      // descriptor of S hi in ring slot rs (MN-major operands: LBO 8192, SBO 1024)
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 8192, 1024);
      uint64_t dsh = dbase;
      for (int item = blockIdx.x; item < g.n_items && ok; item += gridDim.x, ++i) {
        const int buf = i & 1;
        const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
        if (!mbar_wait(&tempty[buf], aph ^ 1u, g.status)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * 128u;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = rs;
          const uint32_t ph = rph;
          const uint64_t sh0 = dsh;  // S hi of this slot; S lo, A hi, A lo follow kOpBytes apart
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
            dsh = dbase;
          } else {
            dsh += kCStage >> 4;
          }
          if (!mbar_wait(&full[s], ph, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          constexpr uint64_t kOp = kOpBytes >> 4, kRow16 = 2048u >> 4;  // 16 token rows of 128 bytes
#pragma unroll
          for (int kk = 0; kk < 4; ++kk) {
            const uint64_t sh = sh0 + kk * kRow16, sl = sh + kOp, ah = sh + 2 * kOp, al = sh + 3 * kOp;
            tc_mma_f16(d, sh, ah, idesc, (kb | kk) != 0 ? 1u : 0u);
            tc_mma_f16(d, sh, al, idesc, 1u);
            tc_mma_f16(d, sl, ah, idesc, 1u);
          }
          tc_commit(&empty[s]);
        }
        tc_commit(&tfull[buf]);
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    const int etid = threadIdx.x - 64;  // 0..127 over the four epilogue warps
    int i = 0;
    for (int item = blockIdx.x; item < g.n_items; item += gridDim.x, ++i) {
      const int buf = i & 1;
      const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
      uint32_t ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[buf], aph, g.status) ? 1u : 0u;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      tc_fence_after();
      // All four warps must agree before the shared staging is used.
      ok = __syncthreads_and_named(ok);
      if (!ok) break;
      const int b = item / g.n_tiles, tile = item % g.n_tiles;
      const uint32_t tb = tmem + buf * 128u + (static_cast<uint32_t>(q * 32) << 16);
      const size_t zrow = static_cast<size_t>(b);
      for (int j = 0; j < 4; ++j) {
        float v[32];
        tmem_ld32(tb + 32 * j, v);
#pragma unroll
        for (int c = 0; c < 32; ++c) stage_buf[(q * 32 + lane) * 33 + c] = v[c];
        named_bar_sync(1, 128);
        const int e0 = g.grp_start[tile * 4 + j], e1 = g.grp_start[tile * 4 + j + 1];
        for (int e = e0 + etid; e < e1; e += 4 * 128) {
          int4 en[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int eu = e + u * 128;
            en[u] = eu < e1 ? __ldg(&g.ent[eu]) : make_int4(-1, 0, 0, 0);
          }
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            if (en[u].x < 0) continue;
            const int r = en[u].x, off = en[u].y;
            const float val = __int_as_float(en[u].z) * stage_buf[(off >> 8) * 33 + (off & 31)];
            if (g.z) g.z[zrow * g.ldz + r] = val;
            if (g.zhi) {
              const __nv_bfloat16 h = __float2bfloat16_rn(val);
              g.zhi[zrow * g.ldzb + r] = h;
              g.zlo[zrow * g.ldzb + r] = __float2bfloat16_rn(val - __bfloat162float(h));
            }
          }
        }
        named_bar_sync(1, 128);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_relaxed(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 256);
}

// k_tc_ekfac -- EK-FAC eigenvalue correction (Sec. 2.2 "EK-FAC approximation":
// the mean square of each coordinate of the gradients in the K-FAC eigenbasis,
// App. C.2: over examples, sequence-level gradients). For one 128 x 128 tile
// (rt, ct) of the full d_out x d_in coordinate block and a run of examples,
// G~_b[tile] is formed exactly as in k_tc_contract (3 MMAs per K step over the
// tokens) and its squares are summed over the run in TMEM (columns 256..383),
// so each item writes one fp32 partial tile. Items are chunk-major
// (item = chunk * n_tiles + tile): CTAs running together read the same
// examples' operands through L2.
struct EkfacArgs {
  int T, stages, n_rt, n_ct, n_tiles, n_items, bpc, B, nblkS, nblkA, d_out, d_in;
  float* part;  // [n_chunks][d_out][d_in]
  unsigned* status;
};

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_ekfac(const __grid_constant__ CUtensorMap tmShi, const __grid_constant__ CUtensorMap tmSlo,
               const __grid_constant__ CUtensorMap tmAhi, const __grid_constant__ CUtensorMap tmAlo,
               const EkfacArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(g.stages) * kCStage);
  uint64_t* empty = full + g.stages;
  uint64_t* tfull = empty + g.stages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  const int nkb = (g.T + 63) / 64;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmShi);
    tma_prefetch_desc(&tmSlo);
    tma_prefetch_desc(&tmAhi);
    tma_prefetch_desc(&tmAlo);
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      bool ok = true;
      for (int item = blockIdx.x; item < g.n_items && ok; item += gridDim.x) {
        const int chunk = item / g.n_tiles, tile = item % g.n_tiles;
        const int rt = tile / g.n_ct, ct = tile % g.n_ct;
        const int b1 = min(g.B, (chunk + 1) * g.bpc);
        for (int b = chunk * g.bpc; b < b1 && ok; ++b) {
          const int zs = b * g.nblkS + rt, za = b * g.nblkA + ct;
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const int s = rs;
            const uint32_t ph = rph;
            if (++rs == g.stages) {
              rs = 0;
              rph ^= 1u;
            }
            if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) {
              ok = false;
              break;
            }
            uint8_t* st = smem + static_cast<size_t>(s) * kCStage;
            mbar_arrive_expect_tx(&full[s], kCStage);
            const int t0 = kb * 64;
            tma_load_3d(st + 0 * kOpBytes, &tmShi, 0, t0, zs, &full[s]);
            tma_load_3d(st + 0 * kOpBytes + 8192, &tmShi, 64, t0, zs, &full[s]);
            tma_load_3d(st + 1 * kOpBytes, &tmSlo, 0, t0, zs, &full[s]);
            tma_load_3d(st + 1 * kOpBytes + 8192, &tmSlo, 64, t0, zs, &full[s]);
            tma_load_3d(st + 2 * kOpBytes, &tmAhi, 0, t0, za, &full[s]);
            tma_load_3d(st + 2 * kOpBytes + 8192, &tmAhi, 64, t0, za, &full[s]);
            tma_load_3d(st + 3 * kOpBytes, &tmAlo, 0, t0, za, &full[s]);
            tma_load_3d(st + 3 * kOpBytes + 8192, &tmAlo, 64, t0, za, &full[s]);
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16_f32(128, 128, 1, 1);
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      int i = 0;  // examples issued by this CTA (selects the TMEM buffer)
      bool ok = true;
      for (int item = blockIdx.x; item < g.n_items && ok; item += gridDim.x) {
        const int chunk = item / g.n_tiles;
        const int b1 = min(g.B, (chunk + 1) * g.bpc);
        for (int b = chunk * g.bpc; b < b1 && ok; ++b, ++i) {
          const int buf = i & 1;
          const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
          if (!mbar_wait(&tempty[buf], aph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + buf * 128u;
          for (int kb = 0; kb < nkb; ++kb, ++it) {
            const int s = rs;
            const uint32_t ph = rph;
            if (++rs == g.stages) {
              rs = 0;
              rph ^= 1u;
            }
            if (!mbar_wait(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(smem + static_cast<size_t>(s) * kCStage);
#pragma unroll
            for (int kk = 0; kk < 4; ++kk) {
              const uint32_t o = kk * 2048u;  // 16 token rows of 128 bytes
              const uint64_t sh = sdesc_sw128(sa + 0 * kOpBytes + o, 8192, 1024);
              const uint64_t sl = sdesc_sw128(sa + 1 * kOpBytes + o, 8192, 1024);
              const uint64_t ah = sdesc_sw128(sa + 2 * kOpBytes + o, 8192, 1024);
              const uint64_t al = sdesc_sw128(sa + 3 * kOpBytes + o, 8192, 1024);
              tc_mma_f16(d, sh, ah, idesc, (kb | kk) != 0 ? 1u : 0u);
              tc_mma_f16(d, sh, al, idesc, 1u);
              tc_mma_f16(d, sl, ah, idesc, 1u);
            }
            tc_commit(&empty[s]);
          }
          tc_commit(&tfull[buf]);
        }
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    const uint32_t lane_base = static_cast<uint32_t>(q * 32) << 16;
    const int row_in = q * 32 + lane;
    int i = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < g.n_items && ok; item += gridDim.x) {
      const int chunk = item / g.n_tiles, tile = item % g.n_tiles;
      const int rt = tile / g.n_ct, ct = tile % g.n_ct;
      const int b0 = chunk * g.bpc, b1 = min(g.B, (chunk + 1) * g.bpc);
      for (int b = b0; b < b1; ++b, ++i) {
        const int buf = i & 1;
        const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
        uint32_t w_ok = 1;
        if (lane == 0) w_ok = mbar_wait(&tfull[buf], aph, g.status) ? 1u : 0u;
        w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
        __syncwarp();
        tc_fence_after();
        if (!__syncthreads_and_named(w_ok)) {
          ok = false;
          break;
        }
        for (int j = 0; j < 4; ++j) {
          float v[32], acc[32];
          tmem_ld32(tmem + lane_base + buf * 128u + 32 * j, v);
          if (b == b0) {
#pragma unroll
            for (int c = 0; c < 32; ++c) acc[c] = __fmul_rn(v[c], v[c]);
          } else {
            tmem_ld32(tmem + lane_base + 256u + 32 * j, acc);
#pragma unroll
            for (int c = 0; c < 32; ++c) acc[c] = __fadd_rn(acc[c], __fmul_rn(v[c], v[c]));
          }
          if (b + 1 < b1) {
            tmem_st32(tmem + lane_base + 256u + 32 * j, acc);
          } else {
            const int row = rt * 128 + row_in, col0 = ct * 128 + 32 * j;
            if (row < g.d_out) {
              float* dst = g.part + (static_cast<size_t>(chunk) * g.d_out + row) * g.d_in + col0;
#pragma unroll
              for (int c = 0; c < 32; ++c)
                if (col0 + c < g.d_in) dst[c] = acc[c];
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_relaxed(&tempty[buf]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, 512);
}

// sumsq[j * ld + i] (+)= sum over chunks c of part[c][j][i], chunks in order (fp64).
__global__ void k_ekfac_finalize(const float* __restrict__ part, int n_chunks, int d_out, int d_in,
                                 double* __restrict__ sumsq, int ld, int accumulate) {
  const size_t n = static_cast<size_t>(d_out) * d_in;
  for (size_t e = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; e < n;
       e += static_cast<size_t>(gridDim.x) * blockDim.x) {
    double t = 0.0;
    for (int c = 0; c < n_chunks; ++c) t += static_cast<double>(part[static_cast<size_t>(c) * n + e]);
    const size_t o = (e / d_in) * static_cast<size_t>(ld) + e % d_in;
    sumsq[o] = accumulate ? sumsq[o] + t : t;
  }
}

size_t gemm_smem_bytes(int BN, int stages, int nA, int nW = 1) {
  return 1024 + static_cast<size_t>(stages) * (nA * kABytes + nW * BN * 128u) + (2 * stages + 1) * 8 + 16;
}

size_t contract_smem_bytes(int stages) {
  return 1024 + static_cast<size_t>(stages) * kCStage + kCStageBuf + (2 * stages + 4) * 8 + 16;
}


// ------------------------------------------------------------------------
// k_tc_rotate -- persistent rotation GEMM: D = X W^T written as bf16 hi/lo.
// One CTA per SM walks a static tile schedule (tile t -> M block t / nN,
// N block t % nN, so the nN CTAs sharing an activation block run together and
// the block is read from HBM once). Two TMEM accumulators alternate between
// tiles: the MMA warp fills one while the epilogue warps drain the other.
// Epilogue: 32-column TMEM loads, hi/lo split, 32-byte stores (a full sector
// per thread). The output is blocked for the contraction that reads it:
// element (row = b*T + t, col) sits at ((b * (ldo/128) + col/128) * T + t) * 128
// + col % 128, so one 128-column block of one example is T*256 contiguous bytes.
struct RotArgs {
  int M, K, BN, stages, nN, n_tiles, ldo, T, nbias;
  __nv_bfloat16* hi;
  __nv_bfloat16* lo;
  const float* bias;        // per output column (the constant-1 input channel), or null
  const int32_t* lengths;   // tokens kept per example (later tokens give 0), or null
  unsigned* status;
};

// Bias channel and token lengths, applied to one W-column chunk of one output
// row before the hi/lo split.
template <int W>
__device__ __forceinline__ void rot_fixup(const RotArgs& g, int row, int col, float (&v)[W]) {
  if (g.bias) {
#pragma unroll
    for (int e = 0; e < W; ++e) v[e] += col + e < g.nbias ? __ldg(g.bias + col + e) : 0.f;
  }
  if (g.lengths) {
    const int bex = row / g.T;
    if (row - bex * g.T >= __ldg(g.lengths + bex)) {
#pragma unroll
      for (int e = 0; e < W; ++e) v[e] = 0.f;
    }
  }
}

// One W-column chunk (W = 32 or 16) of one output row: fix-ups, hi/lo split,
// 32-byte stores into the blocked layout (element (row = b T + t, col) at
// ((b (ldo / 128) + col / 128) T + t) 128 + col % 128).
template <int W>
__device__ __forceinline__ void rot_store(const RotArgs& g, int row, int col, float (&v)[W]) {
  rot_fixup<W>(g, row, col, v);
  uint32_t h[W / 2], l[W / 2];
#pragma unroll
  for (int e = 0; e < W / 2; ++e) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(v[2 * e]);
    const __nv_bfloat16 h1 = __float2bfloat16_rn(v[2 * e + 1]);
    h[e] = pack_bf16x2(h0, h1);
    l[e] = pack_bf16x2(__float2bfloat16_rn(v[2 * e] - __bfloat162float(h0)),
                       __float2bfloat16_rn(v[2 * e + 1] - __bfloat162float(h1)));
  }
  const int bex = row / g.T, tok = row - bex * g.T;
  // 16-column pieces: tiles start on multiples of 16, so a piece never crosses a
  // 128-column block (a 32-column chunk may, and is placed piece by piece).
#pragma unroll
  for (int q = 0; q < W / 16; ++q) {
    const int cq = col + 16 * q;
    const size_t off = ((static_cast<size_t>(bex) * (g.ldo >> 7) + (cq >> 7)) * g.T + tok) * 128 + (cq & 127);
    uint32_t w[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) w[e] = h[8 * q + e];
    st_global_v8(g.hi + off, w);
#pragma unroll
    for (int e = 0; e < 8; ++e) w[e] = l[8 * q + e];
    st_global_v8(g.lo + off, w);
  }
}

// Drains one accumulator row of a BN-column tile (BN a multiple of 16).
__device__ __forceinline__ void rot_drain(const RotArgs& g, uint32_t tb, int row, int n0) {
  int c = 0;
  for (; c + 32 <= g.BN; c += 32) {
    float v[32];
    tmem_ld32(tb + c, v);
    if (row < g.M && n0 + c < g.ldo) rot_store<32>(g, row, n0 + c, v);
  }
  if (c < g.BN) {
    float v[16];
    tmem_ld16(tb + c, v);
    if (row < g.M && n0 + c < g.ldo) rot_store<16>(g, row, n0 + c, v);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    k_tc_rotate(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                const RotArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t stage_bytes = kABytes + static_cast<uint32_t>(g.BN) * 128u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(g.stages) * stage_bytes);
  uint64_t* empty = full + g.stages;
  uint64_t* tfull = empty + g.stages;  // accumulator ready, per TMEM buffer
  uint64_t* tempty = tfull + 2;        // accumulator drained, per TMEM buffer
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  const uint32_t tcols = g.BN <= 64 ? 128u : g.BN <= 128 ? 256u : 512u;
  const uint32_t bstride = tcols / 2;
  const int nkb = (g.K + 63) / 64;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], 4);  // one arrive per epilogue warp
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, tcols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      bool ok = true;
      for (int t = blockIdx.x; t < g.n_tiles && ok; t += gridDim.x) {
        const int m0 = (t / g.nN) * 128, n0 = (t % g.nN) * g.BN;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = rs;
          const uint32_t ph = rph;
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
          }
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          uint8_t* st = smem + static_cast<size_t>(s) * stage_bytes;
          mbar_arrive_expect_tx(&full[s], stage_bytes);
          tma_load_2d(st, &tmX, kb * 64, m0, &full[s]);
          tma_load_2d(st + kABytes, &tmW, kb * 64, n0, &full[s]);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // The issuing thread's own work per K block is kept minimal (one lane issues
      // every MMA, so its instruction latency paces the tensor pipe): ring slot,
      // phase and operand descriptors advance incrementally. A descriptor's
      // address field is (byte address >> 4), so +2 steps 32 bytes (K = 16 bf16).
      const uint32_t idesc = idesc_bf16_f32(128, g.BN, 0, 0);
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      const uint64_t dstage = stage_bytes >> 4, dab = kABytes >> 4;
      uint64_t da = dbase;  // descriptor of operand A in ring slot rs
      int rs = 0;           // ring slot of the next K block
      uint32_t rph = 0;     // and its phase parity
      int i = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < g.n_tiles && ok; t += gridDim.x, ++i) {
        const int buf = i & 1;
        const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
        if (!mbar_wait(&tempty[buf], aph ^ 1u, g.status)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * bstride;
        for (int kb = 0; kb < nkb; ++kb) {
          const int s = rs;
          const uint32_t ph = rph;
          const uint64_t a0 = da, b0 = da + dab;
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
            da = dbase;
          } else {
            da += dstage;
          }
          if (!mbar_wait(&full[s], ph, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          tc_mma_f16(d, a0, b0, idesc, kb != 0 ? 1u : 0u);
          tc_mma_f16(d, a0 + 2, b0 + 2, idesc, 1u);
          tc_mma_f16(d, a0 + 4, b0 + 4, idesc, 1u);
          tc_mma_f16(d, a0 + 6, b0 + 6, idesc, 1u);
          tc_commit(&empty[s]);
        }
        tc_commit(&tfull[buf]);
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    int i = 0;
    for (int t = blockIdx.x; t < g.n_tiles; t += gridDim.x, ++i) {
      const int buf = i & 1;
      const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
      uint32_t ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[buf], aph, g.status) ? 1u : 0u;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      tc_fence_after();
      if (!ok) break;
      const int m0 = (t / g.nN) * 128, n0 = (t % g.nN) * g.BN;
      const int row = m0 + q * 32 + lane;
      const uint32_t tb = tmem + buf * bstride + (static_cast<uint32_t>(q * 32) << 16);
      rot_drain(g, tb, row, n0);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_relaxed(&tempty[buf]);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, tcols);
}

size_t rotate_smem_bytes(int BN, int stages) {
  return 1024 + static_cast<size_t>(stages) * (kABytes + BN * 128u) + (2 * stages + 4) * 8 + 16;
}


// ------------------------------------------------------------------------
// k_tc_rotate2 -- the rotation GEMM on CTA pairs (tcgen05 cta_group::2,
// M = 256). Each CTA of a pair loads its own 128 activation rows and its own
// half of the BN eigenvector rows (no multicast), so per-SM shared-memory
// traffic per MMA flop drops by a third against one CTA per tile; the leader
// CTA (rank 0) issues the M = 256 MMAs, whose accumulator rows are split over
// the two CTAs' TMEM. Pipeline completion (TMA bytes) and accumulator release
// are counted on the leader's barriers; MMA completion is multicast to both
// CTAs. Epilogue as in k_tc_rotate (blocked hi/lo output).
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    k_tc_rotate2(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                 const RotArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const int half = g.BN / 2;  // W rows held by this CTA
  const uint32_t stage_bytes = kABytes + static_cast<uint32_t>(half) * 128u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + static_cast<size_t>(g.stages) * stage_bytes);
  uint64_t* empty = full + g.stages;
  uint64_t* tfull = empty + g.stages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);
  const uint32_t tcols = g.BN <= 64 ? 128u : g.BN <= 128 ? 256u : 512u;
  const uint32_t bstride = tcols / 2;
  const int nkb = (g.K + 63) / 64;
  const int cl = blockIdx.x >> 1, ncl = gridDim.x >> 1;

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmX);
    tma_prefetch_desc(&tmW);
    for (int s = 0; s < g.stages; ++s) {
      mbar_init(&full[s], 2);   // one expect_tx arrive from each CTA (leader's copy is used)
      mbar_init(&empty[s], 1);  // MMA completion, multicast to both CTAs
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);   // multicast to both CTAs
      mbar_init(&tempty[b], 8);  // 4 epilogue warps x 2 CTAs (leader's copy is used)
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc_pair(tmem_slot, tcols);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // barriers of both CTAs initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    if (lane == 0) {
      uint32_t it = 0;
      int rs = 0;         // ring slot of pipeline iteration it (it % stages)
      uint32_t rph = 0;  // and its phase parity ((it / stages) & 1)
      bool ok = true;
      for (int t = cl; t < g.n_tiles && ok; t += ncl) {
        const int m0 = (t / g.nN) * 256 + static_cast<int>(rank) * 128;
        const int n0 = (t % g.nN) * g.BN + static_cast<int>(rank) * half;
        for (int kb = 0; kb < nkb; ++kb, ++it) {
          const int s = rs;
          const uint32_t ph = rph;
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
          }
          if (!mbar_wait(&empty[s], ph ^ 1u, g.status)) {
            ok = false;
            break;
          }
          const uint32_t st = smem_u32(smem + static_cast<size_t>(s) * stage_bytes);
          const uint32_t fl = mapa_shared(smem_u32(&full[s]), 0);
          mbar_arrive_expect_tx_cluster(fl, stage_bytes);
          tma_load_2d_pair(st, &tmX, kb * 64, m0, fl);
          tma_load_2d_pair(st + kABytes, &tmW, kb * 64, n0, fl);
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // as in k_tc_rotate: slot, phase and descriptors advance incrementally
      const uint32_t idesc = idesc_bf16_f32(256, g.BN, 0, 0);
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      const uint64_t dstage = stage_bytes >> 4, dab = kABytes >> 4;
      uint64_t da = dbase;
      int rs = 0;
      uint32_t rph = 0;
      int i = 0;
      bool ok = true;
      for (int t = cl; t < g.n_tiles && ok; t += ncl, ++i) {
        const int buf = i & 1;
        const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
        if (!mbar_wait(&tempty[buf], aph ^ 1u, g.status)) break;
        tc_fence_after();
        const uint32_t d = tmem + buf * bstride;
        for (int kb = 0; kb < nkb; ++kb) {
          const int s = rs;
          const uint32_t ph = rph;
          const uint64_t a0 = da, b0 = da + dab;
          if (++rs == g.stages) {
            rs = 0;
            rph ^= 1u;
            da = dbase;
          } else {
            da += dstage;
          }
          if (!mbar_wait(&full[s], ph, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          tc_mma_f16_pair(d, a0, b0, idesc, kb != 0 ? 1u : 0u);
          tc_mma_f16_pair(d, a0 + 2, b0 + 2, idesc, 1u);
          tc_mma_f16_pair(d, a0 + 4, b0 + 4, idesc, 1u);
          tc_mma_f16_pair(d, a0 + 6, b0 + 6, idesc, 1u);
          tc_commit_pair_mc(&empty[s], 0x3);
        }
        tc_commit_pair_mc(&tfull[buf], 0x3);
      }
    }
    __syncwarp();
  } else {
    const int q = warp & 3;
    int i = 0;
    for (int t = cl; t < g.n_tiles; t += ncl, ++i) {
      const int buf = i & 1;
      const uint32_t aph = static_cast<uint32_t>(i >> 1) & 1u;
      uint32_t ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[buf], aph, g.status) ? 1u : 0u;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      __syncwarp();
      tc_fence_after();
      if (!ok) break;
      const int m0 = (t / g.nN) * 256 + static_cast<int>(rank) * 128, n0 = (t % g.nN) * g.BN;
      const int row = m0 + q * 32 + lane;
      const uint32_t tb = tmem + buf * bstride + (static_cast<uint32_t>(q * 32) << 16);
      rot_drain(g, tb, row, n0);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(&tempty[buf]), 0));
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while its peer may still signal it
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem, tcols);
}

size_t rotate2_smem_bytes(int BN, int stages) {
  return 1024 + static_cast<size_t>(stages) * (kABytes + (BN / 2) * 128u) + (2 * stages + 4) * 8 + 16;
}

}  // namespace

static int tmap_bf16_2d(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t rows,
                        uint64_t row_stride_elems, uint32_t box_inner, uint32_t box_rows) {
  const uint64_t dims[2] = {inner, rows};
  const uint64_t strides[1] = {row_stride_elems * 2};
  const uint32_t box[2] = {box_inner, box_rows};
  return make_tmap(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, base, dims, strides, box,
                   CU_TENSOR_MAP_SWIZZLE_128B);
}

// Blocked intermediate [B * nblk][T][128] (bf16): box of 64 columns x 64 tokens.
static int tmap_bf16_blocked(CUtensorMap* tm, const void* base, uint64_t T, uint64_t nbatch) {
  const uint64_t dims[3] = {128, T, nbatch};
  const uint64_t strides[2] = {128 * 2, 128 * 2 * T};
  const uint32_t box[3] = {64, 64, 1};
  return make_tmap(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, base, dims, strides, box,
                   CU_TENSOR_MAP_SWIZZLE_128B);
}

static cudaError_t launch_tc_gemm_impl(int M, int N, int K, const void* X0, const void* X1, int ldx,
                                      const void* W, const void* W1, int ldw, int Wrows, int splits, int epi,
                                      void* out0, void* out1, int ldo, size_t slab, float alpha,
                                      TcGemmCfg cfg, unsigned* status, cudaStream_t st) {
  if (M <= 0 || N <= 0) return cudaSuccess;
  const int nA = X1 ? 2 : 1;
  const int nW = W1 ? 2 : 1;
  CUtensorMap tX0, tX1, tW, tW1;
  if (tmap_bf16_2d(&tX0, X0, static_cast<uint64_t>(K), static_cast<uint64_t>(M), ldx, 64, 128))
    return cudaErrorInvalidValue;
  if (nA > 1) {
    if (tmap_bf16_2d(&tX1, X1, K, M, ldx, 64, 128)) return cudaErrorInvalidValue;
  } else {
    tX1 = tX0;
  }
  if (tmap_bf16_2d(&tW, W, K, Wrows, ldw, 64, cfg.BN)) return cudaErrorInvalidValue;
  if (nW > 1) {
    if (tmap_bf16_2d(&tW1, W1, K, Wrows, ldw, 64, cfg.BN)) return cudaErrorInvalidValue;
  } else {
    tW1 = tW;
  }
  const int nkb = (K + 63) / 64;
  splits = max(1, min(splits, nkb));
  const int kbps = (nkb + splits - 1) / splits;
  splits = (nkb + kbps - 1) / kbps;
  GemmArgs g;
  g.M = M;
  g.N = N;
  g.K = K;
  g.BN = cfg.BN;
  g.stages = cfg.stages;
  g.nA = nA;
  g.nW = nW;
  g.kbps = kbps;
  g.epi = epi;
  g.ldo = ldo;
  g.alpha = alpha;
  g.out0 = out0;
  g.out1 = out1;
  g.slab = slab;
  g.status = status;
  const size_t smem = gemm_smem_bytes(cfg.BN, cfg.stages, nA, nW);
  cudaError_t e = cudaFuncSetAttribute(k_tc_gemm, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid((N + cfg.BN - 1) / cfg.BN, (M + 127) / 128, splits);
  k_tc_gemm<<<grid, kThreads, smem, st>>>(tX0, tX1, tW, tW1, g);
  return cudaGetLastError();
}

cudaError_t launch_tc_gemm(int M, int N, int K, const void* X0, const void* X1, int ldx,
                                const void* W, int ldw, int Wrows, int splits, int epi,
                                void* out0, void* out1, int ldo, size_t slab, TcGemmCfg cfg,
                                unsigned* status, cudaStream_t st) {
  return launch_tc_gemm_impl(M, N, K, X0, X1, ldx, W, nullptr, ldw, Wrows, splits, epi, out0, out1, ldo,
                             slab, 1.0f, cfg, status, st);
}

cudaError_t launch_tc_gemm_hl(int M, int N, int K, const void* Ah, const void* Al, int lda, const void* Bh,
                              const void* Bl, int ldb, float* out, int ldo, float alpha, unsigned* status,
                              cudaStream_t st) {
  // 128-column tiles: a stage holds 2 x 16 KB of A and 2 x 16 KB of B, three stages.
  return launch_tc_gemm_impl(M, N, K, Ah, Al, lda, Bh, Bl, ldb, N, 1, 1, out, nullptr, ldo, 0, alpha,
                             TcGemmCfg{128, 3}, status, st);
}

// CTA pairs measured faster for short reductions (K <= 1536: the hi/lo
// epilogue dominates and halving the per-SM operand stream helps) and for few
// output columns (n <= 256: the activations stream from HBM and every 128-row
// tile re-reads the whole eigenvector operand from L2, which the pair halves;
// OLMo-2-1B stack 1,487 -> 1,557 examples/s), and slower for long reductions
// with many columns.
static bool rotate_pairs(int K, int n) { return K <= 1536 || n <= 256; }

// N tile width for `n` output columns: as few tiles of at most 256 columns as
// is cheapest, each a multiple of `gran` (16: the tcgen05 N granularity, for one
// CTA and for CTA pairs, whose halves of N / 2 rows are whole 8-row swizzle
// atoms), counting a fixed per-tile overhead of 32 columns.
int rotate_bn(int n, int gran) {
  const int n0 = (n + 255) / 256;
  int best = 0, best_cost = 1 << 30;
  for (int nN = n0; nN <= n0 + 1; ++nN) {
    const int bn = ((n + nN - 1) / nN + gran - 1) / gran * gran;
    const int cost = nN * bn + 32 * nN;
    if (cost < best_cost) {
      best_cost = cost;
      best = bn;
    }
  }
  return best;
}

cudaError_t launch_tc_rotate(int M, int K, const void* X, int ldx, const void* W, int ldw, int Wrows,
                             void* hi, void* lo, int ldo, int T, const float* bias,
                             const int32_t* lengths, int num_sms, unsigned* status, cudaStream_t st) {
  if (M <= 0) return cudaSuccess;
  const bool pairs = rotate_pairs(K, Wrows);
  const int BN = rotate_bn(Wrows, 16);
  // As many pipeline stages as fit in 227 KB of shared memory (at most 8).
  int stages = 2;
  while (stages < 8 && rotate_smem_bytes(BN, stages + 1) <= 232448) ++stages;
  CUtensorMap tX, tW;
  if (tmap_bf16_2d(&tX, X, static_cast<uint64_t>(K), static_cast<uint64_t>(M), ldx, 64, 128) ||
      tmap_bf16_2d(&tW, W, K, Wrows, ldw, 64, BN))
    return cudaErrorInvalidValue;
  RotArgs g;
  g.M = M;
  g.K = K;
  g.BN = BN;
  g.stages = stages;
  g.nN = (Wrows + BN - 1) / BN;  // columns past the last tile (padding up to ldo) are not written
  g.n_tiles = ((M + 127) / 128) * g.nN;
  g.ldo = ldo;
  g.T = T;
  g.hi = static_cast<__nv_bfloat16*>(hi);
  g.lo = static_cast<__nv_bfloat16*>(lo);
  g.bias = bias;
  g.nbias = Wrows;
  g.lengths = lengths;
  g.status = status;
  if (pairs) {
    // CTA pairs: tiles of 256 rows, W split in halves of BN / 2 rows.
    CUtensorMap tWh;
    if (tmap_bf16_2d(&tWh, W, K, Wrows, ldw, 64, BN / 2)) return cudaErrorInvalidValue;
    int st2 = 2;
    while (st2 < 8 && rotate2_smem_bytes(BN, st2 + 1) <= 232448) ++st2;
    g.stages = st2;
    g.n_tiles = ((M + 255) / 256) * g.nN;
    const size_t smem = rotate2_smem_bytes(BN, st2);
    cudaError_t e = cudaFuncSetAttribute(k_tc_rotate2, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int clusters = std::min(g.n_tiles, std::max(1, num_sms / 2));
    k_tc_rotate2<<<2 * clusters, kThreads, smem, st>>>(tX, tWh, g);
    return cudaGetLastError();
  }
  const size_t smem = rotate_smem_bytes(BN, stages);
  cudaError_t e = cudaFuncSetAttribute(k_tc_rotate, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int grid = std::min(g.n_tiles, std::max(1, num_sms));
  k_tc_rotate<<<grid, kThreads, smem, st>>>(tX, tW, g);
  return cudaGetLastError();
}

int tc_gemm_splits_used(int K, int splits) {
  const int nkb = (K + 63) / 64;
  splits = max(1, min(splits, nkb));
  const int kbps = (nkb + splits - 1) / splits;
  return (nkb + kbps - 1) / kbps;
}

cudaError_t launch_tc_contract(const void* St_hi, const void* St_lo, int ldS, const void* At_hi,
                               const void* At_lo, int ldA, int B, int T, const eogp_plan* plan,
                               float* z, int ldz, void* zhi, void* zlo, int ldzb, int stages,
                               int num_sms, unsigned* status, cudaStream_t st) {
  if (B <= 0 || plan->n_tiles() == 0) return cudaSuccess;
  CUtensorMap tSh, tSl, tAh, tAl;
  const uint64_t nS = static_cast<uint64_t>(B) * (ldS / 128), nA = static_cast<uint64_t>(B) * (ldA / 128);
  if (tmap_bf16_blocked(&tSh, St_hi, T, nS) || tmap_bf16_blocked(&tSl, St_lo, T, nS) ||
      tmap_bf16_blocked(&tAh, At_hi, T, nA) || tmap_bf16_blocked(&tAl, At_lo, T, nA))
    return cudaErrorInvalidValue;
  ContractArgs g;
  g.T = T;
  g.nblkS = ldS / 128;
  g.nblkA = ldA / 128;
  g.stages = stages;
  g.n_tiles = plan->n_tiles();
  g.n_items = g.n_tiles * B;
  g.tile_rc = plan->d_tile_rc;
  g.grp_start = plan->d_grp_start;
  g.ent = reinterpret_cast<const int4*>(plan->d_ent);
  g.z = z;
  g.ldz = ldz;
  g.zhi = static_cast<__nv_bfloat16*>(zhi);
  g.zlo = static_cast<__nv_bfloat16*>(zlo);
  g.ldzb = ldzb;
  g.status = status;
  const size_t smem = contract_smem_bytes(stages);
  cudaError_t e = cudaFuncSetAttribute(k_tc_contract, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int grid = std::min(g.n_items, std::max(1, num_sms));
  k_tc_contract<<<grid, kThreads, smem, st>>>(tSh, tSl, tAh, tAl, g);
  return cudaGetLastError();
}

size_t ekfac_smem_bytes(int stages) {
  return 1024 + static_cast<size_t>(stages) * kCStage + (2 * stages + 4) * 8 + 16;
}

int ekfac_chunks(int B, int n_tiles, int num_sms) {
  // Enough items for about two per SM, each chunk as long as possible.
  const int want_items = 2 * std::max(1, num_sms);
  int nch = std::max(1, std::min(B, (want_items + n_tiles - 1) / n_tiles));
  const int bpc = (B + nch - 1) / nch;
  return (B + bpc - 1) / bpc;
}

cudaError_t launch_tc_ekfac(const void* St_hi, const void* St_lo, int ldS, const void* At_hi,
                            const void* At_lo, int ldA, int B, int T, int d_out, int d_in, float* part,
                            int n_chunks, double* sumsq, int ld, int accumulate, int stages, int num_sms,
                            unsigned* status, cudaStream_t st) {
  if (B <= 0) return cudaSuccess;
  CUtensorMap tSh, tSl, tAh, tAl;
  const uint64_t nS = static_cast<uint64_t>(B) * (ldS / 128), nA = static_cast<uint64_t>(B) * (ldA / 128);
  if (tmap_bf16_blocked(&tSh, St_hi, T, nS) || tmap_bf16_blocked(&tSl, St_lo, T, nS) ||
      tmap_bf16_blocked(&tAh, At_hi, T, nA) || tmap_bf16_blocked(&tAl, At_lo, T, nA))
    return cudaErrorInvalidValue;
  EkfacArgs g;
  g.T = T;
  g.stages = stages;
  g.n_rt = (d_out + 127) / 128;
  g.n_ct = (d_in + 127) / 128;
  g.n_tiles = g.n_rt * g.n_ct;
  g.bpc = (B + n_chunks - 1) / n_chunks;
  g.n_items = g.n_tiles * ((B + g.bpc - 1) / g.bpc);
  g.B = B;
  g.nblkS = ldS / 128;
  g.nblkA = ldA / 128;
  g.d_out = d_out;
  g.d_in = d_in;
  g.part = part;
  g.status = status;
  const size_t smem = ekfac_smem_bytes(stages);
  cudaError_t e = cudaFuncSetAttribute(k_tc_ekfac, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int grid = std::min(g.n_items, std::max(1, num_sms));
  k_tc_ekfac<<<grid, kThreads, smem, st>>>(tSh, tSl, tAh, tAl, g);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_ekfac_finalize<<<std::max(1, num_sms) * 4, 256, 0, st>>>(part, (B + g.bpc - 1) / g.bpc, d_out, d_in,
                                                            sumsq, ld, accumulate);
  return cudaGetLastError();
}
