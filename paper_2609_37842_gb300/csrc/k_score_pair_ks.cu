// One-bit (CODES) scoring of one module against at most 64 queries on CTA
// pairs, with two MMA-issuing threads (Sec. 3.3 Eq. onebit_influence; App. B.3
// scan): k_score_pair_ks.
//
// Why two issuers. A thread issues a tcgen05.mma about every 64 cycles
// whatever N is, and an N = 64 e2m1 MMA of a pair (M = 256, K = 64) occupies
// the tensor pipe for only about 32: one issuing thread leaves the pipe half
// idle at 64 queries, and every wait-fence-commit round of that thread idles it
// further. Measured back to back on 76 pairs: one thread 4,980 TFLOP/s at
// N = 64, two threads with their own accumulators 7,907, four 9,719 (the e2m1
// rate). Here two threads split the K range of every pipeline group: of the
// group's four 256-bit stages, issuer 0 runs stages 0 and 1 into accumulator
// d_A (TMEM columns 0-63), issuer 1 stages 2 and 3 into d_B (columns 64-127).
// The drain adds the two: both hold exact small integers (|d| <= k < 2^24), so
// d_A + d_B is the module's d_u exactly and the scores are bitwise those of the
// one-issuer kernel and the oracle's float32 evaluation.
//
// Ring invariants. Both issuers wait on the same full barrier of a group and
// each commits once to the group's empty barrier (count 2), so a group is done
// when both halves are; each issuer's own groups complete in order, hence so do
// the groups (a group's completion is the later of its two halves, and both
// sequences are ordered). That keeps the lagged reuse valid: the query stages
// of group gj are refilled once group gj - NQ is done, and the A slots form a
// ring of single stages (all eleven TMEM slots, not whole groups of four), the
// slot of stage s refilled once the group of stage s - 11 is done, so the last
// stage of group gj waits for group gj - 2 but its first three only for gj - 3.
// A waiter always waits for a group whose predecessor on the same barrier it
// has already seen complete, so no barrier phase can be passed early.
//
// The two accumulators take the columns the one-issuer kernel gives its two
// double-buffered accumulators, so a tile's MMAs wait for the drain of the
// previous tile. The drain keeps that wait short: it reads d_A and d_B into
// registers, releases them, and only then scales and stores the scores, while
// the next tile's MMAs run.
//
// Warps (16, 128 registers a thread): 0-7 expand (two per TMEM lane quarter,
// two stages of each group each), 8-11 drain (one per lane quarter, all 64
// columns), 12 owns TMEM and, in the leader CTA, is issuer 0, 13 loads the code
// boxes, 14 the query tiles, 15 is issuer 1 (leader CTA).
#include "score_tc.cuh"

namespace eogp {
namespace sc {
namespace {

constexpr int kBN = 64;                        // queries per tile (template width)
constexpr int kG = 4;                          // 256-bit stages per group (one code box)
constexpr int kQStages = 20;                   // query stages in shared memory
constexpr int kNQ = kQStages / kG;             // groups of query stages
constexpr int kCodeRing = 8;                   // code boxes in flight
constexpr int kSlots = (512 - 2 * kBN - 32) / 32;  // A slots of 32 TMEM columns, one stage each
constexpr uint32_t kAcol0 = 2u * kBN;          // first A column (after d_A, d_B)
constexpr uint32_t kSfa = kAcol0 + 32u * kSlots, kSfb = kSfa + 16u;
constexpr int kExpW = 8;                       // expander warps
constexpr int kDrW0 = kExpW;                   // first drain warp
constexpr int kDrW = 4;                        // drain warps
constexpr int kIss0Warp = kDrW0 + kDrW;        // 12
constexpr int kCodeWarp = kIss0Warp + 1;       // 13
constexpr int kQueryWarp = kIss0Warp + 2;      // 14
constexpr int kIss1Warp = kIss0Warp + 3;       // 15
constexpr int kThreads = (kIss1Warp + 1) * 32; // 512
constexpr int kCodeBoxWords = 32;              // 1024 code bits of a row per box
constexpr uint32_t kCodeBox = 128u * 128u;     // 128 rows x 128 bytes
constexpr uint32_t kStage = static_cast<uint32_t>(kBN / 2) * 128u;  // a CTA's query rows of a stage
static_assert(kSfb + 16u <= 512u, "TMEM budget");
static_assert(kSlots >= 2 * kG && kNQ * kG >= kSlots, "rings: A slots for two groups, at least as many query stages");

// Shared memory (after 1024-byte alignment): query ring, code ring, query
// scales of the current query tile, barriers.
constexpr uint32_t kCodeOff = kQStages * kStage;
constexpr uint32_t kSqOff = kCodeOff + kCodeRing * kCodeBox;
constexpr uint32_t kBarOff = kSqOff + kBN * 4;
constexpr uint32_t kSmemTotal = kBarOff + (2 * kNQ + 2 + 2 * kCodeRing + 2) * 8 + 16;

// An issuer's half of a group: its two stages (A slots at a0, a1; query stages
// at descriptors b0, b1), four K = 64 MMAs each.
__device__ __forceinline__ void issue_half(uint32_t d, uint32_t a0, uint32_t a1, uint64_t b0, uint64_t b1,
                                           uint32_t idesc, uint32_t sfa, uint32_t sfb, bool first) {
#pragma unroll
  for (int kk = 0; kk < 4; ++kk)
    tc_mma_f4_ta_pair(d, a0 + 8u * kk, b0 + 2 * kk, idesc, sfa, sfb, (!first || kk != 0) ? 1u : 0u);
#pragma unroll
  for (int kk = 0; kk < 4; ++kk) tc_mma_f4_ta_pair(d, a1 + 8u * kk, b1 + 2 * kk, idesc, sfa, sfb, 1u);
}

__global__ void __launch_bounds__(kThreads, 1)
    k_score_pair_ks(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmC,
                    const __grid_constant__ ScoreTcArgs g) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  float* sq = reinterpret_cast<float*>(smem + kSqOff);
  // group gj: full / empty barrier gj % NQ, query stages of slot gj % NQ, A
  // slots of slot gj % NG
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kBarOff);
  uint64_t* empty = full + kNQ;
  uint64_t* dfull = empty + kNQ;
  uint64_t* dempty = dfull + 1;
  uint64_t* cfull = dempty + 1;
  uint64_t* cempty = cfull + kCodeRing;
  uint64_t* fin = cempty + kCodeRing;  // [2]: each issuer's last commit (leader)
  uint32_t* tslot = reinterpret_cast<uint32_t*>(fin + 2);
  const int nst = g.D / 256;  // 256-bit stages per tile (a multiple of kG)
  const int nbx = nst / kG;   // code boxes (= groups) per tile

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmC);
    for (int s = 0; s < kNQ; ++s) {
      // leader's copy: per CTA the query producer's expect_tx arrive (+ its TMA
      // bytes) and the eight expander warps
      mbar_init(&full[s], 2 * (1 + kExpW));
      mbar_init(&empty[s], 2);  // both issuers' commits, multicast to both CTAs
    }
    mbar_init(dfull, 2);             // both issuers' commits, multicast
    mbar_init(dempty, 2 * kDrW);     // every drain warp of both CTAs (leader's copy)
    for (int b = 0; b < kCodeRing; ++b) {
      mbar_init(&cfull[b], 1);       // the producer's expect_tx arrive (+ TMA bytes)
      mbar_init(&cempty[b], kExpW);  // every expander warp, once per box
    }
    mbar_init(&fin[0], 1);
    mbar_init(&fin[1], 1);
    fence_barrier_init();
  }
  if (warp == kIss0Warp) tmem_alloc_pair(tslot, 512);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp < kExpW) {
    // ---------------------------------------------------------- expanders
    // Warp w expands the rows of TMEM lane quarter w % 4, stages 2 (w / 4) and
    // 2 (w / 4) + 1 of every group: wait for the group's slots, two 16-byte
    // loads and 32 e2m1 columns per stage, one tcgen05.wait::st, one arrive.
    const int q4 = warp & 3, half = warp >> 2;
    const int r = q4 * 32 + lane;  // stored row in the CTA's tile = TMEM lane
    const uint32_t a_lane = tmem + (static_cast<uint32_t>(q4 * 32) << 16);
    if (half == 0) {  // unit scale factors (ue8m0 0x7F = 1.0) of A and B, once
      uint32_t v[16];
#pragma unroll
      for (int e = 0; e < 16; ++e) v[e] = 0x7F7F7F7Fu;
      tmem_st16_issue(a_lane + kSfa, v);
      tmem_st16_issue(a_lane + kSfb, v);
      tmem_wait_st();  // ordered before this warp's first arrive on a full barrier
    }
    const uint32_t row_sw = static_cast<uint32_t>(r & 7);
    uint32_t gbase = 0;  // groups (= boxes) of earlier tiles
    long long seen = -1; // latest group this warp has seen complete
    bool ok = true;
    for (int tile = tile_begin<false, true>(g), tstep = tile_step<false, true>(), tend = tile_end<false, true>(g);
         tile < tend && ok; tile += tstep) {
      for (int bt = 0; bt < nbx; ++bt) {
        const uint32_t gj = gbase + bt;
        const int cs = static_cast<int>(gj % kCodeRing);
        if (!warp_wait(&cfull[cs], (gj / kCodeRing) & 1u, g.status)) {
          ok = false;
          break;
        }
        const uint8_t* crow = smem + kCodeOff + cs * kCodeBox + r * 128;
#pragma unroll
        for (int s2 = 0; s2 < 2; ++s2) {
          const int st = 2 * half + s2;
          const uint32_t sg = gj * kG + st;  // stage index over this CTA's tiles
          // its A slot is free once the group of stage sg - kSlots is done
          if (sg >= static_cast<uint32_t>(kSlots)) {
            const uint32_t gp = (sg - kSlots) / kG;
            if (static_cast<long long>(gp) > seen) {
              if (!warp_wait(&empty[gp % kNQ], (gp / kNQ) & 1u, g.status)) {
                ok = false;
                break;
              }
              seen = gp;
              tc_fence_after();  // the MMAs that read the slot before are done
            }
          }
          const int c = 2 * st;  // the stage's two 16-byte chunks of the row
          const uint4 w0 = *reinterpret_cast<const uint4*>(crow + ((c ^ row_sw) << 4));
          const uint4 w1 = *reinterpret_cast<const uint4*>(crow + (((c + 1) ^ row_sw) << 4));
          const uint32_t acol = a_lane + kAcol0 + 32u * (sg % kSlots);
          expand_half_tmem(acol, w0);
          expand_half_tmem(acol + 16u, w1);
        }
        if (!ok) break;
        tmem_wait_st();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(&full[gj % kNQ]), 0));
          mbar_arrive(&cempty[cs]);  // this warp is done reading box gj
        }
      }
      gbase += nbx;
    }
  } else if (warp < kIss0Warp) {
    // ---------------------------------------------------------- drain
    // Warp 8 + w drains TMEM lane quarter w: d_u = d_A + d_B of the 64 query
    // columns into registers, release of both accumulators, then the scores
    // fl(fl(s_q s_i) d_u) (one module: fl(0 + term)) stored to the output.
    const int q4 = warp & 3;
    const int rr = q4 * 32 + lane;
    const int ep = (warp - kDrW0) * 32 + lane;  // drain thread 0 .. 127
    const uint32_t lane_base = static_cast<uint32_t>(q4 * 32) << 16;
    // one query tile (the launch checks it): its scales once, for every tile
    if (ep < kBN) sq[ep] = (ep < g.BNq && ep < g.Q) ? g.qs[static_cast<size_t>(ep) * g.ldqs] : 0.f;
    named_bar_sync(2, kDrW * 32);
    uint32_t tl = 0;  // tiles of this CTA so far
    for (int tile = tile_begin<false, true>(g), tstep = tile_step<false, true>(), tend = tile_end<false, true>(g);
         tile < tend; tile += tstep, ++tl) {
      const int i0 = tile_row0<true>(tile % g.n_it);
      const int row = i0 + rr;
      const float si = row < g.N ? g.ts[static_cast<size_t>(row) * g.ldts] : 0.f;
      uint32_t w_ok = 1;
      if (lane == 0) w_ok = mbar_wait(dfull, tl & 1u, g.status) ? 1u : 0u;
      w_ok = __shfl_sync(0xffffffffu, w_ok, 0);
      if (!w_ok) break;
      tc_fence_after();
      float d[kBN];
#pragma unroll
      for (int h = 0; h < kBN / 32; ++h) {
        uint32_t a[32], b[32];
        tmem_ld32_issue(tmem + lane_base + 32u * h, a);
        tmem_ld32_issue(tmem + lane_base + kBN + 32u * h, b);
        tmem_wait_ld(a);
        tmem_wait_ld(b);
#pragma unroll
        for (int j = 0; j < 32; ++j) d[32 * h + j] = __fadd_rn(__uint_as_float(a[j]), __uint_as_float(b[j]));
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(dempty), 0));  // the MMAs run on
      if (row < g.N) {
#pragma unroll
        for (int c = 0; c < kBN; ++c)
          if (c < g.BNq && c < g.Q)
            g.out[static_cast<size_t>(c) * g.ldo + row] = __fadd_rn(0.f, __fmul_rn(__fmul_rn(sq[c], si), d[c]));
      }
    }
  } else if (warp == kIss0Warp || warp == kIss1Warp) {
    if (lane == 0 && rank == 0) {
      // ---------------------------------------------------------- issuers (leader)
      // Issuer h runs stages 2h, 2h + 1 of every group into its own accumulator.
      const int half = warp == kIss0Warp ? 0 : 1;
      const uint32_t idesc = idesc_mxf4_f32(256, g.BNq);
      const uint32_t sfa = tmem + kSfa, sfb = tmem + kSfb;
      const uint32_t d = tmem + static_cast<uint32_t>(half * kBN);
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      constexpr uint64_t kGroupDesc = (static_cast<uint64_t>(kG) * kStage) >> 4;  // descriptor step per group
      uint64_t dq = dbase;             // query stages of query slot rq
      int rq = 0;
      uint32_t sa = 0;                 // A slot of the group's first stage (stage index % kSlots)
      uint32_t rph = 0, tl = 0;
      bool ok = true;
      for (int tile = tile_begin<false, true>(g), tstep = tile_step<false, true>(), tend = tile_end<false, true>(g);
           tile < tend && ok; tile += tstep, ++tl) {
        // both accumulators drained (the drain releases them together)
        if (!mbar_wait_cluster(dempty, (tl & 1u) ^ 1u, g.status)) break;
        tc_fence_after();
        for (int gi = 0; gi < nbx; ++gi) {
          const int s = rq;
          const uint32_t ph = rph;
          const uint64_t b0 = dq + ((2 * half * kStage) >> 4), b1 = b0 + (kStage >> 4);
          uint32_t s0 = sa + 2 * half, s1 = s0 + 1;
          if (s0 >= static_cast<uint32_t>(kSlots)) s0 -= kSlots;
          if (s1 >= static_cast<uint32_t>(kSlots)) s1 -= kSlots;
          const uint32_t a0 = tmem + kAcol0 + 32u * s0, a1 = tmem + kAcol0 + 32u * s1;
          if (++rq == kNQ) {
            rq = 0;
            rph ^= 1u;
            dq = dbase;
          } else {
            dq += kGroupDesc;
          }
          sa += kG;
          if (sa >= static_cast<uint32_t>(kSlots)) sa -= kSlots;
          // both CTAs' query bytes and expander warps
          if (!mbar_wait(&full[s], ph, g.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          issue_half(d, a0, a1, b0, b1, idesc, sfa, sfb, gi == 0);
          tc_commit_pair_mc(&empty[s], 0x3);
        }
        if (ok) tc_commit_pair_mc(dfull, 0x3);
      }
      // every MMA of this thread done before TMEM is released (also after a
      // timeout above)
      tc_commit_pair_mc(&fin[half], 0x1);
      mbar_wait(&fin[half], 0, g.status);
    }
    __syncwarp();
  } else if (warp == kCodeWarp) {
    // ---------------------------------------------------------- code producer
    if (lane == 0) {
      uint32_t gbase = 0;
      bool ok = true;
      for (int tile = tile_begin<false, true>(g), tstep = tile_step<false, true>(), tend = tile_end<false, true>(g);
           tile < tend && ok; tile += tstep) {
        const int i0 = tile_row0<true>(tile % g.n_it);
        for (int bt = 0; bt < nbx; ++bt) {
          const uint32_t b = gbase + bt;
          const int cs = static_cast<int>(b % kCodeRing);
          if (!mbar_wait(&cempty[cs], ((b / kCodeRing) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&cfull[cs], kCodeBox);
          tma_load_2d(smem + kCodeOff + cs * kCodeBox, &tmC, bt * kCodeBoxWords, i0, &cfull[cs]);
        }
        gbase += nbx;
      }
    }
    __syncwarp();
  } else if (warp == kQueryWarp) {
    // ---------------------------------------------------------- query producer
    // This CTA's half of the query rows of each stage of a group, as soon as both
    // issuers release the group; the bytes are counted on the leader's barrier.
    if (lane == 0) {
      const uint32_t qbytes = static_cast<uint32_t>(g.BNq / 2) * 128u;
      uint32_t gbase = 0;
      bool ok = true;
      for (int tile = tile_begin<false, true>(g), tstep = tile_step<false, true>(), tend = tile_end<false, true>(g);
           tile < tend && ok; tile += tstep) {
        const int qrow = (tile / g.n_it) * g.BNq + static_cast<int>(rank) * (g.BNq / 2);
        for (int bt = 0; bt < nbx; ++bt) {
          const uint32_t gj = gbase + bt;
          const int s = static_cast<int>(gj % kNQ);  // free once the MMAs of group gj - NQ are done
          if (!mbar_wait(&empty[s], ((gj / kNQ) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          const uint32_t fl = mapa_shared(smem_u32(&full[s]), 0);
          mbar_arrive_expect_tx_cluster(fl, kG * qbytes);
#pragma unroll
          for (int st = 0; st < kG; ++st)
            tma_load_2d_pair(smem_u32(smem + (s * kG + st) * kStage), &tmQ, (bt * kG + st) * 128, qrow, fl);
        }
        gbase += nbx;
      }
    }
    __syncwarp();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while its peer may still signal it
  tc_fence_after();
  if (warp == kIss0Warp) tmem_dealloc_pair(tmem, 512);
}

}  // namespace

size_t pair_ks_smem_need() { return 1024 + kSmemTotal; }

cudaError_t launch_pair_ks(const CUtensorMap& tq, const CUtensorMap& tc, const ScoreTcArgs& g, int grid,
                           cudaStream_t st) {
  // one module, one query tile of at most 64 queries, whole groups
  if (g.U != 1 || g.BNq > kBN || g.BNq % 32 || g.Q > g.BNq || g.D % (256 * kG)) return cudaErrorInvalidValue;
  const size_t smem = pair_ks_smem_need();
  cudaError_t e =
      cudaFuncSetAttribute(k_score_pair_ks, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, k_score_pair_ks, tq, tc, g);
}

}  // namespace sc
}  // namespace eogp
