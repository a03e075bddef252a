// One-bit (CODES) scoring with e2m1 operands on CTA pairs (Sec. 3.3 Eq.
// onebit_influence; App. B.3 scan): k_score_pair.
//
// A pair works on 256 stored rows (MMA M = 256, tcgen05 cta_group::2): each
// CTA expands its own 128 rows into its own TMEM (operand A) and loads its own
// half of the tile's queries (operand B, BNq / 2 rows per CTA, no multicast);
// the leader CTA (rank 0) issues the MMAs, whose accumulator rows land in each
// CTA's TMEM, so each CTA dequantises its own rows exactly as the one-CTA
// kernel does (dequant_role). Against one CTA per 128-row tile this halves the
// query operand's stream from L2 per stored row.
//
// The +-1 values are e2m1 (+1 = 0x2, -1 = 0xA) multiplied by kind::mxf4 with
// every block scale 1 (ue8m0 0x7F), K = 64 per MMA: products and partial sums
// are small integers, so d_u is exact and the scores are bitwise identical to
// the popcount kernels and the oracle's float32 evaluation.
//
// Rings:
//  * code boxes (shared memory, 4 to 8 x 16 KB): 128 rows x 1024 code bits,
//    128-byte swizzle, loaded by TMA by a producer warp as far ahead as the
//    ring allows, so HBM latency is hidden by the ring rather than by registers;
//  * pipeline groups of G 256-bit stages: per stage a query operand tile in
//    shared memory (BNq / 2 rows x 128 bytes, loaded by a second producer warp)
//    and an A slot of 32 TMEM columns (the expanded stored rows). One barrier
//    pair per group: the MMA issuer waits once, issues 4 G MMAs and commits
//    once. The query tiles sit in a deeper ring (NQ groups) than the A slots
//    (NG groups, all TMEM leaves): the query stages of group gj are loaded once
//    group gj - NQ is done, its A slots refilled once group gj - NG is done,
//    both read from the one commit per group, so the queries' L2 latency is off
//    the A slots' round trip.
//  * issuing threads: a thread issues an MMA about every 64 cycles whatever N
//    is, plus ~330 cycles per wait-fence-commit round: at 256 bits per round
//    the rounds, not the tensor pipe, set the pace (measured: 589 cycles per
//    four N = 256 MMAs, 8.4 of 9.7 PFLOP/s), at 512 bits the tensor pipe does
//    (1024 cycles per eight, 9.7 PFLOP/s). An N = 64 MMA takes as long to issue
//    as an N = 128 one, so 64-query tiles take four stages per group (and one
//    module of 64 queries has its own two-issuer kernel, k_score_pair_ks.cu).
//    128-query tiles of several modules have two accumulators and two issuers,
//    issuer b running the modules of accumulator b, so one thread's rounds
//    overlap the other's MMAs. Groups then complete out of order, which the
//    lagged reuse allows as long as no thread waits on a barrier phase before
//    it has seen the previous phase of that barrier complete (a parity wait
//    cannot tell a phase from the one two ahead): the expanders and the query
//    producer wait on every group's empty barrier in order, and both issuers
//    wait on every group's full barrier in order, issuing only their own. (An
//    earlier version whose issuers waited only on their own groups' barriers
//    passed a phase early and faulted the GPU, Xid 13, on the 4.2M-code scan.)
// Each expander warp takes the 32 rows of one TMEM lane quarter, a whole group
// per round: two 16-byte shared-memory loads and the e2m1 expansion per stage,
// the TMEM stores, and one relaxed arrive on the leader's barrier of the group. That arrive orders enough: it is issued after
// tcgen05.wait::st, which returns only once the thread's TMEM stores have
// completed, and after the tcgen05 fence; the leader issues the MMAs only after
// observing it; and in the pair MMA each SM's tensor core reads operand A from
// its own CTA's TMEM, which no cache sits in front of. (The pair rotation
// kernel releases its accumulators the same way.) Measured on the scan at
// Q = 1024: 23.0 ms with relaxed arrives, 30.0 ms with CTA-scope release,
// 30.9 ms with cluster-scope release, 44.8 ms with one thread of the peer
// forwarding every stage with one cluster-scope release.
//
// Warps: 0-3 expand, 4-11 dequantise (two per TMEM lane quarter, half of the
// query columns each, which halves the drain of the accumulator the MMAs of a
// 256-query tile wait for), 12 owns TMEM and, in the leader, issues the MMAs
// (of accumulator 0 with two issuers), 13 loads the code boxes, 14 the query
// tiles, 15 is the second issuer. Sixteen warps leave 128 registers a thread.
#include <algorithm>
#include <atomic>

#include "score_tc.cuh"

namespace eogp {
namespace sc {
namespace {

constexpr int kPrExpWarps = 4;                   // expander warps: one per TMEM lane quarter
constexpr int kPrDq0 = kPrExpWarps;              // first dequantise warp
constexpr int kPrDqWarps = 8;                    // dequantise warps: two per TMEM lane quarter
constexpr int kPrMmaWarp = kPrDq0 + kPrDqWarps;
constexpr int kCodeWarp = kPrMmaWarp + 1;
constexpr int kQueryWarp = kPrMmaWarp + 2;
constexpr int kIss1Warp = kPrMmaWarp + 3;         // second MMA issuer (two accumulators of several modules)
constexpr int kPairThreads = (kIss1Warp + 1) * 32;
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
constexpr int pr_slots() {
  return (512 - pr_dbufs<BN>() * BN - 32) / 32;
}
// Only 128-query tiles serve several modules (a running score, kept in the
// dequantise warps' registers); 64-query tiles serve one (their TMEM has no
// room for a second accumulator pair), and 256-query tiles keep one
// accumulator.
template <int BN>
constexpr bool pr_running() {
  return BN == 128;
}
// Code boxes in flight and query stages: as many as the shared memory holds.
template <int BN>
constexpr int pr_code_ring() {
  return BN == 64 ? 8 : BN == 256 ? 3 : 4;
}
// (16 with 128-query tiles: a multiple of 2 G x the groups of a module, so
// each query-stage slot serves one issuer only, for modules of up to 2048 bits.)
template <int BN>
constexpr int pr_qstages() {
  return BN == 64 ? 20 : BN == 256 ? 10 : 16;
}
// MMA-issuing threads: two with two accumulators of several modules (each
// issues the modules of one accumulator), else one.
template <int BN>
constexpr int pr_issuers() {
  return pr_dbufs<BN>() == 2 && pr_running<BN>() ? 2 : 1;
}
template <int BN>
constexpr uint32_t pr_acol0() {
  return static_cast<uint32_t>(pr_dbufs<BN>() * BN);
}
template <int BN>
constexpr uint32_t pr_sf_col() {
  return pr_acol0<BN>() + 32u * static_cast<uint32_t>(pr_slots<BN>());
}

// Shared memory: the query ring, the code ring, then the layout the dequantise
// role shares with the one-CTA kernel.
template <bool TOPK, int BN, int G>
__host__ __device__ inline TcSmem pr_smem_layout(uint32_t* code_off) {
  constexpr int NQ = pr_qstages<BN>() / G, kCodeRing = pr_code_ring<BN>();
  constexpr uint32_t kStage = static_cast<uint32_t>(BN / 2) * 128u;
  TcSmem l;
  *code_off = NQ * G * kStage;
  l.acc = *code_off + kCodeRing * kCodeBox;
  l.sq = l.acc;  // no running score in shared memory
  l.bars = l.sq + 2 * BN * 4;
  l.lists = l.bars + (2 * NQ + 2 * pr_dbufs<BN>() + 2 * kCodeRing) * 8 + 16;
  l.total = l.lists + (TOPK ? BN * 12 + 8 * 4 * 4 : 0);
  return l;
}

template <bool TOPK, int BN, int G>
__global__ void __launch_bounds__(kPairThreads, 1)
    k_score_pair(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmC,
                 const __grid_constant__ ScoreTcArgs g) {
  constexpr int NG = pr_slots<BN>() / G;      // groups of A slots in TMEM
  constexpr int NQ = pr_qstages<BN>() / G;    // groups of query stages in shared memory
  constexpr int ND = pr_dbufs<BN>();
  constexpr int kCodeRing = pr_code_ring<BN>();
  constexpr uint32_t kStage = static_cast<uint32_t>(BN / 2) * 128u;
  constexpr uint32_t kSfa = pr_sf_col<BN>(), kSfb = kSfa + 16u;
  static_assert(kSfb + 16u <= 512u, "TMEM budget");
  static_assert(NG >= 2 && NQ >= NG, "rings: at least two A groups, at least as many query groups");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint32_t code_off;
  const TcSmem L = pr_smem_layout<TOPK, BN, G>(&code_off);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  float* sq = reinterpret_cast<float*>(smem + L.sq);
  // group gj: full / empty barrier gj % NQ, query stages of slot gj % NQ, A
  // slots of slot gj % NG
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + L.bars);
  uint64_t* empty = full + NQ;
  uint64_t* dfull = empty + NQ;
  uint64_t* dempty = dfull + ND;
  uint64_t* cfull = dempty + ND;
  uint64_t* cempty = cfull + kCodeRing;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(cempty + kCodeRing);
  const int nst = g.D / 256;            // 256-bit stages per tile (a multiple of G)
  const int nbx = (nst + 3) / 4;        // code boxes per tile

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmC);
    for (int s = 0; s < NQ; ++s) {
      // leader's copy: per CTA the query producer's expect_tx arrive (+ its TMA
      // bytes) and the four expander warps
      mbar_init(&full[s], 2 * (1 + kPrExpWarps));
      mbar_init(&empty[s], 1);  // MMA completion of the group, multicast to both CTAs
    }
    for (int b = 0; b < ND; ++b) {
      mbar_init(&dfull[b], 1);   // multicast to both CTAs
      mbar_init(&dempty[b], 2 * kPrDqWarps);  // every dequantise warp of both CTAs (leader's copy)
    }
    for (int b = 0; b < kCodeRing; ++b) {
      mbar_init(&cfull[b], 1);           // the producer's expect_tx arrive (+ TMA bytes)
      mbar_init(&cempty[b], kPrExpWarps);  // every expander warp, once per box
    }
    fence_barrier_init();
  }
  if (warp == kPrMmaWarp) tmem_alloc_pair(tslot, 512);
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers initialised before any remote arrive
  tc_fence_after();
  const uint32_t tmem = *tslot;

  if (warp < kPrExpWarps) {
    // ---------------------------------------------------------- expanders
    // Warp w expands the rows of TMEM lane quarter w, a whole group (G stages,
    // 32 G columns) per round: wait for the group's slots, two 16-byte loads and
    // 32 e2m1 columns per stage, one tcgen05.wait::st, one arrive.
    const int r = warp * 32 + lane;  // stored row in the CTA's tile = TMEM lane
    const uint32_t a_lane = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    {  // unit scale factors (ue8m0 0x7F = 1.0) of A and B, once
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
        // groups never cross a box: a box holds four stages, a group G of 1, 2 or 4
        for (int sub = 0; sub < 4 && 4 * bt + sub < nst; sub += G) {
          const uint32_t gj = (it + 4 * bt + sub) / G;
          const int rp = static_cast<int>(gj % NG);
          // the A slots are free once the MMAs of group gj - NG are done
          if (gj >= NG) {
            const uint32_t gp = gj - NG;
            if (!warp_wait(&empty[gp % NQ], (gp / NQ) & 1u, g.status)) {
              ok = false;
              break;
            }
          }
          tc_fence_after();  // the MMAs that read the slots before are done
#pragma unroll
          for (int st = 0; st < G; ++st) {
            const int c = 2 * (sub + st);  // the stage's two 16-byte chunks of the row
            const uint4 w0 = *reinterpret_cast<const uint4*>(crow + ((c ^ row_sw) << 4));
            const uint4 w1 = *reinterpret_cast<const uint4*>(crow + (((c + 1) ^ row_sw) << 4));
            const uint32_t acol = a_lane + pr_acol0<BN>() + 32u * static_cast<uint32_t>(rp * G + st);
            expand_half_tmem(acol, w0);
            expand_half_tmem(acol + 16u, w1);
          }
          tmem_wait_st();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_relaxed_cluster(mapa_shared(smem_u32(&full[gj % NQ]), 0));
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&cempty[cs]);  // this warp is done reading box b
      }
      it += nst;
      bx += nbx;
    }
  } else if (warp < kPrMmaWarp) {
    dequant_role<EOGP_SCORE_CODES, TOPK, BN, ND, pr_running<BN>(), true, kPrDqWarps, kPrDq0>(g, smem, L, tmem, sq,
                                                                                              dfull, dempty);
  } else if (warp == kPrMmaWarp || warp == kIss1Warp) {
    constexpr int NI = pr_issuers<BN>();
    const int me = warp == kPrMmaWarp ? 0 : 1;
    if (lane == 0 && rank == 0 && me < NI) {
      // ---------------------------------------------------------- MMA issuers (leader)
      // Kept to waits, MMAs and commits. With two issuers, issuer b runs the
      // modules of accumulator b and only the owner of a group issues and
      // commits it. Every thread must see each phase of a barrier it waits on:
      // when all modules have the same number of groups ng and NQ is a multiple
      // of 2 ng, the groups of a full barrier all belong to one issuer, which
      // waits only on its own; otherwise both wait on every group's full
      // barrier in order.
      const uint32_t idesc = idesc_mxf4_f32(256, g.BNq);
      const uint32_t sfa = tmem + kSfa, sfb = tmem + kSfb;
      const uint64_t dbase = sdesc_sw128(smem_u32(smem), 16, 1024);
      constexpr uint64_t kGroupDesc = (static_cast<uint64_t>(G) * kStage) >> 4;  // descriptor step per group
      uint64_t dq = dbase;                   // query stages of query slot rq
      uint32_t acl = tmem + pr_acol0<BN>();  // A slots of A slot ra
      int rq = 0, ra = 0;
      uint32_t rph = 0, gm = 0;
      bool ok = true;
      const int ngu = g.kuni / (256 * G);  // groups of every module (0: modules differ)
      const bool excl = NI == 2 && ngu > 0 && NQ % (2 * ngu) == 0;
      // one group on: query slot rq (phase rph, descriptor dq), A slot ra (columns acl)
      auto advance = [&]() {
        if (++rq == NQ) {
          rq = 0;
          rph ^= 1u;
          dq = dbase;
        } else {
          dq += kGroupDesc;
        }
        if (++ra == NG) {
          ra = 0;
          acl = tmem + pr_acol0<BN>();
        } else {
          acl += 32u * G;
        }
      };
      for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
           tile < tend && ok; tile += tstep) {
        for (int u = 0; u < g.U && ok; ++u, ++gm) {
          const int buf = static_cast<int>(gm % ND);
          const bool mine = NI == 1 || buf == me;
          if (!mine && excl) {  // the other issuer's module: its slots, not its barriers
            for (int gi = 0; gi < ngu; ++gi) advance();
            continue;
          }
          if (mine) {
            if (!mbar_wait_cluster(&dempty[buf], ((gm / ND) & 1u) ^ 1u, g.status)) {
              ok = false;
              break;
            }
            tc_fence_after();
          }
          const uint32_t d = tmem + buf * static_cast<uint32_t>(BN);
          const int ngr = g.k[u] / (256 * G);
          for (int gi = 0; gi < ngr; ++gi) {
            const int s = rq;
            const uint32_t ph = rph;
            const uint64_t b0 = dq;
            const uint32_t at0 = acl;
            advance();
            // both CTAs' query bytes and expander warps (the MMAs read the
            // queries through the async proxy, tracked by the barrier's
            // transaction count)
            if (!mbar_wait(&full[s], ph, g.status)) {
              ok = false;
              break;
            }
            if (!mine) continue;
            tc_fence_after();
#pragma unroll
            for (int st = 0; st < G; ++st)
#pragma unroll
              for (int kk = 0; kk < 4; ++kk)
                tc_mma_f4_ta_pair(d, at0 + 32u * st + 8u * kk, b0 + ((st * kStage) >> 4) + 2 * kk, idesc, sfa,
                                  sfb, (gi | st | kk) != 0 ? 1u : 0u);
            tc_commit_pair_mc(&empty[s], 0x3);
          }
          if (mine && ok) tc_commit_pair_mc(&dfull[buf], 0x3);
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
    // This CTA's half of the query rows of each stage of a group, as soon as the
    // MMAs release the group; the bytes are counted on the leader's barrier.
    if (lane == 0) {
      const uint32_t qbytes = static_cast<uint32_t>(g.BNq / 2) * 128u;
      uint32_t it = 0;
      bool ok = true;
      for (int tile = tile_begin<TOPK, true>(g), tstep = tile_step<TOPK, true>(), tend = tile_end<TOPK, true>(g);
           tile < tend && ok; tile += tstep) {
        const int qrow = (tile / g.n_it) * g.BNq + static_cast<int>(rank) * (g.BNq / 2);
        for (int jt = 0; jt < nst; jt += G) {
          const uint32_t gj = (it + jt) / G;
          const int s = static_cast<int>(gj % NQ);  // free once the MMAs of group gj - NQ are done
          if (!mbar_wait(&empty[s], ((gj / NQ) & 1u) ^ 1u, g.status)) {
            ok = false;
            break;
          }
          const uint32_t fl = mapa_shared(smem_u32(&full[s]), 0);
          mbar_arrive_expect_tx_cluster(fl, G * qbytes);
#pragma unroll
          for (int st = 0; st < G; ++st)
            tma_load_2d_pair(smem_u32(smem + (s * G + st) * kStage), &tmQ, (jt + st) * 128, qrow, fl);
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
  if (warp == kPrMmaWarp) tmem_dealloc_pair(tmem, 512);
}

template <bool TOPK, int BN, int G>
size_t smem_need() {
  uint32_t code_off;
  return 1024 + pr_smem_layout<TOPK, BN, G>(&code_off).total;
}

template <bool TOPK, int BN, int G>
cudaError_t launch(const CUtensorMap& tq, const CUtensorMap& tc, const ScoreTcArgs& g, int grid, cudaStream_t st) {
  const size_t smem = smem_need<TOPK, BN, G>();
  cudaError_t e = cudaFuncSetAttribute(k_score_pair<TOPK, BN, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
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
  return cudaLaunchKernelEx(&cfg, k_score_pair<TOPK, BN, G>, tq, tc, g);
}

template <bool TOPK>
cudaError_t launch_bn(int BN, int G, const CUtensorMap& tq, const CUtensorMap& tc, const ScoreTcArgs& g, int grid,
                      cudaStream_t st) {
  if (BN == 256) return G == 2 ? launch<TOPK, 256, 2>(tq, tc, g, grid, st) : launch<TOPK, 256, 1>(tq, tc, g, grid, st);
  if (BN == 128) return G == 2 ? launch<TOPK, 128, 2>(tq, tc, g, grid, st) : launch<TOPK, 128, 1>(tq, tc, g, grid, st);
  if (G == 4) return launch<TOPK, 64, 4>(tq, tc, g, grid, st);
  return G == 2 ? launch<TOPK, 64, 2>(tq, tc, g, grid, st) : launch<TOPK, 64, 1>(tq, tc, g, grid, st);
}

}  // namespace

size_t pair_smem_need(int BN, int G, bool topk) {
  if (topk) {
    if (BN == 256) return G == 2 ? smem_need<true, 256, 2>() : smem_need<true, 256, 1>();
    if (BN == 128) return G == 2 ? smem_need<true, 128, 2>() : smem_need<true, 128, 1>();
    return G == 4 ? smem_need<true, 64, 4>() : G == 2 ? smem_need<true, 64, 2>() : smem_need<true, 64, 1>();
  }
  if (BN == 256) return G == 2 ? smem_need<false, 256, 2>() : smem_need<false, 256, 1>();
  if (BN == 128) return G == 2 ? smem_need<false, 128, 2>() : smem_need<false, 128, 1>();
  return G == 4 ? smem_need<false, 64, 4>() : G == 2 ? smem_need<false, 64, 2>() : smem_need<false, 64, 1>();
}

int pair_cluster_cap(int num_sms) {
  static std::atomic<int> cache[128];
  int dev = 0;
  const int fallback = std::max(1, num_sms / 2);
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return fallback;
  int v = cache[dev].load(std::memory_order_relaxed);
  if (v > 0) return v;
  const size_t smem = smem_need<true, 128, 1>();
  if (cudaFuncSetAttribute(k_score_pair<true, 128, 1>, cudaFuncAttributeMaxDynamicSharedMemorySize,
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
  if (cudaOccupancyMaxActiveClusters(&n, k_score_pair<true, 128, 1>, &cfg) != cudaSuccess || n < 1) {
    cudaGetLastError();
    return fallback;
  }
  v = std::min(n, fallback);
  cache[dev].store(v, std::memory_order_relaxed);
  return v;
}

cudaError_t launch_pair(int BN, int G, bool topk, const CUtensorMap& tq, const ScoreTcArgs& g, int grid,
                        cudaStream_t st) {
  if (BN != 64 && BN != 128 && BN != 256) return cudaErrorInvalidValue;
  if (G != 1 && G != 2 && !(G == 4 && BN == 64)) return cudaErrorInvalidValue;
  if (BN == 256 && g.U != 1) return cudaErrorInvalidValue;  // 256-query tiles keep no running score
  if (BN == 64 && g.U != 1) return cudaErrorInvalidValue;   // 64-query tiles keep no running score
  for (int u = 0; u < g.U; ++u)
    if (g.k[u] % (256 * G)) return cudaErrorInvalidValue;  // groups never straddle modules
  // stored code rows: boxes of 32 words (1024 bits) x 128 rows, 128-byte swizzle
  CUtensorMap tc;
  const uint64_t cdims[2] = {static_cast<uint64_t>(g.D / 32), static_cast<uint64_t>(g.N)};
  const uint64_t cstr[1] = {static_cast<uint64_t>(g.ldt) * 4};
  const uint32_t cbox[2] = {static_cast<uint32_t>(kCodeBoxWords), 128};
  if (make_tmap(&tc, CU_TENSOR_MAP_DATA_TYPE_UINT32, 2, g.train, cdims, cstr, cbox, CU_TENSOR_MAP_SWIZZLE_128B))
    return cudaErrorInvalidValue;
  // 64 queries of one module in whole 1024-bit groups: two MMA-issuing threads
  if (!topk && BN == 64 && G == 4 && g.Q <= g.BNq) return launch_pair_ks(tq, tc, g, grid, st);
  return topk ? launch_bn<true>(BN, G, tq, tc, g, grid, st) : launch_bn<false>(BN, G, tq, tc, g, grid, st);
}

}  // namespace sc
}  // namespace eogp
