// Influence scoring against stored one-bit codes (Sec. 3.3, Eq. onebit_influence;
// App. B.3, Eq. app_stored_influence; scan cost Eq. app_scan_complexity).
//
// CODES mode (both sides one-bit): for module u with k_u coordinates the +-1
// inner product is k_u - 2 popc(b_i xor b_q), an exact integer. The score is
// dequantised in a fixed fp32 order: acc = fl(acc + fl(fl(s_qu * s_iu) * d_u))
// over modules in order, with explicit round-to-nearest intrinsics so no fused
// multiply-add changes the result: bitwise reproducible.
//
// PAPER mode (query unquantised): sum_u s_iu <y_u, b_iu> with b in {+-1}.
//
// Kernels:
//  k_score_codes_smallq<QT>: Q <= 8 queries; one thread per stored row, query
//    words broadcast from shared memory; stored codes staged through shared
//    memory with coalesced 128-byte row loads. This is the HBM-bound scan.
//  k_score_codes_tiled: 64 stored rows x 64 queries per block, 4 x 4 per thread.
//  k_score_paper_tiled: same tiling, one 32-coordinate word per step.
#include "eogp_dev.cuh"
#include "eogp_internal.h"

namespace {

constexpr int kMaxU = 1024;

struct ModInfo {
  int U;
  int k[kMaxU];
  int off[kMaxU + 1];  // word offsets (CODES) or coordinate offsets (PAPER y)
  int coff[kMaxU + 1];
};

// Chunk c of the stored rows' words: module u, words [wc, wc + nw) of it.
struct Chunk {
  int u, wc, nw;
};

__device__ __forceinline__ bool next_chunk(const ModInfo& mi, Chunk& c) {
  const int wu = mi.off[c.u + 1] - mi.off[c.u];
  if (c.wc + 32 < wu) {
    c.wc += 32;
  } else {
    ++c.u;
    c.wc = 0;
    if (c.u >= mi.U) return false;
  }
  c.nw = min(32, mi.off[c.u + 1] - mi.off[c.u] - c.wc);
  return true;
}

// Stored rows are staged 256 rows x 32 words at a time in shared memory; the
// next chunk's words are loaded into registers (128-bit loads) while the
// current chunk is counted, so loads stay in flight during the popcounts.
// vec requires every module's word count, ldt and the base to be multiples of
// 4 words / 16 bytes.
template <int QT>
__global__ void __launch_bounds__(256) k_score_codes_smallq(
    const uint32_t* __restrict__ train, int ldt, const float* __restrict__ ts, int ldts, int N,
    const __grid_constant__ ModInfo mi, const uint32_t* __restrict__ query, int ldq,
    const float* __restrict__ qs, int ldqs, int Q, float* __restrict__ out, int ldo, int vec) {
  __shared__ uint32_t Ts[256][33];
  __shared__ uint32_t Qw[QT][32];
  const int tid = threadIdx.x;
  const int i0 = blockIdx.x * 256;
  const int q0 = blockIdx.y * QT;
  const int i = i0 + tid;
  float acc[QT];
  int cnt[QT];
#pragma unroll
  for (int a = 0; a < QT; ++a) {
    acc[a] = 0.f;
    cnt[a] = 0;
  }
  // vector loader: iteration r covers rows r*32 + tid/8, words (tid%8)*4 .. +3
  const int lrow = tid >> 3, lword = (tid & 7) * 4;
  uint4 pre[8];
  auto issue = [&](const Chunk& c) {
    const int base = mi.off[c.u] + c.wc;
#pragma unroll
    for (int r = 0; r < 8; ++r) {
      const int row = i0 + r * 32 + lrow;
      pre[r] = make_uint4(0, 0, 0, 0);
      if (row < N && lword < c.nw)
        pre[r] = __ldcs(reinterpret_cast<const uint4*>(train + static_cast<size_t>(row) * ldt + base + lword));
    }
  };
  Chunk cur{0, 0, min(32, mi.off[1] - mi.off[0])};
  if (vec) issue(cur);
  for (;;) {
    if (vec) {
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        uint32_t* d = &Ts[r * 32 + lrow][lword];
        d[0] = pre[r].x;
        d[1] = pre[r].y;
        d[2] = pre[r].z;
        d[3] = pre[r].w;
      }
    } else {
      const int base = mi.off[cur.u] + cur.wc;
#pragma unroll 8
      for (int r = 0; r < 32; ++r) {
        const int e = tid + 256 * r;
        const int row = e >> 5, w = e & 31;
        uint32_t v = 0;
        if (i0 + row < N && w < cur.nw) v = __ldcs(train + static_cast<size_t>(i0 + row) * ldt + base + w);
        Ts[row][w] = v;
      }
    }
    if (tid < QT * 32) {
      const int a = tid >> 5, w = tid & 31;
      uint32_t v = 0;
      if (q0 + a < Q && w < cur.nw) v = query[static_cast<size_t>(q0 + a) * ldq + mi.off[cur.u] + cur.wc + w];
      Qw[a][w] = v;
    }
    __syncthreads();
    Chunk nxt = cur;
    const bool more = next_chunk(mi, nxt);
    if (more && vec) issue(nxt);
    for (int w = 0; w < cur.nw; ++w) {
      const uint32_t t = Ts[tid][w];
#pragma unroll
      for (int a = 0; a < QT; ++a) cnt[a] += __popc(t ^ Qw[a][w]);
    }
    const bool module_done = !more || nxt.u != cur.u;
    if (module_done) {
      if (i < N) {
        const float si = ts[static_cast<size_t>(i) * ldts + cur.u];
#pragma unroll
        for (int a = 0; a < QT; ++a) {
          if (q0 + a < Q) {
            const float sq = qs[static_cast<size_t>(q0 + a) * ldqs + cur.u];
            const float d = static_cast<float>(mi.k[cur.u] - 2 * cnt[a]);
            acc[a] = __fadd_rn(acc[a], __fmul_rn(__fmul_rn(sq, si), d));
          }
        }
      }
#pragma unroll
      for (int a = 0; a < QT; ++a) cnt[a] = 0;
    }
    __syncthreads();
    if (!more) break;
    cur = nxt;
  }
  if (i < N) {
#pragma unroll
    for (int a = 0; a < QT; ++a)
      if (q0 + a < Q) out[static_cast<size_t>(q0 + a) * ldo + i] = acc[a];
  }
}

__global__ void __launch_bounds__(256) k_score_codes_tiled(
    const uint32_t* __restrict__ train, int ldt, const float* __restrict__ ts, int ldts, int N,
    const __grid_constant__ ModInfo mi, const uint32_t* __restrict__ query, int ldq,
    const float* __restrict__ qs, int ldqs, int Q, float* __restrict__ out, int ldo) {
  __shared__ uint32_t Ts[64][33];
  __shared__ uint32_t Qs[64][33];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int i0 = blockIdx.x * 64, q0 = blockIdx.y * 64;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

  for (int u = 0; u < mi.U; ++u) {
    const int w0 = mi.off[u], wu = mi.off[u + 1] - w0;
    int cnt[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) cnt[a][b] = 0;
    for (int wc = 0; wc < wu; wc += 32) {
      const int nw = min(32, wu - wc);
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const int e = tid + 256 * r;
        const int row = e >> 5, w = e & 31;
        uint32_t tv = 0, qv = 0;
        if (w < nw) {
          if (i0 + row < N) tv = train[static_cast<size_t>(i0 + row) * ldt + w0 + wc + w];
          if (q0 + row < Q) qv = query[static_cast<size_t>(q0 + row) * ldq + w0 + wc + w];
        }
        Ts[row][w] = tv;
        Qs[row][w] = qv;
      }
      __syncthreads();
      for (int w = 0; w < nw; ++w) {
        uint32_t t[4], q[4];
#pragma unroll
        for (int a = 0; a < 4; ++a) t[a] = Ts[tx + 16 * a][w];
#pragma unroll
        for (int b = 0; b < 4; ++b) q[b] = Qs[ty + 16 * b][w];
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
          for (int b = 0; b < 4; ++b) cnt[a][b] += __popc(t[a] ^ q[b]);
      }
      __syncthreads();
    }
    float si[4], sq[4];
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + tx + 16 * a;
      si[a] = i < N ? ts[static_cast<size_t>(i) * ldts + u] : 0.f;
    }
#pragma unroll
    for (int b = 0; b < 4; ++b) {
      const int q = q0 + ty + 16 * b;
      sq[b] = q < Q ? qs[static_cast<size_t>(q) * ldqs + u] : 0.f;
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) {
        const float d = static_cast<float>(mi.k[u] - 2 * cnt[a][b]);
        acc[a][b] = __fadd_rn(acc[a][b], __fmul_rn(__fmul_rn(sq[b], si[a]), d));
      }
  }
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const int q = q0 + ty + 16 * b;
    if (q >= Q) continue;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + tx + 16 * a;
      if (i < N) out[static_cast<size_t>(q) * ldo + i] = acc[a][b];
    }
  }
}

__global__ void __launch_bounds__(256) k_score_paper_tiled(
    const uint32_t* __restrict__ train, int ldt, const float* __restrict__ ts, int ldts, int N,
    const __grid_constant__ ModInfo mi, const float* __restrict__ y, int ldy, int Q,
    float* __restrict__ out, int ldo) {
  __shared__ uint32_t Tw[64];
  __shared__ float Ys[64][33];
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int i0 = blockIdx.x * 64, q0 = blockIdx.y * 64;
  float acc[4][4];
#pragma unroll
  for (int a = 0; a < 4; ++a)
#pragma unroll
    for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

  for (int u = 0; u < mi.U; ++u) {
    const int w0 = mi.off[u], ku = mi.k[u], c0 = mi.coff[u];
    float dot[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
      for (int b = 0; b < 4; ++b) dot[a][b] = 0.f;
    for (int wc = 0; wc * 32 < ku; ++wc) {
      const int nc = min(32, ku - wc * 32);
      if (tid < 64) {
        const int i = i0 + tid;
        Tw[tid] = i < N ? train[static_cast<size_t>(i) * ldt + w0 + wc] : 0u;
      }
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const int e = tid + 256 * r;
        const int q = e >> 5, c = e & 31;
        float v = 0.f;
        if (q0 + q < Q && c < nc) v = y[static_cast<size_t>(q0 + q) * ldy + c0 + wc * 32 + c];
        Ys[q][c] = v;
      }
      __syncthreads();
      uint32_t t[4];
#pragma unroll
      for (int a = 0; a < 4; ++a) t[a] = Tw[tx + 16 * a];
      for (int c = 0; c < nc; ++c) {
        float yv[4];
#pragma unroll
        for (int b = 0; b < 4; ++b) yv[b] = Ys[ty + 16 * b][c];
#pragma unroll
        for (int a = 0; a < 4; ++a) {
          // +1.0f for a set bit, -1.0f otherwise.
          const float sg = __uint_as_float(0x3f800000u | ((~(t[a] >> c) & 1u) << 31));
#pragma unroll
          for (int b = 0; b < 4; ++b) dot[a][b] = fmaf(yv[b], sg, dot[a][b]);
        }
      }
      __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + tx + 16 * a;
      const float si = i < N ? ts[static_cast<size_t>(i) * ldts + u] : 0.f;
#pragma unroll
      for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(si, dot[a][b], acc[a][b]);
    }
  }
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const int q = q0 + ty + 16 * b;
    if (q >= Q) continue;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
      const int i = i0 + tx + 16 * a;
      if (i < N) out[static_cast<size_t>(q) * ldo + i] = acc[a][b];
    }
  }
}

bool fill_modinfo(ModInfo& mi, const int* ks, int U) {
  if (U < 1 || U > kMaxU) return false;
  mi.U = U;
  mi.off[0] = 0;
  mi.coff[0] = 0;
  for (int u = 0; u < U; ++u) {
    mi.k[u] = ks[u];
    mi.off[u + 1] = mi.off[u] + (ks[u] + 31) / 32;
    mi.coff[u + 1] = mi.coff[u] + ks[u];
  }
  return true;
}

}  // namespace

cudaError_t launch_score_codes(const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                               const int* ks, int U, const uint32_t* query, int ldq,
                               const float* qs, int ldqs, int Q, float* out, int ldo,
                               cudaStream_t st) {
  ModInfo local;  // passed by value: kernel parameters are copied at launch
  if (!fill_modinfo(local, ks, U)) return cudaErrorInvalidValue;
  if (N <= 0 || Q <= 0) return cudaSuccess;
  if (Q <= 8) {
    const int qt = Q <= 1 ? 1 : Q <= 2 ? 2 : Q <= 4 ? 4 : 8;
    dim3 grid((N + 255) / 256, (Q + qt - 1) / qt);
    int vec = ((ldt & 3) == 0) && ((reinterpret_cast<uintptr_t>(train) & 15) == 0);
    for (int u = 0; u < U; ++u) vec &= (((ks[u] + 31) / 32) % 4) == 0;
    switch (qt) {
      case 1: k_score_codes_smallq<1><<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, query, ldq, qs, ldqs, Q, out, ldo, vec); break;
      case 2: k_score_codes_smallq<2><<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, query, ldq, qs, ldqs, Q, out, ldo, vec); break;
      case 4: k_score_codes_smallq<4><<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, query, ldq, qs, ldqs, Q, out, ldo, vec); break;
      default: k_score_codes_smallq<8><<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, query, ldq, qs, ldqs, Q, out, ldo, vec); break;
    }
  } else {
    dim3 grid((N + 63) / 64, (Q + 63) / 64);
    k_score_codes_tiled<<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, query, ldq, qs, ldqs,
                                              Q, out, ldo);
  }
  return cudaGetLastError();
}

cudaError_t launch_score_paper(const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                               const int* ks, int U, const float* y, int ldy, int Q, float* out,
                               int ldo, cudaStream_t st) {
  ModInfo local;
  if (!fill_modinfo(local, ks, U)) return cudaErrorInvalidValue;
  if (N <= 0 || Q <= 0) return cudaSuccess;
  dim3 grid((N + 63) / 64, (Q + 63) / 64);
  k_score_paper_tiled<<<grid, 256, 0, st>>>(train, ldt, ts, ldts, N, local, y, ldy, Q, out, ldo);
  return cudaGetLastError();
}
