// Throughput probes for the scoring rooflines: the dense tensor-core rates of
// the two +-1 scoring MMAs, tcgen05.mma kind::f8f6f4 (e4m3) and kind::mxf4
// (e2m1 with unit ue8m0 scales), and the integer XOR + popcount rate of the
// CUDA cores (the popcount scoring kernels). None is among the measured
// copy / bf16 GEMM peaks.
//
// MMA probes: one CTA per SM; one thread issues back-to-back M = 128, N = 256
// MMAs (K = 32 e4m3 or K = 64 e2m1) from two fixed shared-memory operand tiles,
// committing to an mbarrier every 64 MMAs and waiting (bounded) one batch
// behind; e4m3 alternates two TMEM accumulators, e2m1 keeps one (the MMAs of a
// CTA run in order) next to its scale-factor columns. POPC probe: every thread
// runs 8 independent XOR + POPC + ADD chains; the sums are written so the work
// is kept.
#include "eogp_dev.cuh"
#include "eogp_internal.h"

using namespace eogp;

namespace {

constexpr int kBatch = 64;

__global__ void __launch_bounds__(128, 1) k_peak_f8(int batches, unsigned* status, unsigned* sink) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* A = smem;          // 128 rows x 128 bytes
  uint8_t* B = smem + 16384;  // 256 rows x 128 bytes
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 16384 + 32768);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int i = threadIdx.x; i < (16384 + 32768) / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0x38383838u, 0xB8B8B8B8u, 0x38383838u, 0xB8B8B8B8u);
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_barrier_init();
  }
  fence_proxy_async_smem();
  if (warp == 0) tmem_alloc(tslot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  if (warp == 0 && lane == 0) {
    const uint32_t idesc = idesc_e4m3_f32(128, 256);
    const uint32_t sa = smem_u32(A), sb = smem_u32(B);
    for (int b = 0; b < batches; ++b) {
      const int buf = b & 1;
      if (b >= 2 && !mbar_wait(&bar[buf], ((b >> 1) - 1) & 1u, status)) break;
      tc_fence_after();
#pragma unroll 4
      for (int i = 0; i < kBatch; ++i) {
        const int kk = i & 3;
        tc_mma_f8(tmem + buf * 256u, sdesc_sw128(sa + kk * 32, 16, 1024), sdesc_sw128(sb + kk * 32, 16, 1024),
                  idesc, i != 0 ? 1u : 0u);
      }
      tc_commit(&bar[buf]);
    }
    // drain the last two batches
    for (int b = batches > 2 ? batches - 2 : 0; b < batches; ++b)
      if (!mbar_wait(&bar[b & 1], (b >> 1) & 1u, status)) break;
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    float v[16];
    tmem_ld16(tmem + (static_cast<uint32_t>(lane) << 16), v);  // keep the result observable
    if (lane == 0 && v[0] == 12345.f) atomicAdd(sink, 1u);
    tmem_dealloc(tmem, 512);
  }
}

__global__ void __launch_bounds__(128, 1) k_peak_f4(int batches, unsigned* status, unsigned* sink) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* bar = reinterpret_cast<uint64_t*>(smem + 16384 + 32768);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bar + 2);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // e2m1 +1 = 0x2, -1 = 0xA
  for (int i = threadIdx.x; i < (16384 + 32768) / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(smem)[i] = make_uint4(0x2A2A2A2Au, 0xA2A2A2A2u, 0x22AA22AAu, 0xAA22AA22u);
  if (threadIdx.x == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    fence_barrier_init();
  }
  fence_proxy_async_smem();
  if (warp == 0) tmem_alloc(tslot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  {  // unit scale factors (ue8m0 0x7F) in columns 256-287, each warp its lane quarter
    uint32_t v[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) v[e] = 0x7F7F7F7Fu;
    const uint32_t q = tmem + (static_cast<uint32_t>(warp * 32) << 16);
    tmem_st16_issue(q + 256u, v);
    tmem_st16_issue(q + 272u, v);
    tmem_wait_st();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0 && lane == 0) {
    const uint32_t idesc = idesc_mxf4_f32(128, 256);
    const uint32_t sb = smem_u32(smem + 16384);
    const uint32_t a_tmem = tmem + 288u;  // A read from TMEM as in the scoring kernel (any values)
    for (int b = 0; b < batches; ++b) {
      const int buf = b & 1;
      if (b >= 2 && !mbar_wait(&bar[buf], ((b >> 1) - 1) & 1u, status)) break;
      tc_fence_after();
#pragma unroll 4
      for (int i = 0; i < kBatch; ++i) {
        const int kk = i & 3;
        tc_mma_f4_ta(tmem, a_tmem + 8u * kk, sdesc_sw128(sb + kk * 32, 16, 1024), idesc, tmem + 256u, tmem + 272u,
                     i != 0 ? 1u : 0u);
      }
      tc_commit(&bar[buf]);
    }
    for (int b = batches > 2 ? batches - 2 : 0; b < batches; ++b)
      if (!mbar_wait(&bar[b & 1], (b >> 1) & 1u, status)) break;
  }
  __syncwarp();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    float v[16];
    tmem_ld16(tmem + (static_cast<uint32_t>(lane) << 16), v);
    if (lane == 0 && v[0] == 12345.f) atomicAdd(sink, 1u);
    tmem_dealloc(tmem, 512);
  }
}

__global__ void __launch_bounds__(256) k_peak_popc(int iters, unsigned* sink) {
  uint32_t x[8], acc[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) {
    x[c] = (threadIdx.x + 1u) * 2654435761u + c * 40503u + blockIdx.x;
    acc[c] = 0;
  }
  for (int i = 0; i < iters; ++i) {
#pragma unroll
    for (int c = 0; c < 8; ++c) {
      x[c] ^= 0x9E3779B9u + static_cast<uint32_t>(i);
      acc[c] += __popc(x[c]);
    }
  }
  uint32_t t = 0;
#pragma unroll
  for (int c = 0; c < 8; ++c) t += acc[c];
  if (t == 0xFFFFFFFFu) atomicAdd(sink, t);
}

// Self-test of the bounded waits: one thread waits, through the same
// mbar_wait every kernel uses, on an mbarrier that nothing arrives on, so the
// wait runs out after `limit` cycles and sets the timeout bit.
__global__ void k_wait_selftest(unsigned* status, long long limit) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_barrier_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) mbar_wait(&bar, 0, status, limit);
  __syncthreads();
}

}  // namespace

cudaError_t run_wait_selftest(unsigned* status, long long limit, cudaStream_t st) {
  k_wait_selftest<<<1, 32, 0, st>>>(status, limit);
  return cudaGetLastError();
}

cudaError_t run_peak_probes(int num_sms, unsigned* status, unsigned* sink, double* f8_tflops,
                            double* f4_tflops, double* popc_words_per_s, cudaStream_t st) {
  cudaEvent_t ev[4];
  for (cudaEvent_t& x : ev) cudaEventCreate(&x);
  // more than half of an SM's shared memory: one CTA (and one TMEM allocation) per SM
  const size_t smem = 140 * 1024;
  cudaError_t e = cudaFuncSetAttribute(k_peak_f8, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_peak_f4, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  const int batches = 4096;
  k_peak_f8<<<num_sms, 128, smem, st>>>(8, status, sink);  // warm-up
  k_peak_f4<<<num_sms, 128, smem, st>>>(8, status, sink);
  cudaEventRecord(ev[0], st);
  k_peak_f8<<<num_sms, 128, smem, st>>>(batches, status, sink);
  cudaEventRecord(ev[1], st);
  k_peak_f4<<<num_sms, 128, smem, st>>>(batches, status, sink);
  cudaEventRecord(ev[2], st);
  const int iters = 1 << 15;
  const int blocks = num_sms * 8;
  k_peak_popc<<<blocks, 256, 0, st>>>(iters, sink);
  cudaEventRecord(ev[3], st);
  e = cudaEventSynchronize(ev[3]);
  if (e != cudaSuccess) return e;
  float ms[3] = {0.f, 0.f, 0.f};
  for (int i = 0; i < 3; ++i) cudaEventElapsedTime(&ms[i], ev[i], ev[i + 1]);
  for (cudaEvent_t& x : ev) cudaEventDestroy(x);
  const double mmas = static_cast<double>(kBatch) * batches * num_sms;
  *f8_tflops = 2.0 * 128 * 256 * 32 * mmas / (ms[0] / 1000.0) / 1e12;
  *f4_tflops = 2.0 * 128 * 256 * 64 * mmas / (ms[1] / 1000.0) / 1e12;
  *popc_words_per_s = static_cast<double>(blocks) * 256 * 8 * iters / (ms[2] / 1000.0);
  return cudaGetLastError();
}
