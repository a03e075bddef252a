// Host-side internals shared by the library's translation units.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <vector>

#include "../../include/eogp.h"

namespace eogp {

// Records a thread-local error message and returns `code`.
int set_error(int code, const char* fmt, ...);
// Clears the thread-local message.
void clear_error();

// Address of the device status word on the current device (nullptr on failure).
unsigned* status_word();

// Current value of a process-wide dispatch option (EOGP_OPT_*).
int option(int which);

// Encodes a tiled TMA descriptor (driver entry point resolved once).
// dims/strides: innermost first; strides in bytes for dims 1..rank-1.
int make_tmap(CUtensorMap* tm, CUtensorMapDataType dt, int rank, const void* base,
              const uint64_t* dims, const uint64_t* strides_bytes, const uint32_t* box,
              CUtensorMapSwizzle swz);

}  // namespace eogp

// Retained-set plan.
struct eogp_plan {
  int d_in = 0, d_out = 0, m = 0;
  double lambda = 0.0;
  int device = -1;
  std::vector<int32_t> j, i;        // canonical order
  std::vector<float> scale;         // (Lambda + lambda)^{-1/2}, fp32
  std::vector<int32_t> R, C;        // distinct rows / columns, ascending
  std::vector<int32_t> posR, posC;  // per retained r: index of j_r in R, of i_r in C
  // Active 128x128 tiles of the R x C block, CSR over entries.
  std::vector<int32_t> tile_rc;     // (rt << 16) | ct
  std::vector<int32_t> tile_start;  // n_tiles + 1
  std::vector<int32_t> grp_start;   // n_tiles * 4 + 1: (tile, co / 32) groups
  std::vector<int32_t> ent;         // 4 ints per entry: r, (ro << 8) | co, scale bits, 0
  std::vector<int32_t> ent_r;       // retained index r
  std::vector<int32_t> ent_off;     // (ro << 8) | co inside the tile
  std::vector<float> ent_scale;
  // Device copies (owned).
  int32_t* d_tile_rc = nullptr;
  int32_t* d_tile_start = nullptr;
  int32_t* d_grp_start = nullptr;
  int32_t* d_ent = nullptr;
  int32_t* d_ent_r = nullptr;
  int32_t* d_ent_off = nullptr;
  float* d_ent_scale = nullptr;
  int32_t* d_posR = nullptr;
  int32_t* d_posC = nullptr;
  float* d_scale = nullptr;
  int32_t* d_R = nullptr;
  int32_t* d_C = nullptr;
  int nR() const { return static_cast<int>(R.size()); }
  int nC() const { return static_cast<int>(C.size()); }
  int n_tiles() const { return static_cast<int>(tile_rc.size()); }
};

// ---------------------------------------------------------------- launchers
// All return cudaError_t of the launch.

// k_pack.cu: x (sum of `splits` partial slabs, slab stride `slab`) -> optional x
// copy, sign codes and scales. One warp per row.
cudaError_t launch_pack(const float* part, int splits, size_t slab, int ldp, int B, int k,
                        float* x_out, int ldx, uint32_t* codes, int ld_codes, float* scales,
                        int ld_scales, unsigned* status, cudaStream_t st);

// k_score.cu
cudaError_t launch_score_codes(const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                               const int* ks, int U, const uint32_t* query, int ldq,
                               const float* qs, int ldqs, int Q, float* out, int ldo,
                               cudaStream_t st);
cudaError_t launch_score_paper(const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                               const int* ks, int U, const float* y, int ldy, int Q, float* out,
                               int ldo, cudaStream_t st);

// k_score_tc.cu: CODES (e4m3 +-1 operands) and PAPER (bf16 hi/lo query x bf16 +-1
// codes) scoring on the tensor cores, dense output or fused top-K.
constexpr int kTopKMax = 32;  // largest K of the fused top-K (kTopKBuf - 32)
constexpr int kTopKBuf = 64;  // running list buffer per query column of the fused top-K
struct TcTopK {
  int K;
  float* lst;  // per-CTA lists [grid][Q][K] (workspace)
  int* lsi;
  float* bufs;  // running list buffers [grid][queries per tile][kTopKBuf] (workspace)
  int* bufi;
  unsigned* gtau;  // [Q] shared thresholds (workspace)
  float* scr;      // per-CTA score scratch (workspace)
  float* out_s;  // final [Q, K] scores / stored indices
  int ld_os;
  int* out_i;
  int ld_oi;
};
bool score_tc_supported(int mode, const int* ks, int U, int Q);
size_t score_tc_ws_bytes(int mode, const int* ks, int U, int Q);
int score_tc_grid(int mode, const int* ks, int U, int N, int Q, int K, int num_sms);
bool score_tc_topk_fits(int mode, const int* ks, int U, int Q, int K);
size_t score_tc_list_buf_bytes(int mode, const int* ks, int U, int Q, int K, int grid);  // each of bufs, bufi
size_t score_tc_scratch_bytes(int mode, const int* ks, int U, int Q, int K, int grid);
cudaError_t launch_score_tc(int mode, const uint32_t* train, int ldt, const float* ts, int ldts, int N,
                            const int* ks, int U, const void* query, int ldq, const float* qs,
                            int ldqs, int Q, float* out, int ldo, const TcTopK* topk, void* ws,
                            int num_sms, unsigned* status, cudaStream_t st);

// k_topk.cu: top-K of a dense [Q, N] score matrix into per-slot lists, and the
// merge of per-slot lists [S][Q][K] (index -1 = empty) into [Q, K].
int topk_dense_slots(int N);
// Largest N k_topk_select ranks (one row per block, held in shared memory).
int topk_select_max_n();
// Per query the K best of a dense [Q, N] score row, written to the final
// outputs (N <= topk_select_max_n(), K <= EOGP_TOPK_MAX).
cudaError_t launch_topk_select(const float* scores, int ld, int Q, int N, int K, float* out_s, int ld_os,
                               int* out_i, int ld_oi, cudaStream_t st);
cudaError_t launch_topk_dense(const float* scores, int ld, int Q, int N, int K, float* lst, int* lsi,
                              cudaStream_t st);
cudaError_t launch_topk_merge(const float* lst, const int* lsi, int S, int Q, int K, float* out_s,
                              int ld_os, int* out_i, int ld_oi, cudaStream_t st);

// EK-FAC eigenvalue correction (k_tc.cu, bf16; k_simt.cu, fp32).
size_t ekfac_smem_bytes(int stages);
int ekfac_chunks(int B, int n_tiles, int num_sms);
cudaError_t launch_tc_ekfac(const void* St_hi, const void* St_lo, int ldS, const void* At_hi,
                            const void* At_lo, int ldA, int B, int T, int d_out, int d_in, float* part,
                            int n_chunks, double* sumsq, int ld, int accumulate, int stages, int num_sms,
                            unsigned* status, cudaStream_t st);
cudaError_t launch_rows_fixup(float* X, int M, int n, int ld, int T, const float* bias,
                              const int32_t* lengths, cudaStream_t st);
cudaError_t launch_sq_accum(const float* G, int rows, int cols, double* sumsq, int ld, int accumulate,
                            cudaStream_t st);

// k_payload.cu: store records (per-module sign bytes + FP16 scale).
size_t payload_row_bytes(const int* ks, int U);
cudaError_t launch_payload_pack(const uint32_t* codes, int ld_codes, const float* scales, int ld_scales, int N,
                                const int* ks, int U, uint8_t* out, size_t ld_out, cudaStream_t st);
cudaError_t launch_payload_unpack(const uint8_t* in, size_t ld_in, int N, const int* ks, int U, uint32_t* codes,
                                  int ld_codes, float* scales, int ld_scales, cudaStream_t st);

// k_peaks.cu: e4m3 tensor-core and XOR + popcount throughput probes.
cudaError_t run_wait_selftest(unsigned* status, long long limit, cudaStream_t st);
cudaError_t run_peak_probes(int num_sms, unsigned* status, unsigned* sink, double* f8_tflops, double* f4_tflops,
                            double* popc_words_per_s, cudaStream_t st);

// k_srht.cu: EOGP-R second stage, one CTA per row (z fp32, or bf16 hi + lo when hilo).
int srht_width(int m);
size_t srht_smem_bytes(int m);
cudaError_t launch_srht(const void* z0, const void* z1, bool hilo, int ldz, int B, int m,
                        const int8_t* signs, const int32_t* rows, int k, float* x, int ldx,
                        uint32_t* codes, int ld_codes, float* scales, int ld_scales, unsigned* status,
                        cudaStream_t st);

// k_simt.cu: C[i][j] = alpha * sum_k A(i,k) B(j,k), A(i,k) = A[i*sai + k*sak], etc.
cudaError_t launch_simt_gemm(int M, int N, int K, float alpha, const float* A, long long sai,
                             long long sak, const float* Bm, long long sbj, long long sbk,
                             float* C, long long ldc, cudaStream_t st);
// z[b*ldz + r] = scale[r] * sum_t St[(b*T+t)*ldS + posR[r]] * At[(b*T+t)*ldA + posC[r]]
cudaError_t launch_contract_f32(const float* At, int ldA, const float* St, int ldS, int B, int T,
                                int m, const int32_t* posR, const int32_t* posC,
                                const float* scale, float* z, int ldz, cudaStream_t st);
cudaError_t launch_gather_rows(const void* src, int ld_src, int elem_bytes, const int32_t* idx,
                               int n_rows, int row_len, void* dst, cudaStream_t st);

// k_tc.cu: tcgen05 kernels (bf16).
struct TcGemmCfg {
  int BN;      // N tile, multiple of 16, <= 256
  int stages;  // smem pipeline depth
};
// D[M x N] = sum_a X_a[M x K] * W[N x K]^T (X_a, W bf16 K-major; W has Wrows
// real rows, rows beyond read as zero). epi 0: out0 = bf16 hi, out1 = bf16 lo
// of D, row stride ldo, columns < ldo written; epi 1: out0 = fp32 partial slab
// per K split (slab elements apart), columns < N written.
cudaError_t launch_tc_gemm(int M, int N, int K, const void* X0, const void* X1, int ldx,
                           const void* W, int ldw, int Wrows, int splits, int epi, void* out0,
                           void* out1, int ldo, size_t slab, TcGemmCfg cfg, unsigned* status,
                           cudaStream_t st);
// out[M x N] (row stride ldo, fp32) = alpha * (Ah Bh^T + Ah Bl^T + Al Bh^T): both
// operands bf16 hi/lo pairs, K-major ([M x K] and [N x K], row strides lda, ldb
// multiples of 8 elements, 16-byte aligned); an operand pair stands for an fp32
// matrix to about 16 significant bits, and lo x lo is below that.
cudaError_t launch_tc_gemm_hl(int M, int N, int K, const void* Ah, const void* Al, int lda, const void* Bh,
                              const void* Bl, int ldb, float* out, int ldo, float alpha, unsigned* status,
                              cudaStream_t st);
// Persistent rotation GEMM: hi/lo = split(X[M x K] W[Wrows x K]^T), columns < ldo
// (a multiple of 128), rows M = B * T, written in the blocked layout
// [B][ldo / 128][T][128] that launch_tc_contract reads.
cudaError_t launch_tc_rotate(int M, int K, const void* X, int ldx, const void* W, int ldw, int Wrows,
                             void* hi, void* lo, int ldo, int T, const float* bias,
                             const int32_t* lengths, int num_sms, unsigned* status, cudaStream_t st);
// Number of K splits launch_tc_gemm actually uses for a requested count.
int tc_gemm_splits_used(int K, int splits);
// Per-example tile-sparse contraction over tokens with the scale-and-gather epilogue.
cudaError_t launch_tc_contract(const void* St_hi, const void* St_lo, int ldS, const void* At_hi,
                               const void* At_lo, int ldA, int B, int T, const eogp_plan* plan,
                               float* z, int ldz, void* zhi, void* zlo, int ldzb, int stages,
                               int num_sms, unsigned* status, cudaStream_t st);

// k_pca.cu
// Whether the fit handles this size (the subspace solver for large problems,
// the dense Jacobi solver otherwise), and the workspace it needs.
bool fit_pca_supported(int n, int m, int k);
// C_in (optional): a summed second moment sum_r z_r z_r^T [m x ldc] of n rows in
// place of Z (covariance route; Z is then unused). ws: fit_pca_ws_bytes(n, m, k)
// bytes, 256-byte aligned (fit_pca_ws_bytes(m, m, k) with C_in).
int fit_pca_device(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype,
                   float* eig, void* ws, unsigned* status, cudaStream_t st, const double* C_in = nullptr,
                   int ldc = 0);
cudaError_t second_moment_device(const float* Z, int n, int m, int ldz, double* C, int ldc, int accumulate,
                                 cudaStream_t st);
size_t fit_pca_ws_bytes(int n, int m, int k);
