/*
 * eogp.h -- C ABI of libeogp, a GB300 (sm_103a) implementation of the
 * data-parallel hot path of EOGP, "Scaling Influence Functions in LLMs through
 * Eigenbasis-Corrected One-Bit Gradient Projection" (arxiv 2609.37842):
 * per-example gradient compression into one-bit codes and influence scoring
 * of queries against the stored codes.
 *
 * Notation (the paper's). One linear module ("module u") has input
 * activations a_t in R^{d_in} and output gradients s_t in R^{d_out} for tokens
 * t = 1..T of an example. Its per-example gradient is G = sum_t s_t a_t^T
 * (d_out x d_in, Sec. 2.2). Q_A, Q_S are the K-FAC eigenbases of the two
 * Kronecker factors (Sec. 2.2, Eq. kfac_factorization) and Lambda[j][i] the
 * (corrected) eigenvalue of the Kronecker coordinate (j, i), i.e. of the basis
 * vector Q_A[:, i] (x) Q_S[:, j] (Eq. ekfac_eigendecompose).
 *
 * General conventions for every entry point:
 *  - Array arguments named "device" are device pointers owned by the caller;
 *    the library never frees or retains them after the call returns.
 *  - Matrices are row-major with an explicit leading dimension in ELEMENTS
 *    (ld >= row length). "bf16" means IEEE bfloat16 stored in uint16.
 *  - Calls that take a stream are asynchronous on that stream (0 = the legacy
 *    default stream) unless stated otherwise; the current CUDA device must be
 *    the device that owns the pointers. They do not allocate: scratch memory
 *    ("workspace") is sized with the matching *_workspace_size call and passed
 *    in, 256-byte aligned.
 *  - Every call returns an int status: EOGP_OK (0) or a negative EOGP_E*
 *    code; eogp_last_error() then returns a thread-local message. Argument
 *    errors are detected on the host before anything is launched.
 *  - Kernels never trap. A bounded wait that expires (or another device-side
 *    fault the kernels detect) sets a device status word; eogp_sync_status()
 *    synchronizes a stream and returns / clears it (EOGP_ETIMEOUT, EOGP_EDEVICE).
 *  - Unsupported shape/dtype combinations return EOGP_EUNSUPPORTED; there is
 *    no CPU fallback.
 */
#ifndef EOGP_H
#define EOGP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without including the CUDA headers. */
typedef struct CUstream_st* eogp_stream_t;

/* ---- status codes ------------------------------------------------------ */
#define EOGP_OK            0
#define EOGP_EINVAL       (-1) /* invalid argument (null pointer, size, stride, alignment) */
#define EOGP_EUNSUPPORTED (-2) /* valid request that this build does not implement */
#define EOGP_ECUDA        (-3) /* a CUDA runtime/driver call failed */
#define EOGP_ETIMEOUT     (-4) /* a kernel's bounded wait expired (from eogp_sync_status) */
#define EOGP_EWORKSPACE   (-5) /* workspace smaller than *_workspace_size reported */
#define EOGP_EDEVICE      (-6) /* other device-side error recorded by a kernel */

/* ---- element types ----------------------------------------------------- */
#define EOGP_F32  0 /* float32 inputs; computed with fp32 CUDA-core kernels */
#define EOGP_BF16 1 /* bfloat16 inputs; tcgen05 tensor-core kernels, fp32 accumulation */

/* ---- eogp_compress_layer output modes ---------------------------------- */
#define EOGP_OUT_FIRST_STAGE 0 /* z = (Lambda_m + lambda I)^{-1/2} Q_m^T g   [B x m] fp32 */
#define EOGP_OUT_COORDS      1 /* x = P^T z                                  [B x k] fp32 */
#define EOGP_OUT_CODES       2 /* sign bits of x (packed) + scale ||x||_1/k              */

/* ---- eogp_score modes -------------------------------------------------- */
#define EOGP_SCORE_CODES 0 /* sum_u s_iu s_qu <b_iu, b_qu>  (both sides one-bit)     */
#define EOGP_SCORE_PAPER 1 /* sum_u s_iu <y_u, b_iu>        (query unquantized)      */
#define EOGP_SCORE_FP    2 /* <y, x>                        (no quantization)        */

/* Last error message of the calling thread ("" if none). Never NULL. */
const char* eogp_last_error(void);

/* Library version string. */
const char* eogp_version(void);

/* Synchronizes `stream`, then returns and clears the device status word of the
 * current device: EOGP_OK, EOGP_ETIMEOUT (a bounded mbarrier/flag wait expired)
 * or EOGP_EDEVICE (another kernel-detected error, e.g. a non-finite input to
 * eogp_pack_sign). EOGP_ECUDA if the synchronization itself failed. */
int eogp_sync_status(eogp_stream_t stream);

/* ---- kernel timing ------------------------------------------------------
 * While enabled (process-wide), every kernel the library launches is
 * bracketed by two CUDA events recorded on the stream it is launched on.
 * eogp_profile_read synchronizes on the recorded events and returns, for one
 * kernel kind, the number of launches and their summed device time; reset = 1
 * releases the records of that kind. Kinds: */
#define EOGP_K_ROTATE   0 /* tcgen05 Kronecker rotation GEMM (A and S sides)    */
#define EOGP_K_CONTRACT 1 /* tcgen05 per-example contraction + gather          */
#define EOGP_K_PROJECT  2 /* tcgen05 second-stage projection (split K)         */
#define EOGP_K_PACK     3 /* sign/scale packing (also the split-K finalise)    */
#define EOGP_K_SCORE    4 /* scoring kernels                                   */
#define EOGP_K_SIMT     5 /* fp32 CUDA-core kernels of the EOGP_F32 path       */
#define EOGP_K_COUNT    6
int eogp_profile_enable(int on);
int eogp_profile_read(int kind, int* launches, double* total_ms, int reset);

/* ---- process-wide dispatch options (no counterpart in the paper) ---------
 * Two choices between implementations that give identical results. They are
 * read, under one setting, by both the workspace-size query and the call, so
 * change them only while no eogp_score / eogp_score_topk call is being
 * prepared or issued on another thread; a workspace sized under one setting
 * may be too small under the other (the call then returns EOGP_EWORKSPACE).
 *   EOGP_OPT_SCORE_OPERAND: one-bit operands of the tensor-core CODES scoring
 *     kernel. 0 (default): e2m1 (kind::mxf4, unit scales) when every module is
 *     a multiple of 256 bits and the stored rows are 16-byte aligned, else
 *     e4m3; 1: always e4m3 (kind::f8f6f4). Scores are bit-identical.
 *   EOGP_OPT_TOPK_PATH: ranking path of eogp_score_topk. 0 (default): chosen
 *     by size; 1: ranking fused into the tensor-core scoring kernel where it
 *     applies; 2: dense scores then a ranking kernel.
 * eogp_set_option returns EOGP_EINVAL for an unknown option or value. */
#define EOGP_OPT_SCORE_OPERAND 0
#define EOGP_OPT_TOPK_PATH     1
int eogp_set_option(int option, int value);
int eogp_get_option(int option, int* value);

/* Throughput probes for the scoring rooflines (no counterpart in the paper: a
 * library convenience). Measures on the current device, synchronously: the dense
 * tcgen05 rates of the two +-1 scoring MMAs in TFLOP/s (one CTA per SM issuing
 * back-to-back M = 128, N = 256 MMAs: kind::f8f6f4 e4m3 with K = 32 from shared
 * memory, kind::mxf4 e2m1 with unit ue8m0 scales, K = 64, A from tensor memory)
 * and the CUDA-core XOR + popcount rate (32-bit words per second). Any output
 * may be NULL.
 * Errors: EOGP_ECUDA, EOGP_ETIMEOUT. */
int eogp_measure_peaks(double* e4m3_tflops, double* e2m1_tflops, double* popc_words_per_s);

/* Self-test of the bounded waits (no counterpart in the paper: a library
 * convenience). Every wait in the library's kernels gives up after a limit
 * (~2 s), sets the timeout bit of the device status word and lets its kernel
 * finish instead of hanging. This call launches one thread on the current
 * device that waits, through the same routine, on an mbarrier nothing will
 * arrive on, with a limit of `limit_cycles` SM clock cycles (1 .. 1e9), then
 * returns what eogp_sync_status(NULL) reports: EOGP_ETIMEOUT when the path
 * works (that read clears the status word; the context stays usable). No fault,
 * trap or hang is involved.
 * Errors: EOGP_EINVAL (limit out of range, checked before any device call),
 * EOGP_ECUDA. */
int eogp_selftest_wait_timeout(long long limit_cycles);

/* ========================================================================
 * Retained-set plan (host; once per module)
 *
 * Selects the m Kronecker eigen-coordinates with the largest eigenvalues
 * (Sec. 3.2: the top-m eigenvectors of Sigma_proxy, Eq. sigma_ekfac, are those
 * of the m largest corrected eigenvalues; Alg. 1 "Select Q_{u,m}, Lambda_{u,m}")
 * and the damping lambda = damping_rel * tr(Lambda)/d (App. C.2,
 * Eq. app_module_damping; the paper uses damping_rel = 0.1).
 * ======================================================================== */
typedef struct eogp_plan eogp_plan;

typedef struct {
  int d_in, d_out, m;
  int nR;        /* distinct rows j of the retained set (size of R)            */
  int nC;        /* distinct columns i (size of C)                             */
  int n_tiles;   /* active 128 x 128 tiles of the R x C block                  */
  double lambda; /* damping actually used                                      */
} eogp_plan_info;

/* Build a plan. Eigenvalues are given EITHER as the two K-FAC factor spectra
 * (lam_S [d_out], lam_A [d_in]; Lambda[j][i] = lam_S[j] * lam_A[i] formed in
 * double) with Lambda == NULL, OR as the full corrected table Lambda
 * [d_out x d_in] (row-major, double) with lam_S == lam_A == NULL. All are HOST
 * arrays, read during the call only.
 * Canonical retained order: eigenvalue descending, ties broken by the
 * Kronecker column position i*d_out + j ascending. R and C are the distinct
 * j / i of the retained set in ascending order.
 * The plan owns small device tables (allocated here on the current device,
 * freed by eogp_plan_destroy); it must be used on that device only.
 * Errors: EOGP_EINVAL (null out, d_in/d_out < 1, m outside [1, d_in*d_out],
 * damping_rel < 0, both or neither eigenvalue forms, non-finite or negative
 * eigenvalues), EOGP_ECUDA. */
int eogp_plan_layer(const double* lam_S, const double* lam_A, const double* Lambda,
                    int d_in, int d_out, int m, double damping_rel, eogp_plan** out);

void eogp_plan_destroy(eogp_plan* plan);

int eogp_plan_get_info(const eogp_plan* plan, eogp_plan_info* info);

/* Host copies of the canonical retained list: j[m], i[m] (int32) and the
 * fp32 scale (Lambda[j][i] + lambda)^{-1/2} of Eq. first_stage. Any output
 * pointer may be NULL. */
int eogp_plan_get_retained(const eogp_plan* plan, int32_t* j, int32_t* i, float* scale);

/* Host copies of R [nR] and C [nC] (either may be NULL). */
int eogp_plan_get_sets(const eogp_plan* plan, int32_t* R, int32_t* C);

/* Gather the retained eigenvectors as rows, the layout eogp_compress_layer
 * reads: which = 0 copies V_full row C[r] (an eigenvector of A, i.e. column
 * C[r] of Q_A) to row r of V_ret [nC x d_in]; which = 1 copies row R[r] of
 * V_full (eigenvectors of S as rows, d_out x d_out) to V_ret [nR x d_out].
 * dtype EOGP_F32 or EOGP_BF16; V_full with leading dimension ld_full; V_ret
 * dense. Device pointers, asynchronous on `stream`. */
int eogp_plan_gather_rows(const eogp_plan* plan, int which, int dtype, const void* V_full,
                          int ld_full, void* V_ret, eogp_stream_t stream);

/* ========================================================================
 * Compression of one module (Alg. 1 "Storing one training example", applied
 * to a batch of B examples; also the query projection y_u = T_u(L_u q_u)).
 * ======================================================================== */
typedef struct {
  int d_in, d_out; /* module shape                                             */
  int T;           /* tokens per example                                       */
  int m;           /* retained first-stage coordinates (= plan m)              */
  int k;           /* PCA output coordinates (sign bits) per example           */
  int dtype;       /* EOGP_F32 or EOGP_BF16: type of a, s, VA, VS, Pt          */
  const void* VA;  /* device [nC x d_in]: row r = eigenvector Q_A[:, C[r]]     */
  const void* VS;  /* device [nR x d_out]: row r = eigenvector Q_S[:, R[r]]    */
  const void* Pt;  /* device [k x m]: row c = PCA direction c (column c of P,
                      App. B.2) over the canonical retained order; may be NULL
                      for EOGP_OUT_FIRST_STAGE or with the SRHT below          */
  const eogp_plan* plan;
  /* EOGP-R (Sec. 3.2 "A scalable alternative to PCA"; App. B.2
     Eq. app_srht_definition): when Pt is NULL and srht_rows is set, the second
     stage is x = sqrt(p/k) R H_p D J z (see eogp_srht) instead of P^T z, with
     k <= p = 2^ceil(log2 m) and m <= EOGP_SRHT_MAX_M.                       */
  const int8_t* srht_signs;  /* device [m]: diagonal of D (< 0 means -1)      */
  const int32_t* srht_rows;  /* device [k]: rows of H_p kept by R, in [0, p)   */
  /* Real-workload plumbing (App. C.1): */
  const float* bias_A;  /* device [nC] fp32, or NULL. Non-NULL: the module has a
                           bias (GPT-2 attributes biases), treated as a constant-1
                           input channel appended after the d_in activations: the
                           plan and Q_A are over d_in + 1 inputs, VA holds the
                           first d_in components of the retained eigenvectors and
                           bias_A[r] = Q_A[d_in][C[r]], their bias-channel component */
  const int32_t* lengths;  /* device [B] or NULL: example b keeps tokens
                           t < lengths[b] (0 <= lengths[b] <= T); later positions
                           are padding and contribute nothing (as s_t = 0)        */
  int bases_on_host;    /* nonzero: VA and VS are host pointers (page-locked for
                           asynchronous copies); each call copies them into its
                           workspace with cudaMemcpyAsync on its stream before the
                           rotations (eigenbases too large to keep resident).
                           A caller that overlaps these copies with the previous
                           layer's compute stages them itself and passes device
                           pointers instead.                                      */
} eogp_layer_desc;

/* Workspace bytes eogp_compress_layer needs for this descriptor, batch B and
 * output mode. */
int eogp_compress_workspace_size(const eogp_layer_desc* L, int B, int out_mode, size_t* bytes);

/* For each example b < B (Sec. 3.2 Eq. first_stage and Eq. second_stage;
 * Sec. 3.3 Eq. onebit):
 *   G~_b = Q_S^T G_b Q_A evaluated on the retained rows/columns only, as
 *          sum_t (V_S s_t)(V_A a_t)^T  (the Kronecker identity of Sec. 2.2),
 *   z_b[r] = (Lambda[j_r][i_r] + lambda)^{-1/2} G~_b[j_r][i_r],
 *   x_b = P^T z_b,
 *   codes_b: bit (c % 32) of word c / 32 is 1 iff x_b[c] >= 0 (App. E.1 byte
 *            order; pad bits 0), scales_b = ||x_b||_1 / k.
 * Inputs: a [B x T x d_in], s [B x T x d_out] (dtype, dense, device).
 * Outputs by out_mode:
 *   FIRST_STAGE: out = z [B x ld_out], ld_out >= m;
 *   COORDS:      out = x [B x ld_out], ld_out >= k;
 *   CODES:       codes [B x ld_codes] uint32 (ld_codes >= ceil(k/32), so a
 *                module's words can sit at an offset inside a wider store row)
 *                and scales[b * ld_scales] fp32; `out` is ignored.
 * BF16 requires d_in, d_out, m multiples of 8 (16-byte TMA strides) and
 * 16-byte aligned a, s, VA, VS, Pt; F32 has no extra constraint.
 * Errors: EOGP_EINVAL, EOGP_EUNSUPPORTED, EOGP_EWORKSPACE, EOGP_ECUDA. */
int eogp_compress_layer(const eogp_layer_desc* L, const void* a, const void* s, int B,
                        int out_mode, float* out, int ld_out, uint32_t* codes, int ld_codes,
                        float* scales, int ld_scales, void* ws, size_t ws_bytes,
                        eogp_stream_t stream);

/* Page-locked host memory for inputs that eogp_compress_layer_host (or the
 * caller) copies to the device, registered with cudaHostRegister and backed by
 * transparent huge pages where that matters. Measured on GB300 systems,
 * host-to-device copies from anonymous memory advised for huge pages ran at the
 * link rate (~211 GB/s) in every trial; cudaHostAlloc'd buffers varied from ~80
 * to ~210 GB/s between allocations, and the same memory on 64 KB base pages
 * ran at ~51 GB/s. Size classes (H = the kernel's huge-page size, 2 MB on
 * 4 KB-page hosts, 512 MB on 64 KB-page arm64 hosts):
 *   bytes >= H/2           a region of its own, whole huge pages;
 *   1 MB <= bytes < H/2    a 4 KB-aligned block of a shared arena of one huge
 *                          page (first fit; the arena is released with its last
 *                          block), so such buffers get huge pages without each
 *                          pinning a whole one;
 *   bytes < 1 MB           whole base pages, no huge-page advice.
 * The memory is zero-filled. eogp_host_free takes only the pointer (NULL is a
 * no-op). Thread-safe. A library convenience with no counterpart in the paper.
 * Errors: EOGP_EINVAL (bytes == 0, ptr NULL, mapping failed, pointer not from
 * eogp_host_alloc), EOGP_ECUDA (registration failed, e.g. no device). */
int eogp_host_alloc(size_t bytes, void** ptr);
int eogp_host_free(void* ptr);

/* Same computation and outputs as eogp_compress_layer, with the inputs a and s
 * in host memory (page-locked, so that the copies run asynchronously): the
 * batch is compressed `chunk` examples at a time (0: about 64 MB of a and s
 * per chunk). Each chunk is copied into the workspace with cudaMemcpyAsync on
 * a copy stream the call creates, double-buffered, so the copy of chunk c + 1
 * overlaps the compute of chunk c on `stream`; the compute of every chunk is
 * queued on `stream`, which therefore orders all of the call's work, and the
 * call releases its copy stream and events itself. The first copies wait for
 * the work already queued on `stream` (the workspace may be memory that such
 * work still uses, as with a stream-ordered allocator). `descriptor->lengths` (if
 * any) is a device array of all B examples. With bases_on_host the eigenbases
 * are copied once per call, not per chunk. a and s must stay valid and
 * unchanged until `stream` reaches the point of the call. A library
 * convenience for inputs that live in host memory: the paper times store
 * construction including its host-to-device transfers (App. E.3) but gives no
 * interface for it.
 * Errors: as eogp_compress_layer; EOGP_EINVAL for chunk < 0. */
int eogp_compress_host_workspace_size(const eogp_layer_desc* L, int B, int chunk, int out_mode,
                                      size_t* bytes);
int eogp_compress_layer_host(const eogp_layer_desc* L, const void* a, const void* s, int B, int chunk,
                             int out_mode, float* out, int ld_out, uint32_t* codes, int ld_codes,
                             float* scales, int ld_scales, void* ws, size_t ws_bytes,
                             eogp_stream_t stream);

/* Several modules (a layer, or a stack of layers) of one batch of B examples
 * with host-memory inputs, in one call: module u (descriptor L[u], inputs a[u]
 * and s[u] in page-locked host memory, outputs codes[u] and scales[u], or
 * out[u]) gets exactly the computation and outputs of
 * eogp_compress_layer_host(L[u], a[u], s[u], B, chunk, out_mode, ...). One
 * out_mode and one set of leading dimensions (ld_out, ld_codes, ld_scales)
 * serve all modules. What the single call adds is overlap across modules. The
 * workspace holds two sets of staging buffers, and of eigenbasis copies with
 * bases_on_host, used by alternate modules. The copies of module u therefore
 * wait only for the compute of module u - 2, and run while module u - 1 is
 * computed. One call per module would wait for each previous module's
 * compute.
 *  - The first two modules' copies wait for the work already queued on
 *    `stream`, as in eogp_compress_layer_host.
 *  - The compute of every module is queued on `stream` in module order.
 *  - The call releases its copy stream and events itself.
 *  - The workspace size is the largest module's staging set twice, plus the
 *    largest eogp_compress_layer workspace. With n = 1 it equals
 *    eogp_compress_host_workspace_size.
 * A library convenience for inputs that live in host memory: the paper times
 * store construction including its host-to-device transfers (App. E.3) but
 * gives no interface for it.
 * Errors: as eogp_compress_layer_host; EOGP_EINVAL for n < 1 or a NULL array
 * or entry. */
int eogp_compress_layers_host_workspace_size(const eogp_layer_desc* const* L, int n, int B, int chunk,
                                             int out_mode, size_t* bytes);
int eogp_compress_layers_host(const eogp_layer_desc* const* L, int n, const void* const* a,
                              const void* const* s, int B, int chunk, int out_mode, float* const* out,
                              int ld_out, uint32_t* const* codes, int ld_codes, float* const* scales,
                              int ld_scales, void* ws, size_t ws_bytes, eogp_stream_t stream);

/* Same computation and outputs as eogp_compress_layer, for callers that cannot
 * allocate device memory (a plugin whose host framework owns every device
 * allocation, a service confined to a memory budget fixed at start-up, a C
 * program with no allocator of its own). The paper has no counterpart: this is
 * a library convenience. Its scratch is a built-in device array of
 * EOGP_STATIC_WORKSPACE_BYTES that every GPU loading the library keeps until
 * the process exits; the call itself allocates nothing.
 *  - Requests whose eogp_compress_workspace_size exceeds the array return
 *    EOGP_EUNSUPPORTED with a message; use a smaller B or eogp_compress_layer.
 *  - All calls on a device share the one array and it keeps the last call's
 *    contents. Calls whose kernels overlap on the GPU (e.g. on two streams
 *    without ordering between them) race on it and corrupt each other's results.
 *  - Every call looks up the array's device address on the current device
 *    (cudaGetSymbolAddress, which allocates nothing), so the address stays
 *    right if the device's context is destroyed and created again. The first
 *    call on a device may also load the library's device code there; make
 *    that first call before any stream capture. */
#define EOGP_STATIC_WORKSPACE_BYTES (32u << 20)
int eogp_compress_layer_static(const eogp_layer_desc* L, const void* a, const void* s, int B,
                               int out_mode, float* out, int ld_out, uint32_t* codes, int ld_codes,
                               float* scales, int ld_scales, eogp_stream_t stream);

/* ========================================================================
 * EK-FAC eigenvalue correction (Sec. 2.2 "EK-FAC approximation": the mean
 * square of each coordinate of the gradients expressed in the K-FAC eigenbasis;
 * App. C.2: averaged over examples, using sequence-level gradients)
 * ======================================================================== */
typedef struct {
  int d_in, d_out; /* module shape                                             */
  int T;           /* tokens per example                                       */
  int dtype;       /* EOGP_F32 or EOGP_BF16: type of a, s, VA, VS              */
  const void* VA;  /* device [d_in x d_in]: row i = eigenvector Q_A[:, i]      */
  const void* VS;  /* device [d_out x d_out]: row j = eigenvector Q_S[:, j]    */
} eogp_ekfac_desc;

int eogp_ekfac_workspace_size(const eogp_ekfac_desc* D, int B, size_t* bytes);

/* For the B examples of a [B x T x d_in], s [B x T x d_out] (dense, device):
 *   sumsq[j * ld + i] (+)= sum_b ((Q_S^T G_b Q_A)[j][i])^2,  G_b = sum_t s_t a_t^T,
 * over the full d_out x d_in coordinate block (fp64 device array, ld >= d_in;
 * added to when `accumulate` is nonzero, overwritten otherwise). The corrected
 * eigenvalues are sumsq / (examples seen); pass them to eogp_plan_layer as
 * the full Lambda table. The per-example coordinates are formed as in
 * eogp_compress_layer (bf16: hi/lo intermediates, 3 MMAs per step), their
 * squares summed in fp32 over runs of examples and the runs added in fp64 in a
 * fixed order (bitwise reproducible).
 * BF16 requires d_in, d_out multiples of 8 and 16-byte aligned a, s, VA, VS.
 * Errors: EOGP_EINVAL, EOGP_EUNSUPPORTED, EOGP_EWORKSPACE, EOGP_ECUDA. */
int eogp_ekfac_accumulate(const eogp_ekfac_desc* D, const void* a, const void* s, int B,
                          double* sumsq, int ld, int accumulate, void* ws, size_t ws_bytes,
                          eogp_stream_t stream);

/* ========================================================================
 * PCA fit (App. B.2 "PCA fitting"; Alg. 1 "fit P_u by uncentered PCA")
 * ======================================================================== */
int eogp_fit_pca_workspace_size(int n, int m, int k, size_t* bytes);

/* Z [n x ldz] fp32 device (rows = first-stage coordinates of n fitting
 * examples). Writes Pt [k x ld_pt] (row c = unit eigenvector c of Z^T Z / n,
 * eigenvalue descending; sign fixed so that its largest-magnitude entry is
 * positive, ties to the lowest index) as EOGP_F32 or EOGP_BF16 (pt_dtype), and
 * eig [k] fp32 (the eigenvalues of Z^T Z / n). Uses the n x n Gram matrix when
 * n < m, as the paper describes. Eigenpairs come from a cyclic Jacobi
 * eigensolver on the device, in fp64. This call BLOCKS the host until the fit
 * is done (it reads a convergence measure once per sweep).
 * Errors: EOGP_EINVAL (k < 1 or k > min(n, m), ldz < m, ld_pt < m),
 * EOGP_EWORKSPACE, EOGP_EUNSUPPORTED (min(n, m) > 12288), EOGP_ECUDA. */
int eogp_fit_pca(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt, int pt_dtype,
                 float* eig, void* ws, size_t ws_bytes, eogp_stream_t stream);

/* The same fit split for data spread over several processes or GPUs (the
 * covariance route of App. B.2: P from Z^T Z / n). Each holder of rows adds its
 * part of the second moment, the parts are summed (one reduction of an m x m
 * fp64 matrix, e.g. over a process group), and the fit runs on the sum.
 *   eogp_second_moment: C [m x ldc] fp64 device (+)= sum_r z_r z_r^T over the n
 *     rows of Z [n x ldz] fp32 device (overwritten when accumulate == 0).
 *   eogp_fit_pca_from_moment: Pt, eig as eogp_fit_pca for the matrix C / n_total
 *     (n_total = rows summed into C); workspace from
 *     eogp_fit_pca_from_moment_workspace_size; m <= 12288; blocks the host.
 * Errors: EOGP_EINVAL, EOGP_EUNSUPPORTED, EOGP_EWORKSPACE, EOGP_ECUDA. */
int eogp_second_moment(const float* Z, int n, int m, int ldz, double* C, int ldc, int accumulate,
                       eogp_stream_t stream);
int eogp_fit_pca_from_moment_workspace_size(int m, int k, size_t* bytes);
int eogp_fit_pca_from_moment(const double* C, int m, int ldc, int n_total, int k, void* Pt, int ld_pt,
                             int pt_dtype, float* eig, void* ws, size_t ws_bytes, eogp_stream_t stream);

/* ========================================================================
 * One-bit encoding (Sec. 3.3 Eq. onebit; Alg. 1 "Store packed binary signs")
 * ======================================================================== */
/* EOGP-R second stage (Sec. 3.2 "A scalable alternative to PCA"; App. B.2
 * Eq. app_srht_definition), applied to rows z of z [B x ldz] fp32 device:
 *   x = sqrt(p/k) R H_p D J z,  p = 2^ceil(log2 m),
 * J zero-pads to p, D = diag(signs) (signs [m] int8 device, < 0 means -1),
 * H_p is the orthonormal Walsh-Hadamard matrix in Sylvester order
 * (H_p[r][c] = (-1)^popcount(r & c) / sqrt(p)), R keeps rows[0..k) (int32
 * device, each in [0, p), distinct; out-of-range rows give 0 and set
 * EOGP_EDEVICE in the device status word). The random signs and rows are the
 * caller's: the same realisation must serve stored examples and queries.
 * Outputs (either may be NULL): x [B x ldx] fp32; codes [B x ld_codes] and
 * scales[b * ld_scales] as in eogp_pack_sign (sign bits of x, ||x||_1 / k).
 * Errors: EOGP_EINVAL, EOGP_EUNSUPPORTED (m > EOGP_SRHT_MAX_M), EOGP_ECUDA. */
#define EOGP_SRHT_MAX_M 32768
int eogp_srht(const float* z, int B, int m, int ldz, const int8_t* signs, const int32_t* rows, int k,
              float* x, int ldx, uint32_t* codes, int ld_codes, float* scales, int ld_scales,
              eogp_stream_t stream);

/* x [B x ldx] fp32 device -> codes [B x ld_codes] uint32 (bit c % 32 of word
 * c / 32 = [x_c >= 0], pad bits 0) and scales[b * ld_scales] = ||x_b||_1 / k
 * (fixed-order reduction: bitwise reproducible). A NaN input sets
 * EOGP_EDEVICE in the device status word. */
int eogp_pack_sign(const float* x, int B, int k, int ldx, uint32_t* codes, int ld_codes,
                   float* scales, int ld_scales, eogp_stream_t stream);

/* ========================================================================
 * Scoring (Sec. 3.3 Eq. onebit_influence; App. B.3 Eq. app_stored_influence;
 * scan cost Eq. app_scan_complexity). Module contributions are summed.
 * ======================================================================== */
int eogp_score_workspace_size(int N, const int* k_per_module, int U, int mode, int Q,
                              size_t* bytes);

/* U modules with k_per_module[u] coordinates (HOST array). A stored row holds
 * the modules' codes back to back, module u starting at word
 * sum_{v<u} ceil(k_v/32); W = total words.
 *   CODES: train = uint32 codes [N x ld_train] (ld_train >= W),
 *          train_scales [N x ld_tscale], query = uint32 codes [Q x ld_query],
 *          query_scales [Q x ld_qscale];
 *          scores[q][i] = sum_u fl(fl(s_qu * s_iu) * (k_u - 2 popc(b_iu ^ b_qu))),
 *          accumulated in fp32 in module order with no fused multiply-add
 *          (bitwise reproducible).
 *   PAPER: train = codes as above, train_scales as above, query = fp32
 *          coordinates [Q x ld_query] (module u at column sum_{v<u} k_v),
 *          query_scales ignored; scores[q][i] = sum_u s_iu <y_qu, b_iu>.
 *          With every k_u a multiple of 64 and the workspace
 *          eogp_score_workspace_size reports (4 Q sum_u k_u bytes), this runs on
 *          the tensor cores with y split into bf16 hi + lo (about 2^-17 relative)
 *          and fp32 sums: |error| <= 1e-5 sum_u s_iu ||y_qu||_1 for k_u <= 16384.
 *   FP:    train = fp32 coordinates [N x ld_train], query = fp32 [Q x ld_query];
 *          scores[q][i] = <y_q, x_i>; scales ignored.
 * scores [Q x ld_scores] fp32 device, ld_scores >= N.
 * ws: 256-byte aligned device workspace of at least eogp_score_workspace_size
 * bytes (0 bytes for the CUDA-core kernels); CODES and PAPER use the tensor
 * cores when it is given, the shape allows (CODES: Q >= 64, k_u % 128 == 0;
 * PAPER: k_u % 64 == 0) and the code rows are aligned (CODES: ld_train % 4 == 0
 * and a 16-byte aligned base; PAPER: ld_train % 2 == 0, 8-byte base). CODES on
 * the tensor cores multiplies exact +-1 operands: e2m1 through the block-scaled
 * fp4 MMA with unit scales when every k_u is a multiple of 256, else e4m3; the
 * scores are the same bit for bit either way.
 * Errors: EOGP_EINVAL, EOGP_EWORKSPACE, EOGP_ECUDA. */
int eogp_score(const void* train, int ld_train, const float* train_scales, int ld_tscale, int N,
               const int* k_per_module, int U, int mode, const void* query, int ld_query,
               const float* query_scales, int ld_qscale, int Q, float* scores, int ld_scores,
               void* ws, size_t ws_bytes, eogp_stream_t stream);

/* ---- store records (App. E.1, Eq. app_payload) --------------------------
 * Per example, for each module u in order: ceil(k_u / 8) bytes of signs
 * (coordinate c at bit c % 8 of byte c / 8) followed by the module's scale as
 * an IEEE half (round to nearest even, little-endian): sum_u (ceil(k_u/8) + 2)
 * bytes, the paper's per-example payload. The paper does not fix the order of
 * signs and scale inside a module's record; signs come first here. */
int eogp_payload_bytes(const int* k_per_module, int U, size_t* bytes_per_example);

/* codes [N x ld_codes] uint32 (modules at their word offsets, as eogp_score
 * reads them) and scales [N x ld_scales] fp32, device -> payload [N x
 * ld_payload] bytes, device (ld_payload >= eogp_payload_bytes). Pad bits of
 * a partial last byte are written as 0.
 * Errors: EOGP_EINVAL, EOGP_ECUDA. */
int eogp_payload_pack(const uint32_t* codes, int ld_codes, const float* scales, int ld_scales, int N,
                      const int* k_per_module, int U, uint8_t* payload, size_t ld_payload,
                      eogp_stream_t stream);

/* Inverse of eogp_payload_pack: payload -> codes (pad bits and pad words 0)
 * and scales (the stored halves, exactly), device.
 * Errors: EOGP_EINVAL, EOGP_ECUDA. */
int eogp_payload_unpack(const uint8_t* payload, size_t ld_payload, int N, const int* k_per_module, int U,
                        uint32_t* codes, int ld_codes, float* scales, int ld_scales, eogp_stream_t stream);

/* ---- ranking (App. C: stored examples ranked per query by score, descending;
 * NDCG@20 reads the first 20) ------------------------------------------- */
#define EOGP_TOPK_MAX 256

int eogp_score_topk_workspace_size(int N, const int* k_per_module, int U, int mode, int Q,
                                   int topk, size_t* bytes);

/* Per query, the `topk` best stored rows under the eogp_score definition of
 * `mode`, without materialising the Q x N scores when the tensor-core kernels
 * apply and topk <= 64 (the ranking then runs in their epilogue; the Q x N
 * matrix is never written). Otherwise the scores go to the workspace and a
 * ranking kernel follows. Arguments as eogp_score, plus:
 *   top_scores [Q x ld_top_scores] fp32 device and top_index [Q x ld_top_index]
 *   int32 device (stored row numbers), ld >= topk: row q lists its best rows by
 *   score descending, equal scores by lower row number; NaN scores never rank;
 *   places beyond N hold (-inf, -1). CODES scores are bitwise those of
 *   eogp_score, so the lists are exact.
 * ws: 256-byte aligned, at least eogp_score_topk_workspace_size bytes.
 * Errors: EOGP_EINVAL (topk outside [1, EOGP_TOPK_MAX], bad sizes),
 *   EOGP_EWORKSPACE, EOGP_EUNSUPPORTED (tensor-core shape with code rows not
 *   aligned as eogp_score's tensor-core path needs), EOGP_ECUDA. */
int eogp_score_topk(const void* train, int ld_train, const float* train_scales, int ld_tscale,
                    int N, const int* k_per_module, int U, int mode, const void* query,
                    int ld_query, const float* query_scales, int ld_qscale, int Q, int topk,
                    float* top_scores, int ld_top_scores, int* top_index, int ld_top_index,
                    void* ws, size_t ws_bytes, eogp_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* EOGP_H */
