// C ABI of libeogp (include/eogp.h): argument checking, the retained-set plan,
// workspace layout and kernel dispatch. No entry point allocates device memory
// except eogp_plan_layer (its small tables, freed by eogp_plan_destroy).
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>
#include <numeric>
#include <vector>

#include "eogp_dev.cuh"
#include "eogp_internal.h"

// Device status word (one per device that loads the library), see eogp_sync_status.
__device__ unsigned int g_eogp_status;

namespace eogp {

static thread_local char g_err[1024];

int set_error(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

void clear_error() { g_err[0] = '\0'; }

// Looked up on every call (cudaGetSymbolAddress allocates nothing and is
// cheap): a cached address would go stale if the device's context were
// destroyed and recreated.
unsigned* status_word() {
  void* p = nullptr;
  if (cudaGetSymbolAddress(&p, g_eogp_status) != cudaSuccess) return nullptr;
  return static_cast<unsigned*>(p);
}

static std::atomic<int> g_opt[2] = {{0}, {0}};

int option(int which) { return (which >= 0 && which < 2) ? g_opt[which].load(std::memory_order_relaxed) : 0; }

static PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int make_tmap(CUtensorMap* tm, CUtensorMapDataType dt, int rank, const void* base,
              const uint64_t* dims, const uint64_t* strides_bytes, const uint32_t* box,
              CUtensorMapSwizzle swz) {
  static std::once_flag once;
  std::call_once(once, [] {
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  if (!g_encode) return set_error(EOGP_ECUDA, "cuTensorMapEncodeTiled is unavailable");
  cuuint64_t d[5];
  cuuint64_t s[4];
  cuuint32_t b[5], es[5];
  for (int r = 0; r < rank; ++r) {
    d[r] = dims[r];
    b[r] = box[r];
    es[r] = 1;
    if (r + 1 < rank) s[r] = strides_bytes[r];
  }
  const CUresult res = g_encode(tm, dt, static_cast<cuuint32_t>(rank), const_cast<void*>(base), d,
                                s, b, es, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (res != CUDA_SUCCESS) return set_error(EOGP_ECUDA, "cuTensorMapEncodeTiled failed (%d)", (int)res);
  return EOGP_OK;
}

}  // namespace eogp

using namespace eogp;

#define CUDA_TRY(x)                                                                      \
  do {                                                                                   \
    cudaError_t e_ = (x);                                                                \
    if (e_ != cudaSuccess)                                                               \
      return set_error(EOGP_ECUDA, "%s failed: %s", #x, cudaGetErrorString(e_));         \
  } while (0)

static inline size_t al256(size_t x) { return (x + 255) & ~size_t(255); }
static inline int round_up(int x, int a) { return (x + a - 1) / a * a; }

// SM count of the current device, cached per device index.
static int sm_count() {
  static std::atomic<int> cache[128];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < 128) {
    const int c = cache[dev].load(std::memory_order_relaxed);
    if (c > 0) return c;
  }
  int v = 0;
  if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0) return 148;
  if (dev < 128) cache[dev].store(v, std::memory_order_relaxed);
  return v;
}

static bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

// ----------------------------------------------------------- kernel timing
namespace {
struct ProfRec {
  cudaEvent_t a, b;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRec> g_prof[EOGP_K_COUNT];
std::vector<cudaEvent_t> g_prof_free;

cudaEvent_t prof_event() {
  if (!g_prof_free.empty()) {
    cudaEvent_t e = g_prof_free.back();
    g_prof_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

// Brackets the launches made during its lifetime with events on `st`.
struct ProfScope {
  int kind;
  cudaStream_t st;
  cudaEvent_t a = nullptr;
  ProfScope(int k, cudaStream_t s) : kind(k), st(s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on) return;
    a = prof_event();
    if (a) cudaEventRecord(a, st);
  }
  ~ProfScope() {
    if (!a) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    cudaEvent_t b = prof_event();
    if (!b) return;
    cudaEventRecord(b, st);
    g_prof[kind].push_back(ProfRec{a, b});
  }
};
}  // namespace

extern "C" int eogp_profile_enable(int on) {
  clear_error();
  std::lock_guard<std::mutex> lk(g_prof_mu);
  g_prof_on = on != 0;
  return EOGP_OK;
}

extern "C" int eogp_profile_read(int kind, int* launches, double* total_ms, int reset) {
  clear_error();
  if (kind < 0 || kind >= EOGP_K_COUNT || !launches || !total_ms) return set_error(EOGP_EINVAL, "bad argument");
  std::lock_guard<std::mutex> lk(g_prof_mu);
  double tot = 0.0;
  for (const ProfRec& r : g_prof[kind]) {
    CUDA_TRY(cudaEventSynchronize(r.b));
    float ms = 0.f;
    CUDA_TRY(cudaEventElapsedTime(&ms, r.a, r.b));
    tot += ms;
  }
  *launches = static_cast<int>(g_prof[kind].size());
  *total_ms = tot;
  if (reset) {
    for (const ProfRec& r : g_prof[kind]) {
      g_prof_free.push_back(r.a);
      g_prof_free.push_back(r.b);
    }
    g_prof[kind].clear();
  }
  return EOGP_OK;
}

extern "C" const char* eogp_last_error(void) { return g_err; }

extern "C" const char* eogp_version(void) { return "eogp-gb300 0.1 (sm_103a)"; }

extern "C" int eogp_sync_status(eogp_stream_t stream) {
  clear_error();
  CUDA_TRY(cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)));
  unsigned* w = status_word();
  if (!w) return set_error(EOGP_ECUDA, "device status word unavailable");
  unsigned v = 0;
  CUDA_TRY(cudaMemcpy(&v, w, sizeof(v), cudaMemcpyDeviceToHost));
  if (v) CUDA_TRY(cudaMemset(w, 0, sizeof(unsigned)));
  if (v & EOGP_ST_TIMEOUT) return set_error(EOGP_ETIMEOUT, "a kernel's bounded wait expired");
  if (v) return set_error(EOGP_EDEVICE, "device-side error flag 0x%x", v);
  return EOGP_OK;
}

// =================================================================== plan

static void plan_free_device(eogp_plan* p) {
  int32_t** ip[] = {&p->d_tile_rc, &p->d_tile_start, &p->d_grp_start, &p->d_ent, &p->d_ent_r,
                    &p->d_ent_off, &p->d_posR,       &p->d_posC,      &p->d_R,
                    &p->d_C};
  for (auto q : ip) {
    if (*q) cudaFree(*q);
    *q = nullptr;
  }
  float** fp[] = {&p->d_ent_scale, &p->d_scale};
  for (auto q : fp) {
    if (*q) cudaFree(*q);
    *q = nullptr;
  }
}

template <typename T>
static int upload(T** dst, const std::vector<T>& src) {
  const size_t bytes = std::max<size_t>(1, src.size()) * sizeof(T);
  CUDA_TRY(cudaMalloc(reinterpret_cast<void**>(dst), bytes));
  if (!src.empty()) CUDA_TRY(cudaMemcpy(*dst, src.data(), src.size() * sizeof(T), cudaMemcpyHostToDevice));
  return EOGP_OK;
}

extern "C" int eogp_plan_layer(const double* lam_S, const double* lam_A, const double* Lambda,
                               int d_in, int d_out, int m, double damping_rel, eogp_plan** out) {
  clear_error();
  if (!out) return set_error(EOGP_EINVAL, "out is NULL");
  *out = nullptr;
  if (d_in < 1 || d_out < 1) return set_error(EOGP_EINVAL, "d_in and d_out must be >= 1");
  const long long d = static_cast<long long>(d_in) * d_out;
  if (d > 0xFFFFFFFFLL) return set_error(EOGP_EUNSUPPORTED, "d_in * d_out must be < 2^32");
  if (m < 1 || m > d) return set_error(EOGP_EINVAL, "m must be in [1, d_in*d_out]");
  if (!(damping_rel >= 0.0) || !std::isfinite(damping_rel))
    return set_error(EOGP_EINVAL, "damping_rel must be finite and >= 0");
  const bool product = (lam_S != nullptr) || (lam_A != nullptr);
  if (product && Lambda) return set_error(EOGP_EINVAL, "give either (lam_S, lam_A) or Lambda");
  if (product && (!lam_S || !lam_A)) return set_error(EOGP_EINVAL, "both lam_S and lam_A are required");
  if (!product && !Lambda) return set_error(EOGP_EINVAL, "no eigenvalues given");
  // A plan made where no CUDA device is visible keeps only its host tables
  // (device = -1); eogp_compress_layer rejects it.
  int dev = -1, ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
    cudaGetLastError();
    dev = -1;
  } else {
    CUDA_TRY(cudaGetDevice(&dev));
  }

  // Eigenvalue of Kronecker position p = i*d_out + j (basis vector Q_A[:,i] (x) Q_S[:,j]).
  auto val = [&](uint32_t p) -> double {
    const uint32_t i = p / static_cast<uint32_t>(d_out), j = p % static_cast<uint32_t>(d_out);
    return product ? lam_S[j] * lam_A[i] : Lambda[static_cast<size_t>(j) * d_in + i];
  };
  // Validate and form the damping lambda = rel * tr(Lambda) / d (Eq. app_module_damping).
  double tr = 0.0;
  if (product) {
    for (int j = 0; j < d_out; ++j)
      if (!std::isfinite(lam_S[j]) || lam_S[j] < 0) return set_error(EOGP_EINVAL, "lam_S must be finite, >= 0");
    for (int i = 0; i < d_in; ++i)
      if (!std::isfinite(lam_A[i]) || lam_A[i] < 0) return set_error(EOGP_EINVAL, "lam_A must be finite, >= 0");
  }
  for (long long p = 0; p < d; ++p) {
    const double v = val(static_cast<uint32_t>(p));
    if (!std::isfinite(v) || v < 0) return set_error(EOGP_EINVAL, "eigenvalues must be finite and >= 0");
    tr += v;
  }
  auto* P = new eogp_plan();
  P->d_in = d_in;
  P->d_out = d_out;
  P->m = m;
  P->device = dev;
  P->lambda = damping_rel * tr / static_cast<double>(d);

  // Top-m selection: value descending, Kronecker position ascending on ties.
  std::vector<uint32_t> pos(static_cast<size_t>(d));
  std::iota(pos.begin(), pos.end(), 0u);
  auto before = [&](uint32_t a, uint32_t b) {
    const double va = val(a), vb = val(b);
    if (va != vb) return va > vb;
    return a < b;
  };
  if (m < d) std::nth_element(pos.begin(), pos.begin() + m, pos.end(), before);
  std::sort(pos.begin(), pos.begin() + m, before);
  pos.resize(m);

  P->j.resize(m);
  P->i.resize(m);
  P->scale.resize(m);
  std::vector<int32_t> rowmap(d_out, -1), colmap(d_in, -1);
  for (int r = 0; r < m; ++r) {
    P->i[r] = static_cast<int32_t>(pos[r] / d_out);
    P->j[r] = static_cast<int32_t>(pos[r] % d_out);
    P->scale[r] = static_cast<float>(1.0 / std::sqrt(val(pos[r]) + P->lambda));
    rowmap[P->j[r]] = 1;
    colmap[P->i[r]] = 1;
  }
  for (int j = 0; j < d_out; ++j)
    if (rowmap[j] >= 0) {
      rowmap[j] = static_cast<int32_t>(P->R.size());
      P->R.push_back(j);
    }
  for (int i = 0; i < d_in; ++i)
    if (colmap[i] >= 0) {
      colmap[i] = static_cast<int32_t>(P->C.size());
      P->C.push_back(i);
    }
  P->posR.resize(m);
  P->posC.resize(m);
  for (int r = 0; r < m; ++r) {
    P->posR[r] = rowmap[P->j[r]];
    P->posC[r] = colmap[P->i[r]];
  }
  // Active 128 x 128 tiles; inside a tile, entries grouped by the 32-column
  // chunk co / 32 that the contraction epilogue stages at a time, canonical
  // order inside a group.
  std::vector<int> order(m);
  std::iota(order.begin(), order.end(), 0);
  auto tkey = [&](int r) { return (static_cast<int64_t>(P->posR[r] / 128) << 32) | (P->posC[r] / 128); };
  auto gkey = [&](int r) { return (P->posC[r] % 128) / 32; };
  std::stable_sort(order.begin(), order.end(), [&](int a, int b) {
    const int64_t ta = tkey(a), tb = tkey(b);
    if (ta != tb) return ta < tb;
    return gkey(a) < gkey(b);
  });
  int64_t last = -1;
  for (int e = 0; e < m; ++e) {
    const int r = order[e];
    const int64_t k = tkey(r);
    if (k != last) {
      P->tile_rc.push_back(static_cast<int32_t>(((P->posR[r] / 128) << 16) | (P->posC[r] / 128)));
      P->tile_start.push_back(e);
      last = k;
    }
    P->ent_r.push_back(r);
    P->ent_off.push_back(((P->posR[r] % 128) << 8) | (P->posC[r] % 128));
    P->ent_scale.push_back(P->scale[r]);
  }
  P->tile_start.push_back(m);
  // Group boundaries: for tile t, group g = co / 32.
  P->grp_start.assign(static_cast<size_t>(P->n_tiles()) * 4 + 1, 0);
  for (int t = 0; t < P->n_tiles(); ++t) {
    int e = P->tile_start[t];
    for (int grp = 0; grp < 4; ++grp) {
      P->grp_start[t * 4 + grp] = e;
      while (e < P->tile_start[t + 1] && (P->ent_off[e] & 255) / 32 == grp) ++e;
    }
  }
  P->grp_start[static_cast<size_t>(P->n_tiles()) * 4] = m;
  P->ent.resize(static_cast<size_t>(m) * 4);
  for (int e = 0; e < m; ++e) {
    int32_t sbits;
    std::memcpy(&sbits, &P->ent_scale[e], 4);
    P->ent[4 * e + 0] = P->ent_r[e];
    P->ent[4 * e + 1] = P->ent_off[e];
    P->ent[4 * e + 2] = sbits;
    P->ent[4 * e + 3] = 0;
  }
  if (P->nR() / 128 >= 32768 || P->nC() / 128 >= 65536) {
    delete P;
    return set_error(EOGP_EUNSUPPORTED, "retained block too large");
  }

  int rc = EOGP_OK;
  if (dev >= 0 && ((rc = upload(&P->d_tile_rc, P->tile_rc)) || (rc = upload(&P->d_tile_start, P->tile_start)) ||
      (rc = upload(&P->d_grp_start, P->grp_start)) || (rc = upload(&P->d_ent, P->ent)) ||
      (rc = upload(&P->d_ent_r, P->ent_r)) || (rc = upload(&P->d_ent_off, P->ent_off)) ||
      (rc = upload(&P->d_ent_scale, P->ent_scale)) || (rc = upload(&P->d_posR, P->posR)) ||
      (rc = upload(&P->d_posC, P->posC)) || (rc = upload(&P->d_scale, P->scale)) ||
      (rc = upload(&P->d_R, P->R)) || (rc = upload(&P->d_C, P->C)))) {
    plan_free_device(P);
    delete P;
    return rc;
  }
  *out = P;
  return EOGP_OK;
}

extern "C" void eogp_plan_destroy(eogp_plan* plan) {
  if (!plan) return;
  if (plan->device >= 0) {
    int cur = -1;
    cudaGetDevice(&cur);
    if (plan->device != cur) cudaSetDevice(plan->device);
    plan_free_device(plan);
    if (cur >= 0 && plan->device != cur) cudaSetDevice(cur);
  }
  delete plan;
}

extern "C" int eogp_plan_get_info(const eogp_plan* plan, eogp_plan_info* info) {
  clear_error();
  if (!plan || !info) return set_error(EOGP_EINVAL, "NULL argument");
  info->d_in = plan->d_in;
  info->d_out = plan->d_out;
  info->m = plan->m;
  info->nR = plan->nR();
  info->nC = plan->nC();
  info->n_tiles = plan->n_tiles();
  info->lambda = plan->lambda;
  return EOGP_OK;
}

extern "C" int eogp_plan_get_retained(const eogp_plan* plan, int32_t* j, int32_t* i, float* scale) {
  clear_error();
  if (!plan) return set_error(EOGP_EINVAL, "NULL plan");
  if (j) std::memcpy(j, plan->j.data(), plan->j.size() * sizeof(int32_t));
  if (i) std::memcpy(i, plan->i.data(), plan->i.size() * sizeof(int32_t));
  if (scale) std::memcpy(scale, plan->scale.data(), plan->scale.size() * sizeof(float));
  return EOGP_OK;
}

extern "C" int eogp_plan_get_sets(const eogp_plan* plan, int32_t* R, int32_t* C) {
  clear_error();
  if (!plan) return set_error(EOGP_EINVAL, "NULL plan");
  if (R) std::memcpy(R, plan->R.data(), plan->R.size() * sizeof(int32_t));
  if (C) std::memcpy(C, plan->C.data(), plan->C.size() * sizeof(int32_t));
  return EOGP_OK;
}

static int check_device(const eogp_plan* plan) {
  if (plan->device < 0) return set_error(EOGP_EINVAL, "plan was built without a CUDA device");
  int dev = 0;
  CUDA_TRY(cudaGetDevice(&dev));
  if (dev != plan->device) return set_error(EOGP_EINVAL, "plan belongs to device %d, current is %d", plan->device, dev);
  return EOGP_OK;
}

extern "C" int eogp_plan_gather_rows(const eogp_plan* plan, int which, int dtype, const void* V_full,
                                     int ld_full, void* V_ret, eogp_stream_t stream) {
  clear_error();
  if (!plan || !V_full || !V_ret) return set_error(EOGP_EINVAL, "NULL argument");
  if (which != 0 && which != 1) return set_error(EOGP_EINVAL, "which must be 0 (A) or 1 (S)");
  if (dtype != EOGP_F32 && dtype != EOGP_BF16) return set_error(EOGP_EINVAL, "bad dtype");
  const int d = which == 0 ? plan->d_in : plan->d_out;
  if (ld_full < d) return set_error(EOGP_EINVAL, "ld_full < row length");
  if (int rc = check_device(plan)) return rc;
  const int n = which == 0 ? plan->nC() : plan->nR();
  const int32_t* idx = which == 0 ? plan->d_C : plan->d_R;
  CUDA_TRY(launch_gather_rows(V_full, ld_full, dtype == EOGP_F32 ? 4 : 2, idx, n, d, V_ret,
                              reinterpret_cast<cudaStream_t>(stream)));
  return EOGP_OK;
}

// ============================================================ compression

namespace {

struct Layout {
  size_t va = 0, vs = 0;  // device copies of host eigenbases (bases_on_host)
  // bf16 path
  int ldA = 0, ldS = 0, ldzb = 0, ldp = 0, splits = 1;
  size_t at_hi = 0, at_lo = 0, st_hi = 0, st_lo = 0, zhi = 0, zlo = 0, part = 0;
  // f32 path
  size_t at = 0, st = 0, z = 0, x = 0;
  size_t total = 0;
};

TcGemmCfg proj_cfg() { return TcGemmCfg{128, 4}; }
constexpr int kContractStages = 3;

int proj_splits(int B, int k, int m) {
  const int tiles = ((B + 127) / 128) * ((k + proj_cfg().BN - 1) / proj_cfg().BN);
  const int nkb = (m + 63) / 64;
  int want = (2 * sm_count() + tiles - 1) / tiles;
  want = std::min(want, std::max(1, nkb / 4));
  return tc_gemm_splits_used(m, std::max(1, want));
}

// EOGP-R descriptor: the SRHT replaces the PCA projection.
bool uses_srht(const eogp_layer_desc* L) { return !L->Pt && L->srht_rows; }

int make_layout(const eogp_layer_desc* L, int B, int mode, Layout* o) {
  const eogp_plan* P = L->plan;
  const size_t M = static_cast<size_t>(B) * L->T;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off += al256(bytes);
    return at;
  };
  if (L->bases_on_host) {
    const size_t esz = L->dtype == EOGP_F32 ? 4 : 2;
    o->va = take(static_cast<size_t>(P->nC()) * L->d_in * esz);
    o->vs = take(static_cast<size_t>(P->nR()) * L->d_out * esz);
  }
  if (L->dtype == EOGP_BF16) {
    o->ldA = round_up(std::max(1, P->nC()), 128);
    o->ldS = round_up(std::max(1, P->nR()), 128);
    o->at_hi = take(M * o->ldA * 2);
    o->at_lo = take(M * o->ldA * 2);
    o->st_hi = take(M * o->ldS * 2);
    o->st_lo = take(M * o->ldS * 2);
    if (mode != EOGP_OUT_FIRST_STAGE) {
      o->ldzb = round_up(L->m, 64);
      o->zhi = take(static_cast<size_t>(B) * o->ldzb * 2);
      o->zlo = take(static_cast<size_t>(B) * o->ldzb * 2);
      if (!uses_srht(L)) {
        o->ldp = round_up(L->k, 16);
        o->splits = proj_splits(B, L->k, L->m);
        o->part = take(static_cast<size_t>(o->splits) * B * o->ldp * 4);
      }
    }
  } else {
    o->at = take(M * P->nC() * 4);
    o->st = take(M * P->nR() * 4);
    if (mode != EOGP_OUT_FIRST_STAGE) o->z = take(static_cast<size_t>(B) * L->m * 4);
    if (mode == EOGP_OUT_CODES && !uses_srht(L)) o->x = take(static_cast<size_t>(B) * L->k * 4);
  }
  o->total = std::max<size_t>(off, 256);
  return EOGP_OK;
}

int check_desc(const eogp_layer_desc* L, int B, int mode) {
  if (!L) return set_error(EOGP_EINVAL, "descriptor is NULL");
  if (!L->plan) return set_error(EOGP_EINVAL, "descriptor has no plan");
  const eogp_plan* P = L->plan;
  const int bias = L->bias_A ? 1 : 0;
  if (L->d_in + bias != P->d_in || L->d_out != P->d_out || L->m != P->m)
    return set_error(EOGP_EINVAL,
                     "descriptor shape (%d%s, %d, m=%d) differs from the plan (%d, %d, m=%d)", L->d_in,
                     bias ? " + bias" : "", L->d_out, L->m, P->d_in, P->d_out, P->m);
  if (L->T < 1) return set_error(EOGP_EINVAL, "T must be >= 1");
  if (B < 0) return set_error(EOGP_EINVAL, "B must be >= 0");
  if (mode < EOGP_OUT_FIRST_STAGE || mode > EOGP_OUT_CODES) return set_error(EOGP_EINVAL, "bad out_mode");
  if (L->dtype != EOGP_F32 && L->dtype != EOGP_BF16) return set_error(EOGP_EINVAL, "bad dtype");
  if (mode != EOGP_OUT_FIRST_STAGE) {
    if (uses_srht(L)) {
      if (L->m > EOGP_SRHT_MAX_M) return set_error(EOGP_EUNSUPPORTED, "SRHT needs m <= %d", EOGP_SRHT_MAX_M);
      if (L->k < 1 || L->k > srht_width(L->m)) return set_error(EOGP_EINVAL, "SRHT k must be in [1, p]");
      if (!L->srht_signs) return set_error(EOGP_EINVAL, "srht_signs is NULL");
    } else {
      if (L->k < 1 || L->k > L->m) return set_error(EOGP_EINVAL, "k must be in [1, m]");
      if (!L->Pt) return set_error(EOGP_EINVAL, "Pt is NULL (and no SRHT given)");
    }
  }
  if (!L->VA || !L->VS) return set_error(EOGP_EINVAL, "VA / VS is NULL");
  if (L->dtype == EOGP_BF16) {
    if (L->d_in % 8 || L->d_out % 8 || L->m % 8)
      return set_error(EOGP_EUNSUPPORTED, "bf16 path needs d_in, d_out, m multiples of 8");
    if ((!L->bases_on_host && (!aligned16(L->VA) || !aligned16(L->VS))) || (L->Pt && !aligned16(L->Pt)))
      return set_error(EOGP_EINVAL, "bf16 operands must be 16-byte aligned");
    if (static_cast<long long>(B) * L->T > 0x7FFFFFFFLL) return set_error(EOGP_EUNSUPPORTED, "B*T too large");
  }
  return EOGP_OK;
}

}  // namespace

extern "C" int eogp_compress_workspace_size(const eogp_layer_desc* L, int B, int out_mode, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  if (int rc = check_desc(L, B, out_mode)) return rc;
  Layout lo;
  make_layout(L, B, out_mode, &lo);
  *bytes = lo.total;
  return EOGP_OK;
}

extern "C" int eogp_compress_layer(const eogp_layer_desc* L, const void* a, const void* s, int B,
                                   int out_mode, float* out, int ld_out, uint32_t* codes,
                                   int ld_codes, float* scales, int ld_scales, void* ws,
                                   size_t ws_bytes, eogp_stream_t stream) {
  clear_error();
  if (int rc = check_desc(L, B, out_mode)) return rc;
  if (B == 0) return EOGP_OK;
  if (!a || !s) return set_error(EOGP_EINVAL, "a / s is NULL");
  if (out_mode == EOGP_OUT_CODES) {
    if (!codes || !scales) return set_error(EOGP_EINVAL, "codes / scales is NULL");
    if (ld_codes < (L->k + 31) / 32 || ld_scales < 1) return set_error(EOGP_EINVAL, "ld_codes / ld_scales too small");
  } else {
    if (!out) return set_error(EOGP_EINVAL, "out is NULL");
    const int need = out_mode == EOGP_OUT_FIRST_STAGE ? L->m : L->k;
    if (ld_out < need) return set_error(EOGP_EINVAL, "ld_out too small");
  }
  if (int rc = check_device(L->plan)) return rc;
  Layout lo;
  make_layout(L, B, out_mode, &lo);
  if (!ws || ws_bytes < lo.total)
    return set_error(EOGP_EWORKSPACE, "workspace of %zu bytes needed, %zu given", lo.total, ws_bytes);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  const eogp_plan* P = L->plan;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  char* w = static_cast<char*>(ws);
  const int M = B * L->T;
  const void* VA = L->VA;
  const void* VS = L->VS;
  if (L->bases_on_host) {
    const size_t esz = L->dtype == EOGP_F32 ? 4 : 2;
    CUDA_TRY(cudaMemcpyAsync(w + lo.va, L->VA, static_cast<size_t>(P->nC()) * L->d_in * esz,
                             cudaMemcpyHostToDevice, st));
    CUDA_TRY(cudaMemcpyAsync(w + lo.vs, L->VS, static_cast<size_t>(P->nR()) * L->d_out * esz,
                             cudaMemcpyHostToDevice, st));
    VA = w + lo.va;
    VS = w + lo.vs;
  }

  if (L->dtype == EOGP_BF16) {
    if (!aligned16(a) || !aligned16(s)) return set_error(EOGP_EINVAL, "a / s must be 16-byte aligned");
    void* at_hi = w + lo.at_hi;
    void* at_lo = w + lo.at_lo;
    void* st_hi = w + lo.st_hi;
    void* st_lo = w + lo.st_lo;
    // Kronecker rotations restricted to the retained columns C / rows R (Sec. 2.2).
    {
      ProfScope ps(EOGP_K_ROTATE, st);
      CUDA_TRY(launch_tc_rotate(M, L->d_in, a, L->d_in, VA, L->d_in, P->nC(), at_hi, at_lo,
                                lo.ldA, L->T, L->bias_A, nullptr, sm_count(), status, st));
    }
    {
      ProfScope ps(EOGP_K_ROTATE, st);
      CUDA_TRY(launch_tc_rotate(M, L->d_out, s, L->d_out, VS, L->d_out, P->nR(), st_hi, st_lo,
                                lo.ldS, L->T, nullptr, L->lengths, sm_count(), status, st));
    }
    // Per-example contraction over tokens + scale/gather into z (Eq. first_stage).
    const bool fs = out_mode == EOGP_OUT_FIRST_STAGE;
    {
      ProfScope ps(EOGP_K_CONTRACT, st);
      CUDA_TRY(launch_tc_contract(st_hi, st_lo, lo.ldS, at_hi, at_lo, lo.ldA, B, L->T, P,
                                  fs ? out : nullptr, ld_out, fs ? nullptr : w + lo.zhi,
                                  fs ? nullptr : w + lo.zlo, lo.ldzb, kContractStages, sm_count(),
                                  status, st));
    }
    if (fs) return EOGP_OK;
    if (uses_srht(L)) {
      // EOGP-R: x = sqrt(p/k) R H_p D J z, with the sign/scale pack in the same kernel.
      ProfScope ps(EOGP_K_PROJECT, st);
      const bool cd = out_mode == EOGP_OUT_CODES;
      CUDA_TRY(launch_srht(w + lo.zhi, w + lo.zlo, true, lo.ldzb, B, L->m, L->srht_signs, L->srht_rows,
                           L->k, cd ? nullptr : out, ld_out, cd ? codes : nullptr, ld_codes,
                           cd ? scales : nullptr, ld_scales, status, st));
      return EOGP_OK;
    }
    // x = P^T z (Eq. second_stage), split over K; then sum + sign/pack (Eq. onebit).
    float* part = reinterpret_cast<float*>(w + lo.part);
    const size_t slab = static_cast<size_t>(B) * lo.ldp;
    {
      ProfScope ps(EOGP_K_PROJECT, st);
      CUDA_TRY(launch_tc_gemm(B, L->k, L->m, w + lo.zhi, w + lo.zlo, lo.ldzb, L->Pt, L->m, L->k,
                              lo.splits, 1, part, nullptr, lo.ldp, slab, proj_cfg(), status, st));
    }
    ProfScope ps(EOGP_K_PACK, st);
    if (out_mode == EOGP_OUT_COORDS)
      CUDA_TRY(launch_pack(part, lo.splits, slab, lo.ldp, B, L->k, out, ld_out, nullptr, 0, nullptr,
                           0, status, st));
    else
      CUDA_TRY(launch_pack(part, lo.splits, slab, lo.ldp, B, L->k, nullptr, 0, codes, ld_codes,
                           scales, ld_scales, status, st));
    return EOGP_OK;
  }

  // fp32 CUDA-core path.
  ProfScope ps(EOGP_K_SIMT, st);
  const float* af = static_cast<const float*>(a);
  const float* sf = static_cast<const float*>(s);
  float* at = reinterpret_cast<float*>(w + lo.at);
  float* stt = reinterpret_cast<float*>(w + lo.st);
  const int nC = P->nC(), nR = P->nR();
  CUDA_TRY(launch_simt_gemm(M, nC, L->d_in, 1.f, af, L->d_in, 1, static_cast<const float*>(VA),
                            L->d_in, 1, at, nC, st));
  CUDA_TRY(launch_simt_gemm(M, nR, L->d_out, 1.f, sf, L->d_out, 1, static_cast<const float*>(VS),
                            L->d_out, 1, stt, nR, st));
  CUDA_TRY(launch_rows_fixup(at, M, nC, nC, L->T, L->bias_A, nullptr, st));
  CUDA_TRY(launch_rows_fixup(stt, M, nR, nR, L->T, nullptr, L->lengths, st));
  float* z = out_mode == EOGP_OUT_FIRST_STAGE ? out : reinterpret_cast<float*>(w + lo.z);
  const int ldz = out_mode == EOGP_OUT_FIRST_STAGE ? ld_out : L->m;
  CUDA_TRY(launch_contract_f32(at, nC, stt, nR, B, L->T, L->m, P->d_posR, P->d_posC, P->d_scale, z,
                               ldz, st));
  if (out_mode == EOGP_OUT_FIRST_STAGE) return EOGP_OK;
  if (uses_srht(L)) {
    const bool cd = out_mode == EOGP_OUT_CODES;
    CUDA_TRY(launch_srht(z, nullptr, false, ldz, B, L->m, L->srht_signs, L->srht_rows, L->k,
                         cd ? nullptr : out, ld_out, cd ? codes : nullptr, ld_codes,
                         cd ? scales : nullptr, ld_scales, status, st));
    return EOGP_OK;
  }
  float* x = out_mode == EOGP_OUT_COORDS ? out : reinterpret_cast<float*>(w + lo.x);
  const int ldx = out_mode == EOGP_OUT_COORDS ? ld_out : L->k;
  CUDA_TRY(launch_simt_gemm(B, L->k, L->m, 1.f, z, ldz, 1, static_cast<const float*>(L->Pt), L->m, 1,
                            x, ldx, st));
  if (out_mode == EOGP_OUT_CODES)
    CUDA_TRY(launch_pack(x, 1, 0, ldx, B, L->k, nullptr, 0, codes, ld_codes, scales, ld_scales,
                         status, st));
  return EOGP_OK;
}

// ================================================================ host-resident inputs

namespace {

// Examples per chunk when the caller passes 0: about 64 MB of a and s.
int host_chunk(const eogp_layer_desc* L, int B, int chunk) {
  if (chunk > 0) return std::min(chunk, std::max(B, 1));
  const size_t esz = L->dtype == EOGP_F32 ? 4 : 2;
  const size_t per = static_cast<size_t>(L->T) * (L->d_in + L->d_out) * esz;
  const size_t c = std::max<size_t>(1, (size_t(64) << 20) / std::max<size_t>(per, 1));
  return static_cast<int>(std::min<size_t>(c, std::max(B, 1)));
}

struct HostLayout {
  int chunk = 1;
  size_t a_bytes = 0, s_bytes = 0;  // one chunk's a and s
  size_t stage[2] = {0, 0};         // double-buffered staging of a chunk's a then s
  size_t va = 0, vs = 0;            // device copies of host eigenbases
  size_t comp = 0, comp_bytes = 0;  // eogp_compress_layer workspace for one chunk
  size_t total = 0;
};

HostLayout host_layout(const eogp_layer_desc* L, int B, int chunk, int mode) {
  HostLayout h;
  h.chunk = host_chunk(L, B, chunk);
  const size_t esz = L->dtype == EOGP_F32 ? 4 : 2;
  h.a_bytes = static_cast<size_t>(h.chunk) * L->T * L->d_in * esz;
  h.s_bytes = static_cast<size_t>(h.chunk) * L->T * L->d_out * esz;
  size_t off = 0;
  for (int i = 0; i < 2; ++i) {
    h.stage[i] = off;
    off += al256(h.a_bytes) + al256(h.s_bytes);
  }
  if (L->bases_on_host) {
    h.va = off;
    off += al256(static_cast<size_t>(L->plan->nC()) * L->d_in * esz);
    h.vs = off;
    off += al256(static_cast<size_t>(L->plan->nR()) * L->d_out * esz);
  }
  eogp_layer_desc d = *L;
  d.bases_on_host = 0;  // the chunks read the device copies
  Layout lo;
  make_layout(&d, h.chunk, mode, &lo);
  h.comp = off;
  h.comp_bytes = lo.total;
  h.total = off + lo.total;
  return h;
}

// Several modules of one host-input call share one workspace: nsets sets of
// staging buffers (and eigenbasis copies), used by alternate modules, each as
// large as the largest module's, then the eogp_compress_layer workspace of the
// largest. With one module this is exactly that module's HostLayout.
struct HostMultiLayout {
  int nsets = 1;
  size_t set_bytes = 0, comp = 0, comp_bytes = 0, total = 0;
};

HostMultiLayout host_multi_layout(const eogp_layer_desc* const* L, int n, int B, int chunk, int mode) {
  HostMultiLayout m;
  m.nsets = n > 1 ? 2 : 1;
  for (int u = 0; u < n; ++u) {
    const HostLayout h = host_layout(L[u], B, chunk, mode);
    m.set_bytes = std::max(m.set_bytes, al256(h.comp));
    m.comp_bytes = std::max(m.comp_bytes, h.comp_bytes);
  }
  m.comp = static_cast<size_t>(m.nsets) * m.set_bytes;
  m.total = m.comp + m.comp_bytes;
  return m;
}

// Stream and events of one host-input call, released when it returns (the
// runtime frees them once the work queued on them has completed). Per set of
// staging buffers: chunk buffer b landed / computed, and the set's last module
// computed.
struct HostCallRes {
  cudaStream_t cs = nullptr;
  cudaEvent_t entry = nullptr, landed[2][2] = {}, done[2][2] = {}, set_done[2] = {};
  ~HostCallRes() {
    if (entry) cudaEventDestroy(entry);
    for (int i = 0; i < 2; ++i) {
      for (int j = 0; j < 2; ++j) {
        if (landed[i][j]) cudaEventDestroy(landed[i][j]);
        if (done[i][j]) cudaEventDestroy(done[i][j]);
      }
      if (set_done[i]) cudaEventDestroy(set_done[i]);
    }
    if (cs) cudaStreamDestroy(cs);
  }
};

int check_host_modules(const eogp_layer_desc* const* L, int n, const void* const* a, const void* const* s,
                       int B, int chunk, int out_mode, float* const* out, uint32_t* const* codes,
                       float* const* scales) {
  if (n < 1) return set_error(EOGP_EINVAL, "n must be >= 1");
  if (!L || !a || !s) return set_error(EOGP_EINVAL, "descriptor / a / s array is NULL");
  if (chunk < 0) return set_error(EOGP_EINVAL, "chunk must be >= 0");
  for (int u = 0; u < n; ++u) {
    if (int rc = check_desc(L[u], B, out_mode)) return rc;
    if (B == 0) continue;
    if (!a[u] || !s[u]) return set_error(EOGP_EINVAL, "a / s of module %d is NULL", u);
    if (out_mode == EOGP_OUT_CODES) {
      if (!codes || !scales || !codes[u] || !scales[u])
        return set_error(EOGP_EINVAL, "codes / scales of module %d is NULL", u);
    } else if (!out || !out[u]) {
      return set_error(EOGP_EINVAL, "out of module %d is NULL", u);
    }
  }
  return EOGP_OK;
}

// The modules' chunks, in order: copies on a copy stream, compute on `st`.
// Module u uses set u % nsets; its copies first wait for the compute of the
// module that last used the set (u - nsets), or, for the first modules, for
// the work already queued on `st`.
int run_host_modules(const eogp_layer_desc* const* L, int n, const void* const* a, const void* const* s, int B,
                     int chunk, int out_mode, float* const* out, int ld_out, uint32_t* const* codes,
                     int ld_codes, float* const* scales, int ld_scales, void* ws, size_t ws_bytes,
                     cudaStream_t st) {
  const HostMultiLayout m = host_multi_layout(L, n, B, chunk, out_mode);
  if (!ws || ws_bytes < m.total)
    return set_error(EOGP_EWORKSPACE, "workspace of %zu bytes needed, %zu given", m.total, ws_bytes);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  for (int u = 0; u < n; ++u)
    if (int rc = check_device(L[u]->plan)) return rc;
  char* w = static_cast<char*>(ws);
  HostCallRes r;
  CUDA_TRY(cudaStreamCreateWithFlags(&r.cs, cudaStreamNonBlocking));
  CUDA_TRY(cudaEventCreateWithFlags(&r.entry, cudaEventDisableTiming));
  for (int i = 0; i < m.nsets; ++i) {
    for (int j = 0; j < 2; ++j) {
      CUDA_TRY(cudaEventCreateWithFlags(&r.landed[i][j], cudaEventDisableTiming));
      CUDA_TRY(cudaEventCreateWithFlags(&r.done[i][j], cudaEventDisableTiming));
    }
    CUDA_TRY(cudaEventCreateWithFlags(&r.set_done[i], cudaEventDisableTiming));
  }
  // Work already queued on `st` (an earlier call) may still read the staging
  // buffers: the first copies wait for it.
  CUDA_TRY(cudaEventRecord(r.entry, st));
  CUDA_TRY(cudaStreamWaitEvent(r.cs, r.entry, 0));
  const bool cd = out_mode == EOGP_OUT_CODES;
  for (int u = 0; u < n; ++u) {
    const eogp_layer_desc* Lu = L[u];
    const int set = u % m.nsets;
    char* base = w + static_cast<size_t>(set) * m.set_bytes;
    // the set is free once the module that used it before has been computed
    if (u >= m.nsets) CUDA_TRY(cudaStreamWaitEvent(r.cs, r.set_done[set], 0));
    const HostLayout h = host_layout(Lu, B, chunk, out_mode);
    const size_t esz = Lu->dtype == EOGP_F32 ? 4 : 2;
    const size_t a_row = static_cast<size_t>(Lu->T) * Lu->d_in * esz;  // bytes of one example's a
    const size_t s_row = static_cast<size_t>(Lu->T) * Lu->d_out * esz;
    eogp_layer_desc d = *Lu;
    if (Lu->bases_on_host) {
      CUDA_TRY(cudaMemcpyAsync(base + h.va, Lu->VA, static_cast<size_t>(Lu->plan->nC()) * Lu->d_in * esz,
                               cudaMemcpyDefault, r.cs));
      CUDA_TRY(cudaMemcpyAsync(base + h.vs, Lu->VS, static_cast<size_t>(Lu->plan->nR()) * Lu->d_out * esz,
                               cudaMemcpyDefault, r.cs));
      d.VA = base + h.va;
      d.VS = base + h.vs;
      d.bases_on_host = 0;
    }
    const int n_chunks = (B + h.chunk - 1) / h.chunk;
    for (int c = 0; c < n_chunks; ++c) {
      const int b0 = c * h.chunk, nb = std::min(h.chunk, B - b0), buf = c & 1;
      char* sa = base + h.stage[buf];
      char* ss = sa + al256(h.a_bytes);
      // Copy stream: the staging buffer is free once chunk c - 2 has been computed.
      if (c >= 2) CUDA_TRY(cudaStreamWaitEvent(r.cs, r.done[set][buf], 0));
      CUDA_TRY(cudaMemcpyAsync(sa, static_cast<const char*>(a[u]) + b0 * a_row, nb * a_row, cudaMemcpyDefault,
                               r.cs));
      CUDA_TRY(cudaMemcpyAsync(ss, static_cast<const char*>(s[u]) + b0 * s_row, nb * s_row, cudaMemcpyDefault,
                               r.cs));
      CUDA_TRY(cudaEventRecord(r.landed[set][buf], r.cs));
      // Compute stream: chunk c once its inputs have landed.
      CUDA_TRY(cudaStreamWaitEvent(st, r.landed[set][buf], 0));
      d.lengths = Lu->lengths ? Lu->lengths + b0 : nullptr;
      if (int rc = eogp_compress_layer(&d, sa, ss, nb, out_mode,
                                       cd ? nullptr : out[u] + static_cast<size_t>(b0) * ld_out, ld_out,
                                       cd ? codes[u] + static_cast<size_t>(b0) * ld_codes : nullptr, ld_codes,
                                       cd ? scales[u] + static_cast<size_t>(b0) * ld_scales : nullptr, ld_scales,
                                       w + m.comp, m.comp_bytes, reinterpret_cast<eogp_stream_t>(st)))
        return rc;
      CUDA_TRY(cudaEventRecord(r.done[set][buf], st));
    }
    CUDA_TRY(cudaEventRecord(r.set_done[set], st));
  }
  return EOGP_OK;
}

}  // namespace

extern "C" int eogp_compress_host_workspace_size(const eogp_layer_desc* L, int B, int chunk,
                                                 int out_mode, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  if (chunk < 0) return set_error(EOGP_EINVAL, "chunk must be >= 0");
  if (int rc = check_desc(L, B, out_mode)) return rc;
  *bytes = host_multi_layout(&L, 1, B, chunk, out_mode).total;
  return EOGP_OK;
}

extern "C" int eogp_compress_layer_host(const eogp_layer_desc* L, const void* a, const void* s, int B,
                                        int chunk, int out_mode, float* out, int ld_out, uint32_t* codes,
                                        int ld_codes, float* scales, int ld_scales, void* ws,
                                        size_t ws_bytes, eogp_stream_t stream) {
  clear_error();
  if (int rc = check_host_modules(&L, 1, &a, &s, B, chunk, out_mode, &out, &codes, &scales)) return rc;
  if (B == 0) return EOGP_OK;
  return run_host_modules(&L, 1, &a, &s, B, chunk, out_mode, &out, ld_out, &codes, ld_codes, &scales, ld_scales,
                          ws, ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int eogp_compress_layers_host_workspace_size(const eogp_layer_desc* const* L, int n, int B, int chunk,
                                                        int out_mode, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  if (n < 1) return set_error(EOGP_EINVAL, "n must be >= 1");
  if (!L) return set_error(EOGP_EINVAL, "descriptor array is NULL");
  if (chunk < 0) return set_error(EOGP_EINVAL, "chunk must be >= 0");
  for (int u = 0; u < n; ++u)
    if (int rc = check_desc(L[u], B, out_mode)) return rc;
  *bytes = host_multi_layout(L, n, B, chunk, out_mode).total;
  return EOGP_OK;
}

extern "C" int eogp_compress_layers_host(const eogp_layer_desc* const* L, int n, const void* const* a,
                                         const void* const* s, int B, int chunk, int out_mode, float* const* out,
                                         int ld_out, uint32_t* const* codes, int ld_codes, float* const* scales,
                                         int ld_scales, void* ws, size_t ws_bytes, eogp_stream_t stream) {
  clear_error();
  if (int rc = check_host_modules(L, n, a, s, B, chunk, out_mode, out, codes, scales)) return rc;
  if (B == 0) return EOGP_OK;
  return run_host_modules(L, n, a, s, B, chunk, out_mode, out, ld_out, codes, ld_codes, scales, ld_scales, ws,
                          ws_bytes, reinterpret_cast<cudaStream_t>(stream));
}

// ================================================================ EK-FAC correction

namespace {

constexpr int kEkfacStages = 3;

struct EkfacLayout {
  int ldA = 0, ldS = 0, n_chunks = 1;
  size_t at_hi = 0, at_lo = 0, st_hi = 0, st_lo = 0, part = 0;  // bf16
  size_t at = 0, st = 0, g = 0;                                 // fp32
  size_t total = 0;
};

int ekfac_check(const eogp_ekfac_desc* D, int B) {
  if (!D) return set_error(EOGP_EINVAL, "descriptor is NULL");
  if (D->d_in < 1 || D->d_out < 1 || D->T < 1 || B < 0) return set_error(EOGP_EINVAL, "bad sizes");
  if (D->dtype != EOGP_F32 && D->dtype != EOGP_BF16) return set_error(EOGP_EINVAL, "bad dtype");
  if (!D->VA || !D->VS) return set_error(EOGP_EINVAL, "VA / VS is NULL");
  if (D->dtype == EOGP_BF16) {
    if (D->d_in % 8 || D->d_out % 8) return set_error(EOGP_EUNSUPPORTED, "bf16 path needs d_in, d_out multiples of 8");
    if (!aligned16(D->VA) || !aligned16(D->VS)) return set_error(EOGP_EINVAL, "bf16 operands must be 16-byte aligned");
    if (static_cast<long long>(B) * D->T > 0x7FFFFFFFLL) return set_error(EOGP_EUNSUPPORTED, "B*T too large");
  }
  return EOGP_OK;
}

EkfacLayout ekfac_layout(const eogp_ekfac_desc* D, int B) {
  EkfacLayout o;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t at = off;
    off += al256(bytes);
    return at;
  };
  const size_t M = static_cast<size_t>(B) * D->T;
  if (D->dtype == EOGP_BF16) {
    o.ldA = round_up(D->d_in, 128);
    o.ldS = round_up(D->d_out, 128);
    o.at_hi = take(M * o.ldA * 2);
    o.at_lo = take(M * o.ldA * 2);
    o.st_hi = take(M * o.ldS * 2);
    o.st_lo = take(M * o.ldS * 2);
    const int n_tiles = (o.ldA / 128) * (o.ldS / 128);
    o.n_chunks = ekfac_chunks(std::max(1, B), n_tiles, sm_count());
    o.part = take(static_cast<size_t>(o.n_chunks) * D->d_out * D->d_in * 4);
  } else {
    o.at = take(M * D->d_in * 4);
    o.st = take(M * D->d_out * 4);
    o.g = take(static_cast<size_t>(D->d_out) * D->d_in * 4);
  }
  o.total = std::max<size_t>(off, 256);
  return o;
}

}  // namespace

extern "C" int eogp_ekfac_workspace_size(const eogp_ekfac_desc* D, int B, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  if (int rc = ekfac_check(D, B)) return rc;
  *bytes = ekfac_layout(D, B).total;
  return EOGP_OK;
}

extern "C" int eogp_ekfac_accumulate(const eogp_ekfac_desc* D, const void* a, const void* s, int B,
                                     double* sumsq, int ld, int accumulate, void* ws, size_t ws_bytes,
                                     eogp_stream_t stream) {
  clear_error();
  if (int rc = ekfac_check(D, B)) return rc;
  if (!sumsq || ld < D->d_in) return set_error(EOGP_EINVAL, "sumsq is NULL or ld < d_in");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (B == 0) {
    if (!accumulate) CUDA_TRY(cudaMemset2DAsync(sumsq, static_cast<size_t>(ld) * 8, 0,
                                                static_cast<size_t>(D->d_in) * 8, D->d_out, st));
    return EOGP_OK;
  }
  if (!a || !s) return set_error(EOGP_EINVAL, "a / s is NULL");
  const EkfacLayout lo = ekfac_layout(D, B);
  if (!ws || ws_bytes < lo.total)
    return set_error(EOGP_EWORKSPACE, "workspace of %zu bytes needed, %zu given", lo.total, ws_bytes);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  char* w = static_cast<char*>(ws);
  const int M = B * D->T;
  if (D->dtype == EOGP_BF16) {
    if (!aligned16(a) || !aligned16(s)) return set_error(EOGP_EINVAL, "a / s must be 16-byte aligned");
    {
      ProfScope ps(EOGP_K_ROTATE, st);
      CUDA_TRY(launch_tc_rotate(M, D->d_in, a, D->d_in, D->VA, D->d_in, D->d_in, w + lo.at_hi,
                                w + lo.at_lo, lo.ldA, D->T, nullptr, nullptr, sm_count(), status, st));
    }
    {
      ProfScope ps(EOGP_K_ROTATE, st);
      CUDA_TRY(launch_tc_rotate(M, D->d_out, s, D->d_out, D->VS, D->d_out, D->d_out, w + lo.st_hi,
                                w + lo.st_lo, lo.ldS, D->T, nullptr, nullptr, sm_count(), status, st));
    }
    ProfScope ps(EOGP_K_CONTRACT, st);
    CUDA_TRY(launch_tc_ekfac(w + lo.st_hi, w + lo.st_lo, lo.ldS, w + lo.at_hi, w + lo.at_lo, lo.ldA, B,
                             D->T, D->d_out, D->d_in, reinterpret_cast<float*>(w + lo.part), lo.n_chunks,
                             sumsq, ld, accumulate, kEkfacStages, sm_count(), status, st));
    return EOGP_OK;
  }
  ProfScope ps(EOGP_K_SIMT, st);
  float* at = reinterpret_cast<float*>(w + lo.at);
  float* stt = reinterpret_cast<float*>(w + lo.st);
  float* G = reinterpret_cast<float*>(w + lo.g);
  CUDA_TRY(launch_simt_gemm(M, D->d_in, D->d_in, 1.f, static_cast<const float*>(a), D->d_in, 1,
                            static_cast<const float*>(D->VA), D->d_in, 1, at, D->d_in, st));
  CUDA_TRY(launch_simt_gemm(M, D->d_out, D->d_out, 1.f, static_cast<const float*>(s), D->d_out, 1,
                            static_cast<const float*>(D->VS), D->d_out, 1, stt, D->d_out, st));
  for (int b = 0; b < B; ++b) {
    // G~_b[j][i] = sum_t S~[b T + t][j] A~[b T + t][i]
    const float* sb = stt + static_cast<size_t>(b) * D->T * D->d_out;
    const float* ab = at + static_cast<size_t>(b) * D->T * D->d_in;
    CUDA_TRY(launch_simt_gemm(D->d_out, D->d_in, D->T, 1.f, sb, 1, D->d_out, ab, 1, D->d_in, G, D->d_in, st));
    CUDA_TRY(launch_sq_accum(G, D->d_out, D->d_in, sumsq, ld, (accumulate || b > 0) ? 1 : 0, st));
  }
  return EOGP_OK;
}

// ================================================================ store records

static int payload_args_ok(const int* ks, int U, long long* W) {
  *W = 0;
  if (!ks || U < 1 || U > 1024) return set_error(EOGP_EINVAL, "need 1 <= U <= 1024 modules");
  for (int u = 0; u < U; ++u) {
    if (ks[u] < 1) return set_error(EOGP_EINVAL, "k_per_module must be >= 1");
    *W += (ks[u] + 31) / 32;
  }
  return EOGP_OK;
}

extern "C" int eogp_payload_bytes(const int* k_per_module, int U, size_t* bytes_per_example) {
  clear_error();
  long long W;
  if (!bytes_per_example) return set_error(EOGP_EINVAL, "bytes_per_example is NULL");
  if (int rc = payload_args_ok(k_per_module, U, &W)) return rc;
  *bytes_per_example = payload_row_bytes(k_per_module, U);
  return EOGP_OK;
}

extern "C" int eogp_payload_pack(const uint32_t* codes, int ld_codes, const float* scales, int ld_scales, int N,
                                 const int* k_per_module, int U, uint8_t* payload, size_t ld_payload,
                                 eogp_stream_t stream) {
  clear_error();
  long long W;
  if (int rc = payload_args_ok(k_per_module, U, &W)) return rc;
  if (N < 0) return set_error(EOGP_EINVAL, "N must be >= 0");
  if (N == 0) return EOGP_OK;
  if (!codes || !scales || !payload) return set_error(EOGP_EINVAL, "NULL argument");
  if (ld_codes < W || ld_scales < U || ld_payload < payload_row_bytes(k_per_module, U))
    return set_error(EOGP_EINVAL, "leading dimension too small");
  CUDA_TRY(launch_payload_pack(codes, ld_codes, scales, ld_scales, N, k_per_module, U, payload, ld_payload,
                               reinterpret_cast<cudaStream_t>(stream)));
  return EOGP_OK;
}

extern "C" int eogp_payload_unpack(const uint8_t* payload, size_t ld_payload, int N, const int* k_per_module,
                                   int U, uint32_t* codes, int ld_codes, float* scales, int ld_scales,
                                   eogp_stream_t stream) {
  clear_error();
  long long W;
  if (int rc = payload_args_ok(k_per_module, U, &W)) return rc;
  if (N < 0) return set_error(EOGP_EINVAL, "N must be >= 0");
  if (N == 0) return EOGP_OK;
  if (!codes || !scales || !payload) return set_error(EOGP_EINVAL, "NULL argument");
  if (ld_codes < W || ld_scales < U || ld_payload < payload_row_bytes(k_per_module, U))
    return set_error(EOGP_EINVAL, "leading dimension too small");
  CUDA_TRY(launch_payload_unpack(payload, ld_payload, N, k_per_module, U, codes, ld_codes, scales, ld_scales,
                                 reinterpret_cast<cudaStream_t>(stream)));
  return EOGP_OK;
}

// ================================================================ probes

extern "C" int eogp_set_option(int opt, int value) {
  clear_error();
  if (opt == EOGP_OPT_SCORE_OPERAND && (value == 0 || value == 1)) {
    g_opt[opt].store(value);
    return EOGP_OK;
  }
  if (opt == EOGP_OPT_TOPK_PATH && value >= 0 && value <= 2) {
    g_opt[opt].store(value);
    return EOGP_OK;
  }
  return set_error(EOGP_EINVAL, "eogp_set_option: unknown option %d or value %d", opt, value);
}

extern "C" int eogp_get_option(int opt, int* value) {
  clear_error();
  if (!value || opt < 0 || opt > 1) return set_error(EOGP_EINVAL, "eogp_get_option: bad option %d", opt);
  *value = g_opt[opt].load();
  return EOGP_OK;
}

extern "C" int eogp_measure_peaks(double* e4m3_tflops, double* e2m1_tflops, double* popc_words_per_s) {
  clear_error();
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  unsigned* sink = nullptr;
  CUDA_TRY(cudaMalloc(reinterpret_cast<void**>(&sink), sizeof(unsigned)));
  double f8 = 0.0, f4 = 0.0, pc = 0.0;
  const cudaError_t e = run_peak_probes(sm_count(), status, sink, &f8, &f4, &pc, nullptr);
  cudaFree(sink);
  if (e != cudaSuccess) return set_error(EOGP_ECUDA, "%s", cudaGetErrorString(e));
  if (int rc = eogp_sync_status(nullptr)) return rc;
  if (e4m3_tflops) *e4m3_tflops = f8;
  if (e2m1_tflops) *e2m1_tflops = f4;
  if (popc_words_per_s) *popc_words_per_s = pc;
  return EOGP_OK;
}

extern "C" int eogp_selftest_wait_timeout(long long limit_cycles) {
  clear_error();
  if (limit_cycles < 1 || limit_cycles > 1000000000LL)
    return set_error(EOGP_EINVAL, "limit_cycles must be in [1, 1e9]");
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  CUDA_TRY(run_wait_selftest(status, limit_cycles, nullptr));
  return eogp_sync_status(nullptr);
}

// ================================================================ SRHT

extern "C" int eogp_srht(const float* z, int B, int m, int ldz, const int8_t* signs, const int32_t* rows,
                         int k, float* x, int ldx, uint32_t* codes, int ld_codes, float* scales,
                         int ld_scales, eogp_stream_t stream) {
  clear_error();
  if (B < 0 || m < 1) return set_error(EOGP_EINVAL, "need B >= 0, m >= 1");
  if (m > EOGP_SRHT_MAX_M) return set_error(EOGP_EUNSUPPORTED, "SRHT needs m <= %d", EOGP_SRHT_MAX_M);
  if (k < 1 || k > srht_width(m)) return set_error(EOGP_EINVAL, "k must be in [1, p = %d]", srht_width(m));
  if (B == 0) return EOGP_OK;
  if (!z || !signs || !rows) return set_error(EOGP_EINVAL, "NULL argument");
  if (ldz < m) return set_error(EOGP_EINVAL, "ldz < m");
  if (x && ldx < k) return set_error(EOGP_EINVAL, "ldx < k");
  if (codes && (!scales || ld_codes < (k + 31) / 32 || ld_scales < 1))
    return set_error(EOGP_EINVAL, "codes need scales and ld_codes >= ceil(k/32)");
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  ProfScope ps(EOGP_K_PROJECT, st);
  CUDA_TRY(launch_srht(z, nullptr, false, ldz, B, m, signs, rows, k, x, ldx, codes, ld_codes, scales,
                       ld_scales, status, st));
  return EOGP_OK;
}

// ================================================================ fit PCA

extern "C" int eogp_fit_pca_workspace_size(int n, int m, int k, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  if (n < 1 || m < 1 || k < 1 || k > std::min(n, m)) return set_error(EOGP_EINVAL, "need 1 <= k <= min(n, m)");
  if (!fit_pca_supported(n, m, k))
    return set_error(EOGP_EUNSUPPORTED, "fit size out of range (dense solver: min(n, m) <= 12288; subspace "
                     "solver: min(n, m) <= 32768 and k + max(64, k / 4) <= 12288)");
  *bytes = fit_pca_ws_bytes(n, m, k);
  return EOGP_OK;
}

extern "C" int eogp_fit_pca(const float* Z, int n, int m, int ldz, int k, void* Pt, int ld_pt,
                            int pt_dtype, float* eig, void* ws, size_t ws_bytes, eogp_stream_t stream) {
  clear_error();
  size_t need = 0;
  if (int rc = eogp_fit_pca_workspace_size(n, m, k, &need)) return rc;
  if (!Z || !Pt || !eig) return set_error(EOGP_EINVAL, "NULL argument");
  if (ldz < m || ld_pt < m) return set_error(EOGP_EINVAL, "ldz / ld_pt must be >= m");
  if (pt_dtype != EOGP_F32 && pt_dtype != EOGP_BF16) return set_error(EOGP_EINVAL, "bad pt_dtype");
  if (!ws || ws_bytes < need) return set_error(EOGP_EWORKSPACE, "workspace of %zu bytes needed", need);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  return fit_pca_device(Z, n, m, ldz, k, Pt, ld_pt, pt_dtype, eig, ws, status_word(),
                        reinterpret_cast<cudaStream_t>(stream));
}

extern "C" int eogp_second_moment(const float* Z, int n, int m, int ldz, double* C, int ldc, int accumulate,
                                  eogp_stream_t stream) {
  clear_error();
  if (n < 0 || m < 1) return set_error(EOGP_EINVAL, "need n >= 0, m >= 1");
  if (!C || ldc < m) return set_error(EOGP_EINVAL, "C is NULL or ldc < m");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (n == 0) {
    if (!accumulate) CUDA_TRY(cudaMemset2DAsync(C, static_cast<size_t>(ldc) * 8, 0, static_cast<size_t>(m) * 8, m, st));
    return EOGP_OK;
  }
  if (!Z || ldz < m) return set_error(EOGP_EINVAL, "Z is NULL or ldz < m");
  CUDA_TRY(second_moment_device(Z, n, m, ldz, C, ldc, accumulate, st));
  return EOGP_OK;
}

extern "C" int eogp_fit_pca_from_moment_workspace_size(int m, int k, size_t* bytes) {
  return eogp_fit_pca_workspace_size(m, m, k, bytes);
}

extern "C" int eogp_fit_pca_from_moment(const double* C, int m, int ldc, int n_total, int k, void* Pt,
                                        int ld_pt, int pt_dtype, float* eig, void* ws, size_t ws_bytes,
                                        eogp_stream_t stream) {
  clear_error();
  size_t need = 0;
  if (int rc = eogp_fit_pca_workspace_size(m, m, k, &need)) return rc;
  if (n_total < 1) return set_error(EOGP_EINVAL, "n_total must be >= 1");
  if (!C || !Pt || !eig) return set_error(EOGP_EINVAL, "NULL argument");
  if (ldc < m || ld_pt < m) return set_error(EOGP_EINVAL, "ldc / ld_pt must be >= m");
  if (pt_dtype != EOGP_F32 && pt_dtype != EOGP_BF16) return set_error(EOGP_EINVAL, "bad pt_dtype");
  if (!ws || ws_bytes < need) return set_error(EOGP_EWORKSPACE, "workspace of %zu bytes needed", need);
  if (reinterpret_cast<uintptr_t>(ws) & 255) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  return fit_pca_device(nullptr, n_total, m, m, k, Pt, ld_pt, pt_dtype, eig, ws, status_word(),
                        reinterpret_cast<cudaStream_t>(stream), C, ldc);
}

// ============================================================== pack, score

extern "C" int eogp_pack_sign(const float* x, int B, int k, int ldx, uint32_t* codes, int ld_codes,
                              float* scales, int ld_scales, eogp_stream_t stream) {
  clear_error();
  if (B < 0 || k < 1) return set_error(EOGP_EINVAL, "need B >= 0, k >= 1");
  if (B == 0) return EOGP_OK;
  if (!x || !codes || !scales) return set_error(EOGP_EINVAL, "NULL argument");
  if (ldx < k || ld_codes < (k + 31) / 32 || ld_scales < 1) return set_error(EOGP_EINVAL, "leading dimension too small");
  unsigned* status = status_word();
  if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
  ProfScope ps(EOGP_K_PACK, reinterpret_cast<cudaStream_t>(stream));
  CUDA_TRY(launch_pack(x, 1, 0, ldx, B, k, nullptr, 0, codes, ld_codes, scales, ld_scales, status,
                       reinterpret_cast<cudaStream_t>(stream)));
  return EOGP_OK;
}

static bool score_args_ok(int N, const int* ks, int U, long long* W, long long* D) {
  *W = *D = 0;
  if (N < 0 || !ks || U < 1 || U > 1024) return false;
  for (int u = 0; u < U; ++u) {
    if (ks[u] < 1) return false;
    *W += (ks[u] + 31) / 32;
    *D += ks[u];
  }
  return true;
}

// Row alignment the tensor-core scoring kernels load stored code rows with.
static bool tc_rows_aligned(int mode, const void* train, int ld_train) {
  const uintptr_t a = reinterpret_cast<uintptr_t>(train);
  return mode == EOGP_SCORE_CODES ? ((ld_train % 4) == 0 && (a & 15) == 0)
                                  : ((ld_train % 2) == 0 && (a & 7) == 0);
}

extern "C" int eogp_score_workspace_size(int N, const int* k_per_module, int U, int mode, int Q,
                                         size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  (void)N;
  *bytes = 0;
  if ((mode == EOGP_SCORE_CODES || mode == EOGP_SCORE_PAPER) && k_per_module && U >= 1 &&
      U <= 1024 && score_tc_supported(mode, k_per_module, U, Q))
    *bytes = score_tc_ws_bytes(mode, k_per_module, U, Q);
  return EOGP_OK;
}

// Dense scoring into `scores`; the tensor-core kernels when the shape, the
// pointers and the workspace allow, otherwise the CUDA-core kernels.
static int score_dense(const void* train, int ld_train, const float* train_scales, int ld_tscale,
                       int N, const int* k_per_module, int U, int mode, const void* query,
                       int ld_query, const float* query_scales, int ld_qscale, int Q,
                       float* scores, int ld_scores, void* ws, size_t ws_bytes, long long W,
                       long long D, cudaStream_t st) {
  if (mode == EOGP_SCORE_CODES || mode == EOGP_SCORE_PAPER) {
    if (!train_scales) return set_error(EOGP_EINVAL, "train_scales is NULL");
    if (mode == EOGP_SCORE_CODES && !query_scales) return set_error(EOGP_EINVAL, "query_scales is NULL");
    if (ld_train < W || ld_tscale < U ||
        (mode == EOGP_SCORE_CODES ? (ld_query < W || ld_qscale < U) : ld_query < D))
      return set_error(EOGP_EINVAL, "leading dimension too small");
    // Tensor-core path when the caller provided the workspace eogp_score_workspace_size
    // asks for and the stored rows are aligned for vector loads; CODES scores are
    // bitwise identical either way.
    const bool tc = score_tc_supported(mode, k_per_module, U, Q) && ws &&
                    ws_bytes >= score_tc_ws_bytes(mode, k_per_module, U, Q) &&
                    tc_rows_aligned(mode, train, ld_train) &&
                    (reinterpret_cast<uintptr_t>(ws) & 255) == 0;
    if (tc) {
      unsigned* status = status_word();
      if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
      CUDA_TRY(launch_score_tc(mode, static_cast<const uint32_t*>(train), ld_train, train_scales,
                               ld_tscale, N, k_per_module, U, query, ld_query, query_scales,
                               ld_qscale, Q, scores, ld_scores, nullptr, ws, sm_count(), status, st));
    } else if (mode == EOGP_SCORE_CODES) {
      CUDA_TRY(launch_score_codes(static_cast<const uint32_t*>(train), ld_train, train_scales,
                                  ld_tscale, N, k_per_module, U, static_cast<const uint32_t*>(query),
                                  ld_query, query_scales, ld_qscale, Q, scores, ld_scores, st));
    } else {
      CUDA_TRY(launch_score_paper(static_cast<const uint32_t*>(train), ld_train, train_scales, ld_tscale,
                                  N, k_per_module, U, static_cast<const float*>(query), ld_query, Q,
                                  scores, ld_scores, st));
    }
  } else if (mode == EOGP_SCORE_FP) {
    if (ld_train < D || ld_query < D) return set_error(EOGP_EINVAL, "leading dimension too small");
    CUDA_TRY(launch_simt_gemm(Q, N, static_cast<int>(D), 1.f, static_cast<const float*>(query), ld_query,
                              1, static_cast<const float*>(train), ld_train, 1, scores, ld_scores, st));
  } else {
    return set_error(EOGP_EINVAL, "bad score mode");
  }
  return EOGP_OK;
}

extern "C" int eogp_score(const void* train, int ld_train, const float* train_scales, int ld_tscale,
                          int N, const int* k_per_module, int U, int mode, const void* query,
                          int ld_query, const float* query_scales, int ld_qscale, int Q,
                          float* scores, int ld_scores, void* ws, size_t ws_bytes,
                          eogp_stream_t stream) {
  clear_error();
  if (N < 0 || Q < 0) return set_error(EOGP_EINVAL, "N, Q must be >= 0");
  long long W, D;
  if (!score_args_ok(N, k_per_module, U, &W, &D))
    return set_error(EOGP_EINVAL, "need 1 <= U <= 1024 modules with k_per_module >= 1");
  if (mode != EOGP_SCORE_CODES && mode != EOGP_SCORE_PAPER && mode != EOGP_SCORE_FP)
    return set_error(EOGP_EINVAL, "bad score mode");
  if (N == 0 || Q == 0) return EOGP_OK;
  if (!train || !query || !scores) return set_error(EOGP_EINVAL, "NULL argument");
  if (ld_scores < N) return set_error(EOGP_EINVAL, "ld_scores < N");
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  ProfScope ps(EOGP_K_SCORE, st);
  return score_dense(train, ld_train, train_scales, ld_tscale, N, k_per_module, U, mode, query,
                     ld_query, query_scales, ld_qscale, Q, scores, ld_scores, ws, ws_bytes, W, D, st);
}

// ---------------------------------------------------------------- top-K
// Workspace plan of eogp_score_topk: fused (tensor-core scoring with the ranking in
// its epilogue) or dense (scores into the workspace, then a ranking kernel).
struct TopkPlan {
  bool fused, select;
  int slots;
  size_t q_bytes, dense_bytes, list_bytes, buf_bytes, scr_bytes, total;
};

// Paths: up to topk_select_max_n() stored rows, dense scores (tensor cores
// where they apply) and a radix select per query row (k_topk_select); beyond,
// the ranking is fused into the tensor-core scoring kernel when it supports the
// request (the Q x N matrix then never reaches HBM), else dense scores, per-slot
// lists and a merge. Measured on the GPT-2 query workload (N = 16384, Q = 1024,
// top 20): fused 2.4 ms, dense + per-slot lists 2.9 ms. EOGP_OPT_TOPK_PATH = 1 / 2
// forces the fused / a dense path.
static int topk_fused_override() {
  const int v = option(EOGP_OPT_TOPK_PATH);
  return v == 1 ? 1 : v == 2 ? 0 : -1;
}

static TopkPlan topk_plan(int N, const int* ks, int U, int mode, int Q, int K) {
  TopkPlan p{};
  const bool tc_ok = (mode == EOGP_SCORE_CODES || mode == EOGP_SCORE_PAPER) &&
                     score_tc_supported(mode, ks, U, Q);
  const int force = topk_fused_override();
  p.fused = tc_ok && score_tc_topk_fits(mode, ks, U, Q, K) && force != 0 &&
            (force == 1 || N > topk_select_max_n());
  p.select = !p.fused && N <= topk_select_max_n();
  p.q_bytes = tc_ok ? score_tc_ws_bytes(mode, ks, U, Q) : 0;
  if (p.fused) {
    p.slots = score_tc_grid(mode, ks, U, N, Q, K, sm_count());
    p.dense_bytes = 0;
  } else {
    p.slots = p.select ? 0 : topk_dense_slots(N);
    p.dense_bytes = al256(static_cast<size_t>(Q) * ((static_cast<size_t>(N) + 3) & ~size_t(3)) * 4);
  }
  p.list_bytes = al256(static_cast<size_t>(p.slots) * Q * K * 4);
  p.buf_bytes = p.fused ? al256(score_tc_list_buf_bytes(mode, ks, U, Q, K, p.slots)) : 0;
  p.scr_bytes = p.fused ? al256(score_tc_scratch_bytes(mode, ks, U, Q, K, p.slots)) : 0;
  p.total = al256(p.q_bytes) + p.dense_bytes + 2 * p.list_bytes + 2 * p.buf_bytes +
            (p.fused ? al256(static_cast<size_t>(Q) * 4) : 0) + p.scr_bytes;
  return p;
}

extern "C" int eogp_score_topk_workspace_size(int N, const int* k_per_module, int U, int mode, int Q,
                                              int topk, size_t* bytes) {
  clear_error();
  if (!bytes) return set_error(EOGP_EINVAL, "bytes is NULL");
  long long W, D;
  if (!score_args_ok(N, k_per_module, U, &W, &D) || Q < 0)
    return set_error(EOGP_EINVAL, "need N, Q >= 0 and 1 <= U <= 1024 modules with k_per_module >= 1");
  if (topk < 1 || topk > EOGP_TOPK_MAX) return set_error(EOGP_EINVAL, "topk must be in [1, %d]", EOGP_TOPK_MAX);
  *bytes = Q == 0 ? 0 : topk_plan(N, k_per_module, U, mode, Q, topk).total;
  return EOGP_OK;
}

extern "C" int eogp_score_topk(const void* train, int ld_train, const float* train_scales,
                               int ld_tscale, int N, const int* k_per_module, int U, int mode,
                               const void* query, int ld_query, const float* query_scales,
                               int ld_qscale, int Q, int topk, float* top_scores, int ld_top_scores,
                               int* top_index, int ld_top_index, void* ws, size_t ws_bytes,
                               eogp_stream_t stream) {
  clear_error();
  if (N < 0 || Q < 0) return set_error(EOGP_EINVAL, "N, Q must be >= 0");
  long long W, D;
  if (!score_args_ok(N, k_per_module, U, &W, &D))
    return set_error(EOGP_EINVAL, "need 1 <= U <= 1024 modules with k_per_module >= 1");
  if (mode != EOGP_SCORE_CODES && mode != EOGP_SCORE_PAPER && mode != EOGP_SCORE_FP)
    return set_error(EOGP_EINVAL, "bad score mode");
  if (topk < 1 || topk > EOGP_TOPK_MAX) return set_error(EOGP_EINVAL, "topk must be in [1, %d]", EOGP_TOPK_MAX);
  if (Q == 0) return EOGP_OK;
  if (!top_scores || !top_index) return set_error(EOGP_EINVAL, "NULL output");
  if (ld_top_scores < topk || ld_top_index < topk) return set_error(EOGP_EINVAL, "output leading dimension < topk");
  if (N > 0 && (!train || !query)) return set_error(EOGP_EINVAL, "NULL argument");
  const TopkPlan p = topk_plan(N, k_per_module, U, mode, Q, topk);
  if (!ws || ws_bytes < p.total) return set_error(EOGP_EWORKSPACE, "workspace too small: need %zu bytes", p.total);
  if ((reinterpret_cast<uintptr_t>(ws) & 255) != 0) return set_error(EOGP_EINVAL, "workspace must be 256-byte aligned");
  uint8_t* w = static_cast<uint8_t*>(ws);
  void* qws = w;
  float* dense = reinterpret_cast<float*>(w + al256(p.q_bytes));
  float* lst = reinterpret_cast<float*>(w + al256(p.q_bytes) + p.dense_bytes);
  int* lsi = reinterpret_cast<int*>(w + al256(p.q_bytes) + p.dense_bytes + p.list_bytes);
  float* bufs = reinterpret_cast<float*>(w + al256(p.q_bytes) + p.dense_bytes + 2 * p.list_bytes);
  int* bufi = reinterpret_cast<int*>(w + al256(p.q_bytes) + p.dense_bytes + 2 * p.list_bytes + p.buf_bytes);
  unsigned* gtau = reinterpret_cast<unsigned*>(w + al256(p.q_bytes) + p.dense_bytes + 2 * p.list_bytes +
                                               2 * p.buf_bytes);
  float* scr = reinterpret_cast<float*>(w + al256(p.q_bytes) + p.dense_bytes + 2 * p.list_bytes +
                                        2 * p.buf_bytes + al256(static_cast<size_t>(Q) * 4));
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  ProfScope ps(EOGP_K_SCORE, st);
  if (p.fused && N > 0) {
    if (!train_scales || (mode == EOGP_SCORE_CODES && !query_scales))
      return set_error(EOGP_EINVAL, "scales are NULL");
    if (ld_train < W || ld_tscale < U ||
        (mode == EOGP_SCORE_CODES ? (ld_query < W || ld_qscale < U) : ld_query < D))
      return set_error(EOGP_EINVAL, "leading dimension too small");
    if (!tc_rows_aligned(mode, train, ld_train))
      return set_error(EOGP_EUNSUPPORTED, mode == EOGP_SCORE_CODES
                                              ? "fused top-K needs 16-byte aligned code rows (ld_train % 4 == 0)"
                                              : "fused top-K needs 8-byte aligned code rows (ld_train % 2 == 0)");
    unsigned* status = status_word();
    if (!status) return set_error(EOGP_ECUDA, "device status word unavailable");
    TcTopK tk{topk, lst, lsi, bufs, bufi, gtau, scr, top_scores, ld_top_scores, top_index, ld_top_index};
    CUDA_TRY(launch_score_tc(mode, static_cast<const uint32_t*>(train), ld_train, train_scales, ld_tscale,
                             N, k_per_module, U, query, ld_query, query_scales, ld_qscale, Q, nullptr,
                             0, &tk, qws, sm_count(), status, st));
    return EOGP_OK;
  }
  const int ldd = (N + 3) & ~3;
  if (N > 0) {
    const int rc = score_dense(train, ld_train, train_scales, ld_tscale, N, k_per_module, U, mode, query,
                               ld_query, query_scales, ld_qscale, Q, dense, ldd, qws, p.q_bytes, W, D, st);
    if (rc != EOGP_OK) return rc;
  }
  if (p.select) {
    CUDA_TRY(launch_topk_select(dense, ldd, Q, N, topk, top_scores, ld_top_scores, top_index, ld_top_index, st));
    return EOGP_OK;
  }
  CUDA_TRY(launch_topk_dense(dense, ldd, Q, N, topk, lst, lsi, st));
  CUDA_TRY(launch_topk_merge(lst, lsi, topk_dense_slots(N), Q, topk, top_scores, ld_top_scores, top_index,
                             ld_top_index, st));
  return EOGP_OK;
}
