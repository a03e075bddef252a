// Compression with built-in scratch memory.
//
// eogp_compress_layer needs a caller-provided workspace. Some callers cannot
// allocate one: a plugin inside a host framework that owns every device
// allocation and forbids direct cudaMalloc, a service that reserves a fixed
// memory budget at start-up and may not grow it later, or a plain C program
// that links only this library and has no allocator to hand. For them,
// eogp_compress_layer_static runs the same kernels on a scratch array that is
// part of the library image: a file-scope device array of
// EOGP_STATIC_WORKSPACE_BYTES, which every GPU that loads the library holds
// until the process exits. The entry point itself calls no cudaMalloc,
// cudaFree or other allocating routine.
#include "eogp_dev.cuh"
#include "eogp_internal.h"

static __device__ __align__(256) unsigned char g_eogp_static_ws[EOGP_STATIC_WORKSPACE_BYTES];

namespace {

// Device address of the scratch array on the current device. In host code the
// array's name is only a host-side stand-in, so the address is looked up with
// the device current, on every call: the lookup allocates nothing, and an
// address kept from an earlier call would be stale if the device's context had
// been destroyed and created again since.
int static_scratch(void** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_eogp_static_ws);
  if (e != cudaSuccess || !p)
    return eogp::set_error(EOGP_ECUDA, "cudaGetSymbolAddress of the built-in scratch failed: %s",
                           cudaGetErrorString(e));
  *out = p;
  return EOGP_OK;
}

}  // namespace

extern "C" int eogp_compress_layer_static(const eogp_layer_desc* L, const void* a, const void* s,
                                          int B, int out_mode, float* out, int ld_out,
                                          uint32_t* codes, int ld_codes, float* scales,
                                          int ld_scales, eogp_stream_t stream) {
  eogp::clear_error();
  size_t need = 0;
  int rc = eogp_compress_workspace_size(L, B, out_mode, &need);
  if (rc != EOGP_OK) return rc;
  if (need > static_cast<size_t>(EOGP_STATIC_WORKSPACE_BYTES))
    return eogp::set_error(EOGP_EUNSUPPORTED,
                           "this batch needs %zu bytes of scratch but the built-in scratch holds "
                           "%zu; use a smaller batch or eogp_compress_layer with a workspace",
                           need, static_cast<size_t>(EOGP_STATIC_WORKSPACE_BYTES));
  void* ws = nullptr;
  rc = static_scratch(&ws);
  if (rc != EOGP_OK) return rc;
  // Nothing in the scratch has to start at zero: every byte the kernels read is
  // written earlier in the same call.
  return eogp_compress_layer(L, a, s, B, out_mode, out, ld_out, codes, ld_codes, scales, ld_scales,
                             ws, static_cast<size_t>(EOGP_STATIC_WORKSPACE_BYTES), stream);
}
