// Page-locked host staging memory backed by transparent huge pages.
//
// Host-to-device copies of the compression inputs (a, s) from page-locked
// memory run at the link's full rate only when the pinned pages map onto few
// large translations: on the GB300 systems this library was measured on,
// cudaHostAlloc'd buffers fed cudaMemcpyAsync at anywhere from ~80 to ~210 GB/s
// from one allocation to the next, while anonymous memory advised for huge
// pages and then registered with cudaHostRegister ran at ~211 GB/s every time.
// eogp_host_alloc maps such a region (aligned to the huge-page size, so the
// kernel can back all of it with huge pages), advises it, registers it, and
// records it so that eogp_host_free can undo both steps from the pointer alone.
#include <sys/mman.h>
#include <unistd.h>

#include <cstdio>
#include <cstring>
#include <cstdint>
#include <mutex>
#include <unordered_map>

#include "eogp_internal.h"

using namespace eogp;

namespace {

struct Region {
  void* base;       // start of the mapping
  size_t map_len;   // length of the mapping
  size_t user_len;  // bytes registered and handed out
};

std::mutex g_mu;
std::unordered_map<uintptr_t, Region>& regions() {
  static std::unordered_map<uintptr_t, Region> r;
  return r;
}

// Huge-page size the kernel uses for anonymous memory (2 MB on 4 KB-page
// systems, 512 MB on 64 KB-page arm64), 2 MB if it cannot be read.
size_t huge_page_bytes() {
  size_t v = 0;
  if (FILE* f = std::fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
    unsigned long long x = 0;
    if (std::fscanf(f, "%llu", &x) == 1) v = static_cast<size_t>(x);
    std::fclose(f);
  }
  return v >= 4096 && (v & (v - 1)) == 0 ? v : (size_t(2) << 20);
}

}  // namespace

extern "C" int eogp_host_alloc(size_t bytes, void** ptr) {
  clear_error();
  if (!ptr) return set_error(EOGP_EINVAL, "ptr is NULL");
  *ptr = nullptr;
  if (bytes == 0) return set_error(EOGP_EINVAL, "bytes must be > 0");
  // Requests of at least one huge page are aligned to and advised for huge
  // pages; smaller ones are rounded to the base page only (on 64 KB-page arm64
  // hosts a huge page is 512 MB, far too much to pin for a small buffer).
  const size_t huge = huge_page_bytes();
  const long ps = sysconf(_SC_PAGESIZE);
  const size_t hp = bytes >= huge ? huge : static_cast<size_t>(ps > 0 ? ps : 4096);
  const size_t len = (bytes + hp - 1) / hp * hp;
  if (len < bytes || len + hp < len) return set_error(EOGP_EINVAL, "size too large");
  // Map one alignment unit more than needed and keep the aligned part.
  void* raw = mmap(nullptr, len + hp, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == MAP_FAILED) return set_error(EOGP_EINVAL, "mmap of %zu bytes failed", len + hp);
  const uintptr_t r = reinterpret_cast<uintptr_t>(raw);
  const uintptr_t a = (r + hp - 1) / hp * hp;
  if (a > r) munmap(raw, a - r);
  const size_t tail = (r + len + hp) - (a + len);
  if (tail) munmap(reinterpret_cast<void*>(a + len), tail);
  void* p = reinterpret_cast<void*>(a);
  if (hp == huge) madvise(p, len, MADV_HUGEPAGE);  // advice only: without it the region still works
  // Fault the region in from the CPU before registering it, so that the pages
  // are placed by ordinary first-touch faults on the advised, aligned range:
  // the configuration the ~211 GB/s copy rate above was measured with.
  std::memset(p, 0, len);
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterDefault);
  if (e != cudaSuccess) {
    munmap(p, len);
    return set_error(EOGP_ECUDA, "cudaHostRegister of %zu bytes failed: %s", len, cudaGetErrorString(e));
  }
  {
    std::lock_guard<std::mutex> g(g_mu);
    regions()[a] = Region{p, len, bytes};
  }
  *ptr = p;
  return EOGP_OK;
}

extern "C" int eogp_host_free(void* ptr) {
  clear_error();
  if (!ptr) return EOGP_OK;
  Region reg;
  {
    std::lock_guard<std::mutex> g(g_mu);
    auto it = regions().find(reinterpret_cast<uintptr_t>(ptr));
    if (it == regions().end()) return set_error(EOGP_EINVAL, "pointer was not returned by eogp_host_alloc");
    reg = it->second;
    regions().erase(it);
  }
  const cudaError_t e = cudaHostUnregister(reg.base);
  munmap(reg.base, reg.map_len);
  if (e != cudaSuccess) return set_error(EOGP_ECUDA, "cudaHostUnregister failed: %s", cudaGetErrorString(e));
  return EOGP_OK;
}
