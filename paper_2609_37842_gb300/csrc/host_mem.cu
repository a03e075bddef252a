// Page-locked host staging memory backed by transparent huge pages.
//
// Host-to-device copies of the compression inputs (a, s) from page-locked
// memory run at the link's full rate only when the pinned pages map onto few
// large translations: on the GB300 systems this library was measured on,
// cudaHostAlloc'd buffers fed cudaMemcpyAsync at anywhere from ~80 to ~210 GB/s
// from one allocation to the next, anonymous memory advised for huge pages and
// then registered with cudaHostRegister ran at ~211 GB/s every time, and the
// same memory on 64 KB base pages (no huge-page advice) at ~51 GB/s.
//
// Three size classes:
//  * at least half a huge page: a region of its own, aligned to and advised for
//    huge pages, registered, recorded so that eogp_host_free can undo both
//    steps from the pointer alone;
//  * from kArenaMin up to half a huge page: a block carved out of a shared
//    arena of one huge page (the same kind of region), first fit over the
//    arena's free list, coalesced on free; an arena is released when its last
//    block is freed. Buffers of tens to hundreds of MB thus sit on huge pages
//    without each pinning a whole one (512 MB on 64 KB-page arm64 hosts);
//  * below kArenaMin: base pages only (no huge-page advice), rounded to whole
//    base pages.
#include <sys/mman.h>
#include <unistd.h>

#include <cstdio>
#include <cstring>
#include <cstdint>
#include <map>
#include <memory>
#include <mutex>
#include <unordered_map>
#include <vector>

#include "eogp_internal.h"

using namespace eogp;

namespace {

constexpr size_t kArenaMin = size_t(1) << 20;  // smaller requests stay on base pages
constexpr size_t kBlockAlign = 4096;           // arena blocks start on 4 KB boundaries

struct Region {
  void* base;       // start of the mapping (aligned)
  size_t map_len;   // length of the mapping and of the registration
};

struct Arena {
  Region reg;
  std::map<size_t, size_t> free;  // offset -> length of each free run
  size_t used = 0;                // bytes handed out
};

struct Block {
  Arena* arena;
  size_t off, len;
};

std::mutex g_mu;
std::unordered_map<uintptr_t, Region>& regions() {
  static std::unordered_map<uintptr_t, Region> r;
  return r;
}
std::unordered_map<uintptr_t, Block>& blocks() {
  static std::unordered_map<uintptr_t, Block> b;
  return b;
}
std::vector<std::unique_ptr<Arena>>& arenas() {
  static std::vector<std::unique_ptr<Arena>> a;
  return a;
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

// Maps, aligns, (for huge pages) advises, faults in and registers `len` bytes
// aligned to `unit` (len a multiple of unit). Returns an error code.
int map_region(size_t len, size_t unit, bool advise_huge, Region* out) {
  // Map one alignment unit more than needed and keep the aligned part.
  void* raw = mmap(nullptr, len + unit, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == MAP_FAILED) return set_error(EOGP_EINVAL, "mmap of %zu bytes failed", len + unit);
  const uintptr_t r = reinterpret_cast<uintptr_t>(raw);
  const uintptr_t a = (r + unit - 1) / unit * unit;
  if (a > r) munmap(raw, a - r);
  const size_t tail = (r + len + unit) - (a + len);
  if (tail) munmap(reinterpret_cast<void*>(a + len), tail);
  void* p = reinterpret_cast<void*>(a);
  if (advise_huge) madvise(p, len, MADV_HUGEPAGE);  // advice only: without it the region still works
  // Fault the region in from the CPU before registering it, so that the pages
  // are placed by ordinary first-touch faults on the advised, aligned range:
  // the configuration the ~211 GB/s copy rate above was measured with.
  std::memset(p, 0, len);
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterDefault);
  if (e != cudaSuccess) {
    munmap(p, len);
    return set_error(EOGP_ECUDA, "cudaHostRegister of %zu bytes failed: %s", len, cudaGetErrorString(e));
  }
  *out = Region{p, len};
  return EOGP_OK;
}

cudaError_t unmap_region(const Region& reg) {
  const cudaError_t e = cudaHostUnregister(reg.base);
  munmap(reg.base, reg.map_len);
  return e;
}

// First fit of `len` bytes in an arena's free list; the arena's offset or SIZE_MAX.
size_t arena_take(Arena* ar, size_t len) {
  for (auto it = ar->free.begin(); it != ar->free.end(); ++it) {
    if (it->second < len) continue;
    const size_t off = it->first, rest = it->second - len;
    ar->free.erase(it);
    if (rest) ar->free.emplace(off + len, rest);
    ar->used += len;
    return off;
  }
  return SIZE_MAX;
}

// Returns a block to its arena's free list, merging it with free neighbours.
void arena_give(Arena* ar, size_t off, size_t len) {
  ar->used -= len;
  auto next = ar->free.lower_bound(off);
  if (next != ar->free.end() && off + len == next->first) {
    len += next->second;
    next = ar->free.erase(next);
  }
  if (next != ar->free.begin()) {
    auto prev = std::prev(next);
    if (prev->first + prev->second == off) {
      prev->second += len;
      return;
    }
  }
  ar->free.emplace(off, len);
}

}  // namespace

extern "C" int eogp_host_alloc(size_t bytes, void** ptr) {
  clear_error();
  if (!ptr) return set_error(EOGP_EINVAL, "ptr is NULL");
  *ptr = nullptr;
  if (bytes == 0) return set_error(EOGP_EINVAL, "bytes must be > 0");
  const size_t huge = huge_page_bytes();
  const long ps = sysconf(_SC_PAGESIZE);
  const size_t base = static_cast<size_t>(ps > 0 ? ps : 4096);
  if (bytes >= kArenaMin && bytes < huge / 2) {
    // A block of a shared huge-page arena.
    const size_t len = (bytes + kBlockAlign - 1) / kBlockAlign * kBlockAlign;
    std::lock_guard<std::mutex> g(g_mu);
    Arena* ar = nullptr;
    size_t off = SIZE_MAX;
    for (auto& a : arenas()) {
      off = arena_take(a.get(), len);
      if (off != SIZE_MAX) {
        ar = a.get();
        break;
      }
    }
    if (!ar) {
      auto fresh = std::make_unique<Arena>();
      if (int rc = map_region(huge, huge, true, &fresh->reg)) return rc;
      fresh->free.emplace(0, huge);
      ar = fresh.get();
      arenas().push_back(std::move(fresh));
      off = arena_take(ar, len);
    }
    char* p = static_cast<char*>(ar->reg.base) + off;
    std::memset(p, 0, len);  // a reused block holds its previous owner's bytes
    blocks()[reinterpret_cast<uintptr_t>(p)] = Block{ar, off, len};
    *ptr = p;
    return EOGP_OK;
  }
  // A region of its own: whole huge pages from half a huge page up, else whole
  // base pages without huge-page advice.
  const size_t unit = bytes >= kArenaMin ? huge : base;
  const size_t len = (bytes + unit - 1) / unit * unit;
  if (len < bytes || len + unit < len) return set_error(EOGP_EINVAL, "size too large");
  Region reg;
  if (int rc = map_region(len, unit, unit == huge, &reg)) return rc;
  {
    std::lock_guard<std::mutex> g(g_mu);
    regions()[reinterpret_cast<uintptr_t>(reg.base)] = reg;
  }
  *ptr = reg.base;
  return EOGP_OK;
}

extern "C" int eogp_host_free(void* ptr) {
  clear_error();
  if (!ptr) return EOGP_OK;
  Region reg{nullptr, 0};
  {
    std::lock_guard<std::mutex> g(g_mu);
    const uintptr_t key = reinterpret_cast<uintptr_t>(ptr);
    auto bt = blocks().find(key);
    if (bt != blocks().end()) {
      Arena* ar = bt->second.arena;
      arena_give(ar, bt->second.off, bt->second.len);
      blocks().erase(bt);
      if (ar->used) return EOGP_OK;
      // last block of the arena: release the arena
      reg = ar->reg;
      auto& v = arenas();
      for (auto it = v.begin(); it != v.end(); ++it)
        if (it->get() == ar) {
          v.erase(it);
          break;
        }
    } else {
      auto it = regions().find(key);
      if (it == regions().end()) return set_error(EOGP_EINVAL, "pointer was not returned by eogp_host_alloc");
      reg = it->second;
      regions().erase(it);
    }
  }
  const cudaError_t e = unmap_region(reg);
  if (e != cudaSuccess) return set_error(EOGP_ECUDA, "cudaHostUnregister failed: %s", cudaGetErrorString(e));
  return EOGP_OK;
}
