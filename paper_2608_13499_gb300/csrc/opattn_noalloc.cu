// opattn_noalloc.cu -- fixed device scratch for opattn_prefill_noalloc.
//
// Some callers cannot let a library call cudaMalloc / cudaMallocAsync: a
// serving engine that reserves nearly all of HBM for its KV cache up front
// and routes every allocation through its own pool, a process whose device
// memory is capped by a quota the caller enforces, or a device where the
// stream-ordered allocator is unavailable.  For them the work list and the
// status word live in this file-scope device array instead of per-call
// scratch.  Every GPU that loads the library holds the array until the
// process exits.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "opattn_internal.h"

namespace opattn {
namespace {

// Room for kNoAllocMaxUnits 32-byte work units, kNoAllocMaxCtas + 1 CTA
// offsets and the status word.
constexpr size_t kNoAllocScratchBytes = kNoAllocMaxUnits * sizeof(UnitRec) + 8192;
static_assert((kNoAllocMaxCtas + 1) * sizeof(int32_t) + 64 <= 8192, "CTA offsets must fit the reserve");

constexpr int kMaxDevices = 64;

}  // namespace
}  // namespace opattn

// In host code this name is only a stand-in for the array; its device
// address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) uint8_t g_opattn_noalloc_scratch[opattn::kNoAllocScratchBytes];

namespace opattn {

// Device address and size of the scratch array on the current device.  The
// first call on a device looks the address up (with that device current)
// and caches it; later calls only read the cache.
int noalloc_scratch(void** ptr, size_t* bytes) {
    static std::mutex mu;
    static void* addr[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return static_cast<int>(e);
    if (dev < 0 || dev >= kMaxDevices) return static_cast<int>(cudaErrorInvalidDevice);
    std::lock_guard<std::mutex> lk(mu);
    if (!addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_opattn_noalloc_scratch);
        if (e != cudaSuccess) return static_cast<int>(e);
        addr[dev] = p;
    }
    *ptr = addr[dev];
    *bytes = kNoAllocScratchBytes;
    return 0;
}

}  // namespace opattn
