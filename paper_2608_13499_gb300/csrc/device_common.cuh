// device_common.cuh -- pieces shared by the prefill and decode kernels:
// bounded mbarrier waits (every wait gives up after a time limit, raises the
// CTA's abort flag and records a timeout in the status word) and the host
// helpers that encode TMA tensor maps.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "opattn_internal.h"
#include "ptx.cuh"

namespace opattn {

constexpr uint64_t kWaitLimitNs = 2000000000ull;  // 2 s: no legitimate wait comes close
constexpr uint64_t kForcedLimitNs = 20000000ull;  // 20 ms: the forced-timeout test
constexpr uint64_t kDrainLimitNs = 200000000ull;  // in-flight copies / MMAs after an abort

// Wait for the phase of parity `parity` of `bar`.  Gives up when another
// thread of the CTA has aborted, or after `limit_ns`, in which case it
// raises the CTA abort flag and records a timeout in the status word.
__device__ __forceinline__ bool bounded_wait(uint32_t bar, uint32_t parity, volatile int32_t* abort_flag,
                                             int32_t* status, uint64_t limit_ns) {
    if (ptx::mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer_ns();
    for (;;) {
        if (ptx::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (ptx::globaltimer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            atomicCAS(status, kDevOk, kDevTimeout);
            return false;
        }
    }
}

// Wait used while shutting down after an abort: ignores the abort flag and
// returns silently after `limit_ns`.
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, uint64_t limit_ns) {
    const uint64_t t0 = ptx::globaltimer_ns();
    while (!ptx::mbar_try_wait(bar, parity)) {
        if (ptx::globaltimer_ns() - t0 > limit_ns) return;
    }
}

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
// cuTensorMapEncodeTiled from the driver (looked up once), or nullptr.
EncodeTiledFn encode_fn();
// [rows, heads, d] bf16 tensor, box of (64 channels, box_heads, box_rows),
// 128-byte swizzle; out-of-range rows read as zero.
bool encode_3d(EncodeTiledFn fn, CUtensorMap* map, const void* base, uint64_t d, uint64_t heads, uint64_t rows,
               uint32_t box_heads, uint32_t box_rows);

}  // namespace opattn
