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

// Launch epoch of a work area (RunWords), read by one thread when the CTA
// starts.  The launch's CTAs all read the same value: it only advances once
// every one of them has passed run_exit.
__device__ __forceinline__ uint32_t run_epoch(const RunWords* run) {
    return *reinterpret_cast<const volatile uint32_t*>(&run->epoch);
}

// Called by one thread of every CTA after the CTA's last access to the work
// area's counters: the last CTA of the launch to get here advances the
// epoch for the next launch of the same work list.
__device__ __forceinline__ void run_exit(RunWords* run, uint32_t epoch) {
    __threadfence();
    if (atomicAdd(&run->exits, 1u) == gridDim.x - 1u) {
        run->exits = 0u;
        __threadfence();
        *reinterpret_cast<volatile uint32_t*>(&run->epoch) = epoch + 1u;
    }
}

// Counts one arrival on a merge counter during launch epoch `epoch` and
// returns the count including it.  The counter holds (epoch << 32 | count);
// a value left by another epoch counts as zero.  The loop only retries while
// another chunk of the same group updates the counter.
__device__ __forceinline__ uint32_t count_arrival(unsigned long long* ctr, uint32_t epoch) {
    unsigned long long old = *reinterpret_cast<volatile unsigned long long*>(ctr);
    for (;;) {
        const uint32_t have = static_cast<uint32_t>(old >> 32) == epoch ? static_cast<uint32_t>(old) : 0u;
        const unsigned long long want = (static_cast<unsigned long long>(epoch) << 32) | (have + 1u);
        const unsigned long long prev = atomicCAS(ctr, old, want);
        if (prev == old) return have + 1u;
        old = prev;
    }
}

using EncodeTiledFn =CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
// cuTensorMapEncodeTiled from the driver (looked up once), or nullptr.
EncodeTiledFn encode_fn();
// [rows, heads, d] bf16 tensor, box of (64 channels, box_heads, box_rows),
// 128-byte swizzle; out-of-range rows read as zero.
bool encode_3d(EncodeTiledFn fn, CUtensorMap* map, const void* base, uint64_t d, uint64_t heads, uint64_t rows,
               uint32_t box_heads, uint32_t box_rows);

}  // namespace opattn
