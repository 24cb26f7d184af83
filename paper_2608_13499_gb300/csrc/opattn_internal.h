// opattn_internal.h -- types shared by the host runtime (opattn_api.cpp) and
// the kernel translation unit (opattn_kernel.cu).  Not part of the public ABI.
#pragma once
#include <cstdint>

#include <cuda_runtime.h>

namespace opattn {

// Tile geometry.  An M-tile is 128 accumulator rows: TPB query tokens x G
// query heads of one kv head (rows ordered token-major, head-minor, which is
// their order in memory).  A work unit is two M-tiles (2 * TPB tokens) of one
// sequence and one kv head; each K/V tile of BN keys feeds both M-tiles and
// all G heads of the group.
constexpr int kRowsPerTile = 128;
constexpr int kBlockN = 128;

inline int tokens_per_tile(int G) { return kRowsPerTile / G; }
inline int tokens_per_unit(int G) { return 2 * tokens_per_tile(G); }

// One work unit; 32 bytes, read by every role of the CTA that owns it.
struct UnitRec {
    int32_t q_tok0;   // packed query row of the unit's first token
    int32_t n_tok;    // valid tokens in the unit (<= 2 * TPB)
    int32_t k_row0;   // packed key row of the sequence's first key
    int32_t Lk;       // keys in the sequence
    int32_t qlim0;    // last visible key index of the first token (= position + Lk - Lq)
    int32_t kvh;      // kv head
    int32_t n_tiles;  // key tiles to visit (0: no row sees a key)
    int32_t seq;      // sequence index (diagnostics only)
};
static_assert(sizeof(UnitRec) == 32, "UnitRec must stay 32 bytes");

// Device status word values (written by the kernel's bounded waits).
constexpr int32_t kDevOk = 0;
constexpr int32_t kDevTimeout = 1;

// Test-only launch flag: the MMA warp waits on a barrier nothing arrives on,
// so the bounded-wait path runs (short limit, error status, clean exit).
constexpr uint32_t kFlagForceTimeout = 1u;

struct LaunchArgs {
    const void* q;
    const void* k;
    const void* v;
    void* o;
    float* lse;
    int64_t total_q;
    int64_t total_k;
    int32_t Hq, Hkv, d;
    float scale;
    const UnitRec* units;     // device
    const int32_t* cta_off;   // device, n_cta + 1
    int32_t n_cta;
    int32_t* status;          // device
    uint32_t flags;
};

// Limits of the allocation-free entry point (opattn_prefill_noalloc), whose
// work list lives in a fixed device array (opattn_noalloc.cu).
constexpr int64_t kNoAllocMaxUnits = 32768;
constexpr int32_t kNoAllocMaxCtas = 1024;
// Implemented in opattn_noalloc.cu: device address and size of that array on
// the current device (looked up on the first call per device).  Returns a
// cudaError_t as int.
int noalloc_scratch(void** ptr, size_t* bytes);

// Implemented in opattn_kernel.cu.  Returns a cudaError_t (as int) or a
// negative value when the tensor maps cannot be encoded.
int launch_prefill(const LaunchArgs& a, cudaStream_t stream);
// Shared memory bytes the kernel needs for head dim d (0 if unsupported).
int kernel_smem_bytes(int d);

}  // namespace opattn
