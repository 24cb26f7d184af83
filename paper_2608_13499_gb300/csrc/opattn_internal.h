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
// all G heads of the group.  A unit normally visits every key tile its
// tokens see; a unit over a long key range may instead be cut into pieces
// (split-KV) that each cover a stretch of its key tiles on its own CTA and
// are merged with their log-sum-exp weights by the piece that finishes last.
constexpr int kRowsPerTile = 128;
constexpr int kBlockN = 128;
constexpr int kUnitRows = 2 * kRowsPerTile;  // accumulator rows of a unit
// Warps of a unit's rows (two M-tiles x four TMEM lane quarters): a split
// unit has one merge counter per warp.
constexpr int kUnitWarps = 8;

inline int tokens_per_tile(int G) { return kRowsPerTile / G; }
inline int tokens_per_unit(int G) { return 2 * tokens_per_tile(G); }

// One work unit (or one piece of a split unit); 52 bytes, read field by
// field by every role of the CTA that owns it (a 16-byte-aligned record read
// with vector loads keeps every field live and made the kernel spill).
constexpr int kUnitFields = 13;
struct UnitRec {
    int32_t q_tok0;    // packed query row of the unit's first token
    int32_t n_tok;     // valid tokens in the unit (<= 2 * TPB)
    int32_t k_row0;    // packed key row of the sequence's first key
    int32_t Lk;        // keys in the sequence
    int32_t qlim0;     // last visible key index of the first token (= position + Lk - Lq)
    int32_t kvh;       // kv head
    int32_t n_tiles;   // key tiles to visit (0: no row sees a key)
    int32_t seq;       // sequence index (block-table row of a paged cache)
    int32_t tile0;     // first key tile visited (0 unless the unit is a later piece of a split unit)
    int32_t part;      // partial slot of the piece, -1 when the unit is not split
    int32_t group;     // merge counters of the split unit (kUnitWarps each), -1 when not split
    int32_t chunk;     // piece index within the unit; its pieces' slots are part - chunk ...
    int32_t n_chunks;  // pieces of the unit (1 when not split)
};
static_assert(sizeof(UnitRec) == kUnitFields * 4, "UnitRec must stay 52 bytes");

// Device status word values (written by the kernel's bounded waits).
constexpr int32_t kDevOk = 0;
constexpr int32_t kDevTimeout = 1;

// Test-only launch flags: the MMA warp waits on a barrier nothing arrives on,
// so the bounded-wait path runs (short limit, error status, clean exit); in
// every CTA, or only in CTA 0 (the other CTAs finish their units, which
// leaves the merge counters of a split launch part-counted).
constexpr uint32_t kFlagForceTimeout = 1u;
constexpr uint32_t kFlagForceTimeoutFirstCta = 2u;

// Run bookkeeping of a work area whose kernel counts chunk arrivals (the
// split-KV merge): run[0] is the launch epoch, run[1] the CTAs of the current
// launch that have exited.  Every CTA reads the epoch when it starts; the
// last CTA to exit advances it.  A merge counter holds (epoch << 32 | count),
// and a counter written under another epoch counts as zero, so a launch that
// stopped early (a wait timed out) leaves nothing behind that a later launch
// of the same work list could miscount.  Both words start at zero.
struct RunWords {
    uint32_t epoch;
    uint32_t exits;
};

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
    // Split units (only when the schedule has any, else nullptr): merge
    // counters (kUnitWarps per split unit), run words, and the pieces'
    // partial results: part_lse [parts][kUnitRows] (log2 domain) and part_o
    // [parts][d / 4][kUnitRows][4] fp32 (normalised O, four channels per row
    // in a 16-byte group so that a warp's 32 rows are 512 contiguous bytes).
    unsigned long long* counters = nullptr;
    RunWords* run = nullptr;
    float* part_lse = nullptr;
    float* part_o = nullptr;
    // Paged K/V (block_table != nullptr): as in DecodeLaunchArgs.
    const int32_t* block_table = nullptr;
    int32_t max_blocks = 0;
    int32_t block_size = 0;
    int64_t num_blocks = 0;
};

// Limits of the allocation-free entry point (opattn_prefill_noalloc), whose
// work list lives in a fixed device array (opattn_noalloc.cu).
constexpr int64_t kNoAllocMaxUnits = 32768;
constexpr int32_t kNoAllocMaxCtas = 1024;
// Implemented in opattn_noalloc.cu: device address and size of that array on
// the current device (looked up on the first call per device).  Returns a
// cudaError_t as int.
int noalloc_scratch(void** ptr, size_t* bytes);

// ------------------------------------------------------------------ decode
// The decode kernel (opattn_decode.cu) computes the same attention for
// sequences with few query tokens: the G * Lq (query token, head) pairs of
// one kv head form the N = kDecCols columns of transposed score and output
// tiles, the 128 keys of a key tile (or the 128 channels of d) their rows.
// Long key ranges are cut into chunks that run as separate work units; each
// writes a partial (O, LSE) and the last unit of a (sequence, kv head) to
// finish merges them.
constexpr int kDecCols = 32;
constexpr int kDecHeadDim = 128;

struct DecUnit {
    int32_t q_tok0;    // packed query row of the sequence's first token
    int32_t nq;        // query tokens of the sequence (nq * G <= kDecCols)
    int32_t k_row0;    // packed key row of the sequence's first key
    int32_t Lk;        // keys in the sequence
    int32_t kvh;       // kv head
    int32_t tile0;     // first key tile of the chunk
    int32_t n_tiles;   // key tiles of the chunk (0: the sequence has no key)
    int32_t part;      // partial slot of the chunk, -1 when the chunk is the whole sequence
    int32_t group;     // merge counter of the (sequence, kv head), -1 when not split
    int32_t chunk;     // chunk index within the (sequence, kv head)
    int32_t n_chunks;  // chunks of the (sequence, kv head)
    int32_t seq;       // sequence index (diagnostics only)
};
static_assert(sizeof(DecUnit) == 48, "DecUnit must stay 48 bytes");

struct DecodeLaunchArgs {
    const void* q;
    const void* k;
    const void* v;
    void* o;
    float* lse;
    int64_t total_q;
    int64_t total_k;
    int32_t Hq, Hkv;
    float scale;
    const DecUnit* units;     // device
    const int32_t* cta_off;   // device, n_cta + 1
    int32_t n_cta;
    int32_t max_cols;         // largest G * Lq of the batch (<= kDecCols)
    unsigned long long* counters;  // device, two per split (sequence, kv head), zeroed once
    RunWords* run;            // device, zeroed once
    float* part_o;            // device, [parts][kDecCols][kDecHeadDim]
    float* part_lse;          // device, [parts][kDecCols] (log2 domain)
    int32_t* status;          // device
    uint32_t flags;
    // Paged K/V (block_table != nullptr): k and v are [num_blocks, block_size,
    // Hkv, d] caches and key j of sequence s lives in page
    // block_table[s * max_blocks + j / block_size], row j % block_size.
    const int32_t* block_table;  // device, [n_seq][max_blocks]
    int32_t max_blocks;
    int32_t block_size;          // 8, 16, 32, 64 or 128
    int64_t num_blocks;
};

// Implemented in opattn_kernel.cu.  Returns a cudaError_t (as int) or a
// negative value when the tensor maps cannot be encoded.
int launch_prefill(const LaunchArgs& a, cudaStream_t stream);
// Implemented in opattn_decode.cu; same return convention.
int launch_decode(const DecodeLaunchArgs& a, cudaStream_t stream);
// Shared memory bytes the kernel needs for head dim d (0 if unsupported).
int kernel_smem_bytes(int d);
// Implemented in opattn_upload.cu: one small kernel on `stream` copies
// `bytes` (a multiple of 16; src and dst 16-byte aligned) from src, which may
// be mapped pinned host memory, to the device buffer dst, and zeroes
// `zero_words` int32 words at `zero`.  Returns a cudaError_t as int.
int launch_upload(const void* src, void* dst, size_t bytes, int32_t* zero, size_t zero_words, cudaStream_t stream);

}  // namespace opattn
