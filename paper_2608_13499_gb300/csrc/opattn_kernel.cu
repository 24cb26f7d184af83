// opattn_kernel.cu -- persistent sm_103a kernel for ragged causal GQA prefill
// attention (tcgen05 MMAs with TMEM accumulators, TMA + mbarrier K/V ring).
//
// What it computes is exact softmax attention (OpScale §2.1: the attention
// operator is O(L^2 b) in the prompt length and is computed FlashAttention
// style, without materialising the L x L score matrix), with query heads
// grouped over kv heads (§5.6) and a bottom-right-aligned causal mask
// (chunked prefill, §6).  Softmax is evaluated online over 128-key tiles
// with base-2 exponentials; the result equals the two-pass definition up to
// rounding.
//
// CTA layout (384 threads, one CTA per SM, persistent over its unit list):
//   warp 0        TMA producer: Q tiles of the unit, then K_j, V_j into a ring
//   warp 1        TMEM owner + MMA issuer (whole warp, one elected lane issues)
//   warps 2-3     idle
//   warps 4-7     softmax / correction / epilogue of M-tile 0 (one row per thread)
//   warps 8-11    the same for M-tile 1
// TMEM (512 columns): S0 | S1 (128 fp32 columns each; P is written back into
// the first 64 columns as packed bf16) | O0 | O1 (d columns each).
// Shared memory: Q of both M-tiles | K/V ring | (d = 128) one 4 KB O staging
// buffer per softmax warp (32 rows x 64 channels, written out by TMA stores).
//
// MMA order per key tile j (after the prologue S0(0), S1(0)):
//   PV0(j), S0(j+1) -> commit S-ready[0] (or O-ready[0] after the last tile)
//   PV1(j), S1(j+1) -> commit S-ready[1] (or O-ready[1])
// so the tensor pipe works on one M-tile while the other M-tile's softmax
// runs.  tcgen05 MMAs from one thread execute in issue order, so S_i(j+1),
// which overwrites P_i(j), never runs before PV_i(j) has read it, and once
// S_i(j+1) has completed so has PV_i(j): the softmax thread may rescale O_i
// right after it sees S-ready.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "device_common.cuh"
#include "opattn_internal.h"
#include "ptx.cuh"

namespace opattn {
namespace {

constexpr int kThreads = 384;
constexpr int kWarpProducer = 0;
constexpr int kWarpMma = 1;
constexpr int kWarpSoftmax = 4;  // first softmax warp; warps 4..7 -> M-tile 0, 8..11 -> M-tile 1

// Largest sum of one tile's exponentials accepted with a reused subtraction
// base; fp32 sums and the fp32 O accumulator stay far from overflow.
constexpr float kMaxTileSum = 18446744073709551616.0f;  // 2^64
constexpr float kLn2 = 0.693147180559945309f;
// Register split: the kernel is compiled for 168 registers per thread at
// launch (384 threads, one CTA per SM = 64512 registers).  Warpgroup 0
// (producer, MMA, two idle warps) gives registers back, the two softmax
// warpgroups take them: 104 * 128 + 200 * 256 = 168 * 384.  The host refuses
// to launch a build whose register count differs, because a split larger
// than the launch total would make setmaxnreg.inc wait forever.
constexpr int kLaunchRegs = 168;
constexpr uint32_t kRegsControl = 104;
constexpr uint32_t kRegsSoftmax = 200;
static_assert(kRegsControl * 128 + kRegsSoftmax * 256 == kLaunchRegs * kThreads, "register split");
constexpr float kLog2e = 1.442695040888963407f;

template <int D>
struct Cfg {
    static_assert(D == 64 || D == 128, "head dim");
    static constexpr int kDBlocks = D / 64;                        // 128-byte swizzle column blocks
    static constexpr int kQTileBytes = kRowsPerTile * D * 2;       // one M-tile of Q
    static constexpr int kSlotBytes = kBlockN * D * 2;             // one K or V tile
    static constexpr int kSlots = D == 128 ? 4 : 12;               // ring depth (K and V alternate)
    static constexpr int kQOff = 0;
    static constexpr int kRingOff = 2 * kQTileBytes;
    // O staging for TMA stores (d = 128 only): per softmax warp 32 rows x 64 channels
    static constexpr bool kTmaStoreO = D == 128;
    static constexpr int kStageBytes = 32 * 128;
    static constexpr int kStageOff = kRingOff + kSlots * kSlotBytes;
    static constexpr int kBarOff = kStageOff + (kTmaStoreO ? 8 * kStageBytes : 0);
    static constexpr int kBarFull = 0;
    static constexpr int kBarEmpty = kSlots;
    static constexpr int kBarQFull = 2 * kSlots;       // + M-tile
    static constexpr int kBarQEmpty = 2 * kSlots + 2;  // + M-tile
    static constexpr int kBarS = 2 * kSlots + 4;       // S ready (+ M-tile)
    static constexpr int kBarO = 2 * kSlots + 6;       // final O ready (+ M-tile)
    static constexpr int kBarP = 2 * kSlots + 8;       // P written, O corrected (+ M-tile)
    static constexpr int kBarDrain = 2 * kSlots + 10;
    static constexpr int kBarNever = 2 * kSlots + 11;
    static constexpr int kNumBars = 2 * kSlots + 12;
    static constexpr int kMiscOff = kBarOff + kNumBars * 8;  // TMEM base address, abort flag
    static constexpr int kSmemBytes = kMiscOff + 16 + 1024;  // + slack for 1024-byte alignment
    static constexpr uint32_t kTmemCols = 512;
    static constexpr uint32_t kColS = 0;    // + 128 * M-tile
    static constexpr uint32_t kColO = 256;  // + D * M-tile
    static constexpr uint32_t kIdescS = ptx::idesc_bf16_f32(kRowsPerTile, kBlockN, false);
    static constexpr uint32_t kIdescPV = ptx::idesc_bf16_f32(kRowsPerTile, D, true);
    static constexpr uint32_t kQTxBytesPerRow = D * 2;
};

struct KParams {
    const UnitRec* units;
    const int32_t* cta_off;
    uint16_t* o;
    float* lse;
    int32_t Hq, G, TPB;
    float scale_log2;  // softmax scale * log2(e)
    int32_t* status;
    uint32_t flags;
    const int32_t* block_table;  // nullptr: packed K/V
    int32_t max_blocks;
    int32_t page_shift;          // log2(page size)
    int32_t o_tma;               // a warp's 32 rows form one TMA box of O (G divides 32, or 32 divides G)
    // split units (nullptr when the work list has none): see LaunchArgs
    unsigned long long* counters;
    RunWords* run;
    float* part_lse;
    float* part_o;
};

template <int D>
__device__ __forceinline__ void run_producer(const CUtensorMap* tmQ, const CUtensorMap* tmK,
                                             const CUtensorMap* tmV, const KParams& p, int ubeg, int uend,
                                             uint32_t sQ, uint32_t sRing, uint32_t sBar,
                                             volatile int32_t* abort_flag) {
    using C = Cfg<D>;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    const uint32_t q_tx = static_cast<uint32_t>(p.G * p.TPB) * C::kQTxBytesPerRow;
    const uint64_t keep = ptx::policy_evict_last();    // K/V tiles are re-read by other q blocks
    const uint64_t stream = ptx::policy_evict_first();  // each Q tile is read once
    uint32_t slot = 0, ring_par = 0;
    uint32_t q_issued[2] = {0u, 0u};
    uint32_t ring_issued = 0;
    bool aborted = false;
    for (int ui = ubeg; ui < uend && !aborted; ++ui) {
        const UnitRec u = p.units[ui];
        if (u.n_tiles <= 0) continue;
        for (int i = 0; i < 2; ++i) {
            if (!bounded_wait(bar(C::kBarQEmpty + i), (q_issued[i] & 1u) ^ 1u, abort_flag, p.status,
                              kWaitLimitNs)) {
                aborted = true;
                break;
            }
            ptx::mbar_arrive_expect_tx(bar(C::kBarQFull + i), q_tx);
#pragma unroll
            for (int b = 0; b < C::kDBlocks; ++b)
                ptx::tma_load_3d_hint(sQ + i * C::kQTileBytes + b * (kRowsPerTile * 128), tmQ,
                                      bar(C::kBarQFull + i), b * 64, u.kvh * p.G, u.q_tok0 + i * p.TPB,
                                      stream);
            ++q_issued[i];
        }
        for (int j = 0; j < u.n_tiles && !aborted; ++j) {
            for (int kv = 0; kv < 2; ++kv) {
                if (!bounded_wait(bar(C::kBarEmpty + slot), ring_par ^ 1u, abort_flag, p.status,
                                  kWaitLimitNs)) {
                    aborted = true;
                    break;
                }
                ptx::mbar_arrive_expect_tx(bar(C::kBarFull + slot), C::kSlotBytes);
#pragma unroll
                for (int b = 0; b < C::kDBlocks; ++b)
                    ptx::tma_load_3d_hint(sRing + slot * C::kSlotBytes + b * (kBlockN * 128), kv ? tmV : tmK,
                                          bar(C::kBarFull + slot), b * 64, u.kvh, u.k_row0 + (u.tile0 + j) * kBlockN,
                                          keep);
                ++ring_issued;
                if (++slot == C::kSlots) {
                    slot = 0;
                    ring_par ^= 1u;
                }
            }
        }
    }
    if (aborted) {
        // Let every copy still in flight land before the CTA exits: at most
        // one outstanding load per ring slot and per Q buffer (the latest).
        for (uint32_t s = 0; s < static_cast<uint32_t>(C::kSlots); ++s) {
            if (ring_issued > s) {
                const uint32_t uses = (ring_issued - s + C::kSlots - 1) / C::kSlots;
                drain_wait(bar(C::kBarFull + s), (uses - 1u) & 1u, kDrainLimitNs);
            }
        }
        for (int i = 0; i < 2; ++i)
            if (q_issued[i] > 0) drain_wait(bar(C::kBarQFull + i), (q_issued[i] - 1u) & 1u, kDrainLimitNs);
    }
}

// Producer for paged K/V caches (whole warp).  Same order and barriers as
// run_producer; a K or V tile is page_size-row boxes, one page per lane:
// lane i fetches the tile's i-th page id from the block table and issues
// that page's boxes at row offset i * page_size of the slot (a multiple of 8
// rows, so the 128-byte swizzle matches a 128-row box).  Pages past the
// sequence's last page repeat it (those keys are masked), so a tile always
// moves kSlotBytes; an out-of-range page id moves the box outside the cache,
// where TMA reads zeros.
template <int D>
__device__ __forceinline__ void run_producer_paged(const CUtensorMap* tmQ, const CUtensorMap* tmK,
                                                   const CUtensorMap* tmV, const KParams& p, int ubeg, int uend,
                                                   uint32_t sQ, uint32_t sRing, uint32_t sBar, int lane,
                                                   volatile int32_t* abort_flag) {
    using C = Cfg<D>;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    auto wait = [&](int b, uint32_t parity) {
        return __all_sync(0xFFFFFFFFu, bounded_wait(bar(b), parity, abort_flag, p.status, kWaitLimitNs));
    };
    const uint32_t q_tx = static_cast<uint32_t>(p.G * p.TPB) * C::kQTxBytesPerRow;
    const uint64_t keep = ptx::policy_evict_last();
    const uint64_t stream = ptx::policy_evict_first();
    const int page_rows = 1 << p.page_shift;
    const int pages_per_tile = kBlockN >> p.page_shift;
    uint32_t slot = 0, ring_par = 0, ring_issued = 0;
    uint32_t q_issued[2] = {0u, 0u};
    bool aborted = false;
    for (int ui = ubeg; ui < uend && !aborted; ++ui) {
        const UnitRec u = p.units[ui];
        if (u.n_tiles <= 0) continue;
        for (int i = 0; i < 2; ++i) {
            if (!wait(C::kBarQEmpty + i, (q_issued[i] & 1u) ^ 1u)) {
                aborted = true;
                break;
            }
            if (lane == 0) {
                ptx::mbar_arrive_expect_tx(bar(C::kBarQFull + i), q_tx);
#pragma unroll
                for (int b = 0; b < C::kDBlocks; ++b)
                    ptx::tma_load_3d_hint(sQ + i * C::kQTileBytes + b * (kRowsPerTile * 128), tmQ,
                                          bar(C::kBarQFull + i), b * 64, u.kvh * p.G, u.q_tok0 + i * p.TPB, stream);
            }
            ++q_issued[i];
        }
        const int last_page = (u.Lk - 1) >> p.page_shift;
        const int32_t* table = p.block_table + static_cast<int64_t>(u.seq) * p.max_blocks;
        for (int j = 0; j < u.n_tiles && !aborted; ++j) {
            // this lane's page of tile j (the page id is the same for K and V)
            int row = 0;
            if (lane < pages_per_tile) {
                const int page_idx = min((((u.tile0 + j) * kBlockN) >> p.page_shift) + lane, last_page);
                row = static_cast<int>(static_cast<uint32_t>(table[page_idx]) << p.page_shift);
            }
            for (int kv = 0; kv < 2; ++kv) {
                if (!wait(C::kBarEmpty + slot, ring_par ^ 1u)) {
                    aborted = true;
                    break;
                }
                if (lane == 0) ptx::mbar_arrive_expect_tx(bar(C::kBarFull + slot), C::kSlotBytes);
                __syncwarp();
                if (lane < pages_per_tile) {
#pragma unroll
                    for (int b = 0; b < C::kDBlocks; ++b)
                        ptx::tma_load_3d_hint(sRing + slot * C::kSlotBytes + b * (kBlockN * 128) + lane * (page_rows * 128),
                                              kv ? tmV : tmK, bar(C::kBarFull + slot), b * 64, u.kvh, row, keep);
                }
                ++ring_issued;
                if (++slot == C::kSlots) {
                    slot = 0;
                    ring_par ^= 1u;
                }
            }
        }
    }
    if (aborted && lane == 0) {
        for (uint32_t s = 0; s < static_cast<uint32_t>(C::kSlots); ++s) {
            if (ring_issued > s) {
                const uint32_t uses = (ring_issued - s + C::kSlots - 1) / C::kSlots;
                drain_wait(bar(C::kBarFull + s), (uses - 1u) & 1u, kDrainLimitNs);
            }
        }
        for (int i = 0; i < 2; ++i)
            if (q_issued[i] > 0) drain_wait(bar(C::kBarQFull + i), (q_issued[i] - 1u) & 1u, kDrainLimitNs);
    }
    __syncwarp();
}

template <int D>
__device__ __forceinline__ void issue_s(uint32_t tmem, int mt, uint32_t sQ, uint32_t sK) {
    using C = Cfg<D>;
    const uint32_t d_tmem = tmem + C::kColS + 128u * mt;
    const uint32_t qbase = sQ + mt * C::kQTileBytes;
#pragma unroll
    for (int ks = 0; ks < D / 16; ++ks) {
        const uint32_t qoff = (ks >> 2) * (kRowsPerTile * 128) + (ks & 3) * 32;
        const uint32_t koff = (ks >> 2) * (kBlockN * 128) + (ks & 3) * 32;
        ptx::mma_ss_warp(d_tmem, ptx::sdesc_sw128(qbase + qoff, 16, 1024), ptx::sdesc_sw128(sK + koff, 16, 1024),
                         C::kIdescS, ks > 0 ? 1u : 0u);
    }
}

template <int D>
__device__ __forceinline__ void issue_pv(uint32_t tmem, int mt, uint32_t sV, bool accumulate) {
    using C = Cfg<D>;
    const uint32_t d_tmem = tmem + C::kColO + static_cast<uint32_t>(D) * mt;
    const uint32_t a_tmem = tmem + C::kColS + 128u * mt;
#pragma unroll
    for (int ks = 0; ks < kBlockN / 16; ++ks) {
        // V tile is [keys][d] (MN-major for this product): 16 keys per step,
        // 64-column blocks kBlockN * 128 bytes apart, 8-key groups 1024 apart.
        ptx::mma_ts_warp(d_tmem, a_tmem + ks * 8, ptx::sdesc_sw128(sV + ks * (16 * 128), kBlockN * 128, 1024),
                         C::kIdescPV, (accumulate || ks > 0) ? 1u : 0u);
    }
}

template <int D>
__device__ __forceinline__ void run_mma(const KParams& p, int ubeg, int uend, uint32_t tmem, uint32_t sQ,
                                        uint32_t sRing, uint32_t sBar, volatile int32_t* abort_flag) {
    using C = Cfg<D>;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    auto slot_addr = [&](uint32_t s) { return sRing + s * C::kSlotBytes; };
    uint32_t slot = 0, ring_par = 0, q_uses = 0;
    uint32_t p_par[2] = {0u, 0u};
    // Run by all 32 lanes of the MMA warp: waits are made warp-uniform and one
    // elected lane issues each MMA and commit.
    auto wait = [&](int b, uint32_t parity) {
        return __all_sync(0xFFFFFFFFu, bounded_wait(bar(b), parity, abort_flag, p.status, kWaitLimitNs));
    };
    bool ok = true;
    if ((p.flags & kFlagForceTimeout) || ((p.flags & kFlagForceTimeoutFirstCta) && blockIdx.x == 0))
        ok = __all_sync(0xFFFFFFFFu, bounded_wait(bar(C::kBarNever), 0u, abort_flag, p.status, kForcedLimitNs));

    for (int ui = ubeg; ui < uend && ok; ++ui) {
        const UnitRec u = p.units[ui];
        const int nT = u.n_tiles;
        if (nT <= 0) continue;
        // prologue: S0(0), S1(0)
        if (!(ok = wait(C::kBarQFull + 0, q_uses & 1u))) break;
        uint32_t kslot = slot;
        if (!(ok = wait(C::kBarFull + kslot, ring_par))) break;
        if (++slot == C::kSlots) { slot = 0; ring_par ^= 1u; }
        ptx::tc_fence_after();
        issue_s<D>(tmem, 0, sQ, slot_addr(kslot));
        ptx::tc_commit_warp(bar(C::kBarS + 0));
        if (nT == 1) ptx::tc_commit_warp(bar(C::kBarQEmpty + 0));
        if (!(ok = wait(C::kBarQFull + 1, q_uses & 1u))) break;
        ptx::tc_fence_after();
        issue_s<D>(tmem, 1, sQ, slot_addr(kslot));
        ptx::tc_commit_warp(bar(C::kBarS + 1));
        if (nT == 1) ptx::tc_commit_warp(bar(C::kBarQEmpty + 1));
        ptx::tc_commit_warp(bar(C::kBarEmpty + kslot));
        ++q_uses;

        for (int j = 0; j < nT; ++j) {
            const uint32_t vslot = slot;
            if (!(ok = wait(C::kBarFull + vslot, ring_par))) break;
            if (++slot == C::kSlots) { slot = 0; ring_par ^= 1u; }
            const bool more = j + 1 < nT;
            // M-tile 0
            if (!(ok = wait(C::kBarP + 0, p_par[0]))) break;
            p_par[0] ^= 1u;
            ptx::tc_fence_after();
            issue_pv<D>(tmem, 0, slot_addr(vslot), j > 0);
            if (more) {
                kslot = slot;
                if (!(ok = wait(C::kBarFull + kslot, ring_par)))
                    break;
                if (++slot == C::kSlots) { slot = 0; ring_par ^= 1u; }
                issue_s<D>(tmem, 0, sQ, slot_addr(kslot));
                if (j + 2 == nT) ptx::tc_commit_warp(bar(C::kBarQEmpty + 0));
                ptx::tc_commit_warp(bar(C::kBarS + 0));
            } else {
                ptx::tc_commit_warp(bar(C::kBarO + 0));
            }
            // M-tile 1
            if (!(ok = wait(C::kBarP + 1, p_par[1]))) break;
            p_par[1] ^= 1u;
            ptx::tc_fence_after();
            issue_pv<D>(tmem, 1, slot_addr(vslot), j > 0);
            if (more) {
                issue_s<D>(tmem, 1, sQ, slot_addr(kslot));
                if (j + 2 == nT) ptx::tc_commit_warp(bar(C::kBarQEmpty + 1));
                ptx::tc_commit_warp(bar(C::kBarS + 1));
                ptx::tc_commit_warp(bar(C::kBarEmpty + kslot));
            } else {
                ptx::tc_commit_warp(bar(C::kBarO + 1));
            }
            ptx::tc_commit_warp(bar(C::kBarEmpty + vslot));
        }
    }
    // Every MMA this warp issued must finish before TMEM is released.
    ptx::tc_commit_warp(bar(C::kBarDrain));
    drain_wait(bar(C::kBarDrain), 0u, kDrainLimitNs);
}

// N consecutive TMEM columns of this thread's lane into registers.
template <int N>
__device__ __forceinline__ void load_row(uint32_t taddr, uint32_t* r) {
    if constexpr (N == 128) {
        ptx::tmem_ld128(taddr, r);
    } else {
#pragma unroll
        for (int c = 0; c < N; c += 32) ptx::tmem_ld32(taddr + c, r + c);
    }
    ptx::tmem_wait_ld();
    ptx::tmem_ld_fence<N>(r);
}

// Scores of keys beyond this row's last visible key (column > last) -> -inf.
__device__ __forceinline__ void mask_row(uint32_t* s, int last) {
#pragma unroll
    for (int c = 0; c < kBlockN; ++c)
        if (c > last) s[c] = __float_as_uint(-INFINITY);
}

// Row max of 128 scores: 8 independent chains of 16, 3-input max.
__device__ __forceinline__ float row_max(const uint32_t* s) {
    float mx[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) {
        const uint32_t* v = s + 16 * t;
        float a = ptx::max3f(__uint_as_float(v[0]), __uint_as_float(v[1]), __uint_as_float(v[2]));
#pragma unroll
        for (int i = 3; i < 15; i += 2) a = ptx::max3f(a, __uint_as_float(v[i]), __uint_as_float(v[i + 1]));
        mx[t] = fmaxf(a, __uint_as_float(v[15]));
    }
    return ptx::max3f(ptx::max3f(mx[0], mx[1], mx[2]), ptx::max3f(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7]));
}

// p = 2^(s*c - m) for the 128 scores of this row, packed in place as bf16
// pairs into s[0..63]; `sum` gets the sum of the fp32 values, `sumh` the
// sum of the bf16-rounded values the PV MMA consumes.  Per pair: one packed
// FMA, two ex2, one bf16x2 pack, one packed add and two mixed-precision adds.
__device__ __forceinline__ void exp_row(uint32_t* s, float c, float m, float& sum, float& sumh) {
    const float msub = m == -INFINITY ? 0.f : m;
    const uint64_t cc2 = ptx::f32x2(c, c);
    const uint64_t nm2 = ptx::f32x2(-msub, -msub);
    uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};  // (0.f, 0.f) pairs
    float hs[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int c2 = 0; c2 < kBlockN / 2; ++c2) {
        const uint64_t x = ptx::f32x2(__uint_as_float(s[2 * c2]), __uint_as_float(s[2 * c2 + 1]));
        float y0, y1;
        ptx::f32x2_split(ptx::fma_f32x2(x, cc2, nm2), y0, y1);
        const float p0 = ptx::ex2_approx(y0);
        const float p1 = ptx::ex2_approx(y1);
        const uint32_t pk = ptx::pack_bf16x2(p0, p1);
        acc[c2 & 3] = ptx::add_f32x2(acc[c2 & 3], ptx::f32x2(p0, p1));
        hs[(c2 & 3) * 2] = ptx::add_bf16lo(hs[(c2 & 3) * 2], pk);
        hs[(c2 & 3) * 2 + 1] = ptx::add_bf16hi(hs[(c2 & 3) * 2 + 1], pk);
        s[c2] = pk;
    }
    float a = 0.f;
#pragma unroll
    for (int t = 0; t < 4; ++t) {
        float a0, a1;
        ptx::f32x2_split(acc[t], a0, a1);
        a += a0 + a1;
    }
    sum = a;
    sumh = ((hs[0] + hs[1]) + (hs[2] + hs[3])) + ((hs[4] + hs[5]) + (hs[6] + hs[7]));
}

template <int D>
__device__ __forceinline__ void store_zero_row(const KParams& p, int64_t row_idx) {
    uint4* dst = reinterpret_cast<uint4*>(p.o + row_idx * D);
#pragma unroll
    for (int i = 0; i < D / 8; ++i) dst[i] = make_uint4(0u, 0u, 0u, 0u);
    p.lse[row_idx] = -INFINITY;
}

// Epilogue of one row: O / l -> bf16 into this warp's staging buffer and out
// with TMA stores when all 32 rows of the warp belong to the unit (the box
// would otherwise write rows of the next sequence) and d = 128, else with
// predicated 16-byte stores per row.  The staging image is the 128-byte-swizzled box
// (64 channels x the warp's 32 rows): 16-byte chunk c of row r sits at chunk
// c ^ (r & 7), so the 32 lanes' writes of one chunk fill all 32 banks four
// times over.
template <int D>
__device__ __forceinline__ void store_o_rows(const KParams& p, const CUtensorMap* tmO, uint32_t sStage, uint32_t tO,
                                             float inv_l, bool valid, int64_t row_idx, int lane, int32_t c_head,
                                             int32_t c_tok) {
    if (Cfg<D>::kTmaStoreO && p.o_tma && __all_sync(0xFFFFFFFFu, valid)) {
#pragma unroll
        for (int b = 0; b < D / 64; ++b) {
            uint32_t w[32];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                uint32_t ov[32];
                load_row<32>(tO + 64 * b + 32 * h, ov);
#pragma unroll
                for (int t = 0; t < 16; ++t)
                    w[16 * h + t] =
                        ptx::pack_bf16x2(__uint_as_float(ov[2 * t]) * inv_l, __uint_as_float(ov[2 * t + 1]) * inv_l);
            }
            if (lane == 0) ptx::bulk_wait_read_all();  // the previous store from this buffer has read it
            __syncwarp();
            const uint32_t row = sStage + static_cast<uint32_t>(lane) * 128u;
#pragma unroll
            for (int c = 0; c < 8; ++c)
                ptx::st_shared_v4(row + ((static_cast<uint32_t>(c) ^ (lane & 7u)) << 4), w[4 * c], w[4 * c + 1],
                                  w[4 * c + 2], w[4 * c + 3]);
            ptx::fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                ptx::tma_store_3d(tmO, sStage, 64 * b, c_head, c_tok);
                ptx::bulk_commit_group();
            }
        }
        return;
    }
#pragma unroll
    for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t ov[32];
        load_row<32>(tO + 32 * ch, ov);
        uint32_t w[16];
#pragma unroll
        for (int t = 0; t < 16; ++t)
            w[t] = ptx::pack_bf16x2(__uint_as_float(ov[2 * t]) * inv_l, __uint_as_float(ov[2 * t + 1]) * inv_l);
        if (valid) {
            uint4* dst = reinterpret_cast<uint4*>(p.o + row_idx * D + ch * 32);
            dst[0] = make_uint4(w[0], w[1], w[2], w[3]);
            dst[1] = make_uint4(w[4], w[5], w[6], w[7]);
            dst[2] = make_uint4(w[8], w[9], w[10], w[11]);
            dst[3] = make_uint4(w[12], w[13], w[14], w[15]);
        }
    }
}

// Epilogue of one warp's rows for a piece of a split unit.  The piece writes
// its partial result, O / lh in fp32 and the log2-domain LSE of each row,
// then counts itself on the warp's merge counter of the unit.  The piece
// that brings the counter to n_chunks (in this launch's epoch) merges the
// pieces' partials of its 32 rows, O = sum_k 2^(lse_k - M) O_k / W with
// M = max_k lse_k and W = sum_k 2^(lse_k - M), LSE = M + log2 W, puts O
// back into its TMEM accumulator and stores it like an unsplit unit.  Every
// piece of a unit has the same rows in the same warps, so a warp only ever
// reads partials of its own rows and needs no other warp of its CTA.
template <int D>
__device__ __forceinline__ void store_piece(const KParams& p, const CUtensorMap* tmO, uint32_t sStage, uint32_t tO,
                                            const UnitRec& u, int row_u, int warp_u, float inv_l, float lse2,
                                            bool valid, int64_t row_idx, int lane, uint32_t epoch, int32_t c_head,
                                            int32_t c_tok) {
    // [part][d / 4][kUnitRows][4]: the warp's 32 rows are 512 contiguous bytes per channel quad
    float4* po = reinterpret_cast<float4*>(p.part_o + static_cast<int64_t>(u.part) * kUnitRows * D) + row_u;
#pragma unroll
    for (int ch = 0; ch < D / 32; ++ch) {
        uint32_t ov[32];
        load_row<32>(tO + 32 * ch, ov);
#pragma unroll
        for (int t = 0; t < 8; ++t)
            po[(ch * 8 + t) * kUnitRows] =
                make_float4(__uint_as_float(ov[4 * t]) * inv_l, __uint_as_float(ov[4 * t + 1]) * inv_l,
                            __uint_as_float(ov[4 * t + 2]) * inv_l, __uint_as_float(ov[4 * t + 3]) * inv_l);
    }
    p.part_lse[static_cast<int64_t>(u.part) * kUnitRows + row_u] = lse2;
    __threadfence();
    __syncwarp();
    uint32_t count = 0;
    if (lane == 0) count = count_arrival(p.counters + static_cast<int64_t>(u.group) * kUnitWarps + warp_u, epoch);
    count = __shfl_sync(0xFFFFFFFFu, count, 0);
    if (count != static_cast<uint32_t>(u.n_chunks)) return;
    __threadfence();
    const int part0 = u.part - u.chunk;
    const float* pl = p.part_lse + static_cast<int64_t>(part0) * kUnitRows + row_u;
    float M = -INFINITY;
    for (int k = 0; k < u.n_chunks; ++k) M = fmaxf(M, __ldcg(pl + k * kUnitRows));
    float W = 0.f;
    for (int k = 0; k < u.n_chunks; ++k) {
        const float lk = __ldcg(pl + k * kUnitRows);
        W += lk == -INFINITY ? 0.f : ptx::ex2_approx(lk - M);
    }
    const float inv_w = W > 0.f ? 1.f / W : 0.f;
    const float4* src0 = reinterpret_cast<const float4*>(p.part_o + static_cast<int64_t>(part0) * kUnitRows * D) + row_u;
#pragma unroll 1
    for (int ch = 0; ch < D / 32; ++ch) {
        float acc[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) acc[i] = 0.f;
#pragma unroll 1
        for (int k = 0; k < u.n_chunks; ++k) {
            const float lk = __ldcg(pl + k * kUnitRows);
            const float wk = lk == -INFINITY ? 0.f : ptx::ex2_approx(lk - M) * inv_w;
            const float4* src = src0 + static_cast<int64_t>(k) * (kUnitRows * D / 4) + ch * 8 * kUnitRows;
            float4 x[8];
#pragma unroll
            for (int t = 0; t < 8; ++t) x[t] = __ldcg(src + t * kUnitRows);
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                acc[4 * t] = fmaf(wk, x[t].x, acc[4 * t]);
                acc[4 * t + 1] = fmaf(wk, x[t].y, acc[4 * t + 1]);
                acc[4 * t + 2] = fmaf(wk, x[t].z, acc[4 * t + 2]);
                acc[4 * t + 3] = fmaf(wk, x[t].w, acc[4 * t + 3]);
            }
        }
        uint32_t ov[32];
#pragma unroll
        for (int i = 0; i < 32; ++i) ov[i] = __float_as_uint(acc[i]);
        ptx::tmem_st32(tO + 32 * ch, ov);
    }
    ptx::tmem_wait_st();
    store_o_rows<D>(p, tmO, sStage, tO, 1.f, valid, row_idx, lane, c_head, c_tok);
    if (valid) p.lse[row_idx] = W > 0.f ? (M + log2f(W)) * kLn2 : -INFINITY;
}

// kPieces: the work list has pieces of split units.
template <int D, bool kPieces>
__device__ __forceinline__ void softmax_units(const KParams& p, const CUtensorMap* tmO, int ubeg, int uend,
                                              uint32_t tmem, uint32_t sBar, uint32_t sStage, int warp, int lane,
                                              uint32_t epoch, volatile int32_t* abort_flag) {
    using C = Cfg<D>;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    const int mt = (warp - kWarpSoftmax) >> 2;  // M-tile
    const int quarter = warp & 3;               // TMEM lane quarter this warp may access
    const int r = quarter * 32 + lane;          // accumulator row
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t tS = tmem + lane_off + C::kColS + 128u * mt;
    const uint32_t tO = tmem + lane_off + C::kColO + static_cast<uint32_t>(D) * mt;
    const int G = p.G, TPB = p.TPB;
    const int tok_in_tile = r / G;
    const int head_in_group = r - tok_in_tile * G;
    const bool in_tile = r < G * TPB;
    const float cl = p.scale_log2;
    uint32_t s_par = 0, o_par = 0;

    for (int ui = ubeg; ui < uend; ++ui) {
        const UnitRec u = p.units[ui];
        const int tok = mt * TPB + tok_in_tile;  // token index within the unit
        const bool valid = in_tile && tok < u.n_tok;
        const int64_t row_idx = static_cast<int64_t>(u.q_tok0 + tok) * p.Hq + u.kvh * G + head_in_group;
        if (u.n_tiles <= 0) {
            if (valid) store_zero_row<D>(p, row_idx);
            continue;
        }
        // Key limits relative to the unit's first visited tile (tile0 > 0 for a
        // later piece of a split unit): this row's last visible key, and the
        // smallest such limit in the M-tile.
        const int kofs = u.tile0 * kBlockN;
        const int lim = min(u.qlim0 + tok, u.Lk - 1) - kofs;
        const int tile_min_lim = min(u.qlim0 + mt * TPB, u.Lk - 1) - kofs;
        float m = -INFINITY;  // subtraction base, log2 domain
        float l = 0.f;        // running sum of the probabilities (fp32, for LSE)
        float lh = 0.f;       // running sum of the bf16-rounded probabilities PV consumes (normalises O)
        for (int j = 0; j < u.n_tiles; ++j) {
            bool ok = bounded_wait(bar(C::kBarS + mt), s_par, abort_flag, p.status, kWaitLimitNs);
            if (!__all_sync(0xFFFFFFFFu, ok)) return;
            s_par ^= 1u;
            ptx::tc_fence_after();
            uint32_t s[kBlockN];
            load_row<kBlockN>(tS, s);
            const int kbase = j * kBlockN;
            const bool masked = kbase + kBlockN - 1 > tile_min_lim;  // diagonal or tail tile
            if (masked) mask_row(s, lim - kbase);
            // Subtraction base m: the exact row max on the unit's first tile
            // (and while some row of the warp has none yet); later tiles reuse
            // it, since O / l and LSE = m + log2(l) are exact for any base.
            // A tile whose exponentials sum beyond kMaxTileSum is redone with
            // its own exact max (O and the sums rescaled).
            float alpha = 1.f;
            bool rescale = false;
            if (__any_sync(0xFFFFFFFFu, j == 0 || m == -INFINITY)) {
                const float m_tile = row_max(s) * cl;
                if (j == 0) {
                    m = m_tile;
                } else if (m_tile > m) {
                    alpha = m == -INFINITY ? 0.f : ptx::ex2_approx(m - m_tile);
                    m = m_tile;
                    rescale = true;
                }
            }
            float sum, sumh;
            exp_row(s, cl, m, sum, sumh);
            if (__any_sync(0xFFFFFFFFu, !(sum <= kMaxTileSum))) {
                load_row<kBlockN>(tS, s);
                if (masked) mask_row(s, lim - kbase);
                const float m_tile = row_max(s) * cl;
                if (m_tile > m) {
                    alpha *= m == -INFINITY ? 0.f : ptx::ex2_approx(m - m_tile);
                    m = m_tile;
                    rescale = true;
                }
                exp_row(s, cl, m, sum, sumh);
            }
            l = l * alpha + sum;
            lh = lh * alpha + sumh;
            ptx::tmem_st64(tS, s);
            ptx::tmem_wait_st();
            if (__any_sync(0xFFFFFFFFu, rescale)) {
#pragma unroll
                for (int ch = 0; ch < D / 32; ++ch) {
                    uint32_t ov[32];
                    load_row<32>(tO + 32 * ch, ov);
#pragma unroll
                    for (int t = 0; t < 32; ++t) ov[t] = __float_as_uint(__uint_as_float(ov[t]) * alpha);
                    ptx::tmem_st32(tO + 32 * ch, ov);
                }
                ptx::tmem_wait_st();
            }
            ptx::tc_fence_before();
            ptx::mbar_arrive(bar(C::kBarP + mt));
        }
        bool ok = bounded_wait(bar(C::kBarO + mt), o_par, abort_flag, p.status, kWaitLimitNs);
        if (!__all_sync(0xFFFFFFFFu, ok)) return;
        o_par ^= 1u;
        ptx::tc_fence_after();
        // O is normalised by the sum of the same rounded weights the PV MMA
        // used (a weighted mean of V rows); LSE uses the unrounded sum.
        const float inv_l = lh > 0.f ? 1.f / lh : 0.f;
        const float lse_v = l > 0.f ? (m + log2f(l)) * kLn2 : -INFINITY;
        // origin of the TMA box of this warp's 32 rows: (channel, head, token)
        const int tok_w = mt * TPB + (quarter * 32) / G;
        const int head_w = (quarter * 32) % G;
        if constexpr (kPieces) {
            if (u.part >= 0) {
                store_piece<D>(p, tmO, sStage, tO, u, mt * kRowsPerTile + r, mt * 4 + quarter, inv_l,
                               l > 0.f ? m + log2f(l) : -INFINITY, valid, row_idx, lane, epoch, u.kvh * G + head_w,
                               u.q_tok0 + tok_w);
                continue;
            }
        }
        store_o_rows<D>(p, tmO, sStage, tO, inv_l, valid, row_idx, lane, u.kvh * G + head_w, u.q_tok0 + tok_w);
        if (valid) p.lse[row_idx] = lse_v;
    }
}

// Softmax warpgroup role; lane 0 lets its TMA stores finish before the CTA
// exits, also when a wait timed out.
template <int D, bool kPieces>
__device__ __forceinline__ void run_softmax(const KParams& p, const CUtensorMap* tmO, int ubeg, int uend,
                                            uint32_t tmem, uint32_t sBar, uint32_t sStage, int warp, int lane,
                                            uint32_t epoch, volatile int32_t* abort_flag) {
    softmax_units<D, kPieces>(p, tmO, ubeg, uend, tmem, sBar, sStage, warp, lane, epoch, abort_flag);
    if (lane == 0) ptx::bulk_wait_all();
    __syncwarp();
}

// kPieces selects the build for work lists with pieces of split units; lists
// without any run a build that carries none of the piece epilogue (a single
// build measured ~2% slower on unsplit batches).
template <int D, bool kPieces>
__global__ void __launch_bounds__(kThreads, 1)
    opattn_prefill_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                          const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                          const KParams p) {
    using C = Cfg<D>;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;  // 128-byte swizzle atoms need 1024-byte alignment
    uint8_t* gbase = smem_raw + (base - raw);
    const uint32_t sQ = base + C::kQOff;
    const uint32_t sRing = base + C::kRingOff;
    const uint32_t sBar = base + C::kBarOff;
    volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(gbase + C::kMiscOff);
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(gbase + C::kMiscOff + 4);
    volatile uint32_t* epoch_slot = reinterpret_cast<volatile uint32_t*>(gbase + C::kMiscOff + 8);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int i = 0; i < C::kSlots; ++i) {
            ptx::mbar_init(sBar + 8u * (C::kBarFull + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarEmpty + i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(sBar + 8u * (C::kBarQFull + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarQEmpty + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarS + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarO + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarP + i), 128);
        }
        ptx::mbar_init(sBar + 8u * C::kBarDrain, 1);
        ptx::mbar_init(sBar + 8u * C::kBarNever, 1);
        *abort_flag = 0;
        if constexpr (kPieces) *epoch_slot = run_epoch(p.run);
        ptx::fence_mbar_init();
    }
    if (warp == kWarpMma) {
        ptx::tmem_alloc(ptx::smem_addr(const_cast<uint32_t*>(tmem_slot)), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    if (warp == kWarpProducer && lane == 0) {
        ptx::prefetch_tmap(&tmQ);
        ptx::prefetch_tmap(&tmK);
        ptx::prefetch_tmap(&tmV);
        ptx::prefetch_tmap(&tmO);
    }
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t epoch = kPieces ? *epoch_slot : 0u;
    const int ubeg = p.cta_off[blockIdx.x];
    const int uend = p.cta_off[blockIdx.x + 1];

    // Each register-budget change dominates only its own role's code, so the
    // compiler can allocate the softmax path with the larger budget.
    if (warp < kWarpSoftmax) {
        ptx::setmaxnreg_dec<kRegsControl>();
        if (warp == kWarpProducer) {
            if (p.block_table) {
                run_producer_paged<D>(&tmQ, &tmK, &tmV, p, ubeg, uend, sQ, sRing, sBar, lane, abort_flag);
            } else {
                if (lane == 0) run_producer<D>(&tmQ, &tmK, &tmV, p, ubeg, uend, sQ, sRing, sBar, abort_flag);
                __syncwarp();
            }
        } else if (warp == kWarpMma) {
            run_mma<D>(p, ubeg, uend, tmem, sQ, sRing, sBar, abort_flag);
        }
    } else {
        ptx::setmaxnreg_inc<kRegsSoftmax>();
        const uint32_t sStage = base + C::kStageOff + static_cast<uint32_t>(warp - kWarpSoftmax) * C::kStageBytes;
        run_softmax<D, kPieces>(p, &tmO, ubeg, uend, tmem, sBar, sStage, warp, lane, epoch, abort_flag);
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == kWarpMma) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
    if constexpr (kPieces)
        if (threadIdx.x == 0) run_exit(p.run, epoch);
}

template <int D, bool kPieces>
int launch_kernel(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const CUtensorMap& to,
                  const KParams& kp, int n_cta, cudaStream_t stream) {
    using C = Cfg<D>;
    static std::mutex mu;
    static bool attr_done[128] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> g(mu);
        if (dev < 0 || dev >= 128 || !attr_done[dev]) {
            e = cudaFuncSetAttribute(opattn_prefill_kernel<D, kPieces>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     C::kSmemBytes);
            if (e != cudaSuccess) return e;
            if (dev >= 0 && dev < 128) attr_done[dev] = true;
        }
    }
    {
        // The warpgroup register split assumes exactly kLaunchRegs registers
        // per thread at launch; never launch a build that differs.
        static std::once_flag once;
        static int regs = -1;
        std::call_once(once, [] {
            cudaFuncAttributes fa;
            if (cudaFuncGetAttributes(&fa, opattn_prefill_kernel<D, kPieces>) == cudaSuccess) regs = fa.numRegs;
        });
        if (regs != kLaunchRegs) return -6;
    }
    opattn_prefill_kernel<D, kPieces><<<n_cta, kThreads, C::kSmemBytes, stream>>>(tq, tk, tv, to, kp);
    return cudaGetLastError();
}

template <int D>
int launch_d(const LaunchArgs& a, cudaStream_t stream) {
    using C = Cfg<D>;
    EncodeTiledFn fn = encode_fn();
    if (!fn) return -1;
    const int G = a.Hq / a.Hkv;
    const int TPB = kRowsPerTile / G;
    CUtensorMap tq, tk, tv, to;
    // With no keys at all no unit visits a key tile; the K/V maps then only
    // need to be well formed, so they describe one row of q.
    const bool paged = a.block_table != nullptr;
    int page_shift = 0;
    if (paged) {
        while ((1 << page_shift) < a.block_size) ++page_shift;
        if ((1 << page_shift) != a.block_size || a.block_size < 8 || a.block_size > kBlockN) return -5;
    }
    const uint64_t cache_rows = paged ? static_cast<uint64_t>(a.num_blocks) * static_cast<uint64_t>(a.block_size)
                                      : static_cast<uint64_t>(a.total_k);
    const void* kb = cache_rows > 0 ? a.k : a.q;
    const void* vb = cache_rows > 0 ? a.v : a.q;
    const uint64_t krows = cache_rows > 0 ? cache_rows : 1;
    const uint32_t box_rows = paged ? static_cast<uint32_t>(a.block_size) : static_cast<uint32_t>(kBlockN);
    if (!encode_3d(fn, &tq, a.q, D, a.Hq, a.total_q, G, TPB)) return -2;
    if (!encode_3d(fn, &tk, kb, D, a.Hkv, krows, 1, box_rows)) return -3;
    if (!encode_3d(fn, &tv, vb, D, a.Hkv, krows, 1, box_rows)) return -4;
    // O is written by each softmax warp for its 32 rows: G heads x 32 / G
    // tokens, or 32 heads of one token when G > 32.  Other G (3, 5, 6, ...)
    // split a warp's rows across tokens unevenly; those rows use plain stores
    // and the map only needs to be well formed.
    const bool o_tma = G <= 32 ? 32 % G == 0 : G % 32 == 0;
    const uint32_t o_heads = o_tma ? static_cast<uint32_t>(G < 32 ? G : 32) : 1u;
    const uint32_t o_tokens = o_tma ? 32u / o_heads : 1u;
    if (!encode_3d(fn, &to, a.o, D, a.Hq, a.total_q, o_heads, o_tokens)) return -7;

    KParams kp;
    kp.units = a.units;
    kp.cta_off = a.cta_off;
    kp.o = static_cast<uint16_t*>(a.o);
    kp.lse = a.lse;
    kp.Hq = a.Hq;
    kp.G = G;
    kp.TPB = TPB;
    kp.scale_log2 = a.scale * kLog2e;
    kp.status = a.status;
    kp.flags = a.flags;
    kp.block_table = a.block_table;
    kp.max_blocks = a.max_blocks;
    kp.page_shift = page_shift;
    kp.o_tma = o_tma ? 1 : 0;
    kp.counters = a.counters;
    kp.run = a.run;
    kp.part_lse = a.part_lse;
    kp.part_o = a.part_o;
    if (a.part_o) return launch_kernel<D, true>(tq, tk, tv, to, kp, a.n_cta, stream);
    return launch_kernel<D, false>(tq, tk, tv, to, kp, a.n_cta, stream);
}

}  // namespace

// ------------------------------------------------------------------- host

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q = cudaDriverEntryPointSymbolNotFound;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

// [rows, heads, d] bf16 tensor, box of (64 channels, box_heads, box_rows),
// 128-byte swizzle; out-of-range rows read as zero.
bool encode_3d(EncodeTiledFn fn, CUtensorMap* map, const void* base, uint64_t d, uint64_t heads, uint64_t rows,
               uint32_t box_heads, uint32_t box_rows) {
    const cuuint64_t dims[3] = {d, heads, rows};
    const cuuint64_t strides[2] = {d * 2, heads * d * 2};
    const cuuint32_t box[3] = {64, box_heads, box_rows};
    const cuuint32_t estr[3] = {1, 1, 1};
    return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int launch_prefill(const LaunchArgs& a, cudaStream_t stream) {
    if (a.d == 64) return launch_d<64>(a, stream);
    if (a.d == 128) return launch_d<128>(a, stream);
    return -5;
}

int kernel_smem_bytes(int d) {
    if (d == 64) return Cfg<64>::kSmemBytes;
    if (d == 128) return Cfg<128>::kSmemBytes;
    return 0;
}

}  // namespace opattn
