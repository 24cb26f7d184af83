// opattn_decode.cu -- persistent sm_103a kernel for decode-shaped causal GQA
// attention: few query tokens per sequence over a long key range (the decode
// iterations of §3.1, whose per-token latency is the TBT objective).
//
// It computes the same bottom-right-aligned causal softmax attention as the
// prefill kernel.  With G query heads per kv head and Lq <= 32 / G query
// tokens, the (token, head) pairs of one kv head are too few to fill an
// M = 128 tile, so the products are transposed:
//   S^T (128 keys x 32 columns)  = K_tile (128 x d)      . Q^T (d x 32)
//   O^T (d x 32 columns)        += V_tile^T (d x 128 keys) . P^T (128 x 32)
// Both are tcgen05 MMAs with M = 128 (keys, then channels of d) and N = 32,
// so every TMEM lane carries work even at G = 8, Lq = 1.  Column c is query
// token c / G, head c % G of the kv head.  The kernel is bound by HBM: each
// K/V byte is read once and feeds 2 * G * Lq flops.
//
// Softmax runs per column over the keys of a tile, one key per thread (one
// TMEM lane each).  Two softmax warpgroups split the columns: warpgroup w
// owns columns [w * H, w * H + H) of every tile, and both warpgroups' warps
// i and 4 + i read TMEM lane quarter i.  The subtraction base of a column
// is the exact maximum of the chunk's first tile and is reused while no
// score exceeds it by more than 2^kRebaseSlack; a larger score makes the
// warpgroup take the tile's exact maximum and rescale the running sums and
// the O accumulator.  Long key ranges are split into chunks (split-KV); a
// chunk writes its normalised partial O and its log2-domain LSE, and the
// last chunk of a (sequence, kv head) to finish merges the partials with
// LSE weights; each warpgroup counts and merges its own columns.
//
// CTA layout (352 threads, one CTA per SM, persistent over its unit list):
//   warps 0-3  softmax / epilogue / merge of columns [0, H)
//   warps 4-7  the same for columns [H, 2H) (thread t of a warpgroup = TMEM lane t)
//   warp 8     TMA producer: Q^T of the unit, then its K tiles
//   warp 9     TMEM owner + MMA issuer (whole warp, one elected lane issues)
//   warp 10    TMA producer of the V tiles
// TMEM (128 columns): S0 | S1 | S2 (32 fp32 columns each) | O (32 columns).
//
// MMA order within a unit of n tiles (tiles counted across the CTA's units
// as g; S buffer g mod 3, P buffer g mod 2):
//   S(0), S(1), S(2), then per tile: wait P(g), PV(g), S(g + 3)
// S(g + 3) reuses the S buffer of tile g only after P(g) has arrived, i.e.
// after the softmax warps have read S(g); the three S buffers keep the MMA
// round trip off the softmax warps' critical path.
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

constexpr int D = kDecHeadDim;
constexpr int NC = kDecCols;
constexpr int kTile = 128;  // keys per K/V tile
constexpr int kThreadsDec = 352;
constexpr int kWarpProducerDec = 8;   // Q^T and K
constexpr int kWarpMmaDec = 9;
constexpr int kWarpProducerVDec = 10;  // V
constexpr uint32_t kBarWG0 = 1;       // named barrier of softmax warpgroup w: kBarWG0 + w
constexpr uint32_t kWGThreads = 128;
// A score may exceed its column's subtraction base by up to 2^24 in the
// exponential before the base is moved: fp32 sums of up to 2^31 keys and the
// fp32 O accumulator stay far from overflow.
constexpr float kRebaseSlack = 24.f;
constexpr float kLn2Dec = 0.693147180559945309f;
constexpr float kLog2eDec = 1.442695040888963407f;

struct DCfg {
    static constexpr int kQBytes = NC * D * 2;       // Q^T operand: NC rows x d, two 64-channel blocks
    static constexpr int kSlotBytes = kTile * D * 2;  // one K or V tile
    // Two tiles of K and two of V in flight per CTA: with 152 CTAs that is
    // ~19 MB of reads outstanding, enough to keep HBM streaming; three each
    // (~29 MB) measured 3-5% slower.
    static constexpr int kKSlots = 2;
    static constexpr int kVSlots = 2;
    static constexpr int kPBytes = NC * kTile * 2;    // P^T operand: NC rows x 128 keys
    static constexpr int kQOff = 0;                   // two Q buffers (unit parity)
    static constexpr int kKOff = 2 * kQBytes;
    static constexpr int kVOff = kKOff + kKSlots * kSlotBytes;
    static constexpr int kPOff = kVOff + kVSlots * kSlotBytes;  // two P buffers (tile parity)
    static constexpr int kRedOff = kPOff + 2 * kPBytes;         // per warpgroup two [4 warps][16] floats
    static constexpr int kRedBytes = 2 * 2 * 4 * 16 * 4;
    static constexpr int kBarOff = kRedOff + kRedBytes;
    static constexpr int kBarKFull = 0;
    static constexpr int kBarKEmpty = kKSlots;
    static constexpr int kBarVFull = 2 * kKSlots;
    static constexpr int kBarVEmpty = 2 * kKSlots + kVSlots;
    static constexpr int kBarQFull = 2 * kKSlots + 2 * kVSlots;  // + Q buffer
    static constexpr int kBarQEmpty = kBarQFull + 2;
    static constexpr int kSBufs = 3;
    static constexpr int kBarSFull = kBarQEmpty + 2;   // + S buffer
    static constexpr int kBarPFull = kBarSFull + kSBufs;  // + P buffer
    static constexpr int kBarPVDone = kBarPFull + 2;   // + P buffer: PV of that buffer's tile complete
    static constexpr int kBarDrain = kBarPVDone + 2;
    static constexpr int kBarNever = kBarDrain + 1;
    static constexpr int kNumBars = kBarNever + 1;
    static constexpr int kMiscOff = kBarOff + kNumBars * 8;  // TMEM base address, abort flag
    static constexpr int kSmemBytes = kMiscOff + 16 + 1024;  // + slack for 1024-byte alignment
    static constexpr uint32_t kTmemCols = 128;
    static constexpr uint32_t kColS = 0;  // + 32 * S buffer
    static constexpr uint32_t kColO = 96;
    // S^T = K . Q^T: A = K tile (K-major), B = Q^T rows (K-major).
    static constexpr uint32_t kIdescS = ptx::idesc_bf16_f32_ab(kTile, NC, false, false);
    // O^T = V^T . P^T: A = V tile read channel-major (MN-major), B = P^T rows (K-major).
    static constexpr uint32_t kIdescPV = ptx::idesc_bf16_f32_ab(D, NC, true, false);
};
static_assert(DCfg::kSmemBytes <= 232448, "decode kernel shared memory");
static_assert(DCfg::kKOff % 1024 == 0 && DCfg::kVOff % 1024 == 0 && DCfg::kPOff % 1024 == 0,
              "128-byte swizzled operands need 1024-byte alignment");

struct DParams {
    const DecUnit* units;
    const int32_t* cta_off;
    uint16_t* o;
    float* lse;
    int32_t Hq, G, g_shift;  // G = 1 << g_shift
    float scale_log2;         // softmax scale * log2(e)
    unsigned long long* counters;
    RunWords* run;
    float* part_o;
    float* part_lse;
    int32_t* status;
    uint32_t flags;
    const int32_t* block_table;  // nullptr: packed K/V
    int32_t max_blocks;
    int32_t page_shift;          // log2(block_size)
};

// TMA producers (whole warps).  One warp loads the unit's Q^T and its K
// tiles, another its V tiles, so that K loads run ahead as far as the K ring
// allows and are never held behind a V slot (V(j) is freed only by PV(j),
// K(j) already by S(j)).  With packed K/V lane 0 issues a tile as two boxes
// of 128 rows.  With a paged cache lane i fetches the tile's i-th page id
// from the block table and issues that page's boxes; pages past the
// sequence's last page repeat the last page (their keys are masked), so a
// tile always moves kSlotBytes.
template <bool kIsV>
__device__ __forceinline__ void dec_producer(const CUtensorMap* tmQ, const CUtensorMap* tmKV, const DParams& p,
                                             int ubeg, int uend, uint32_t sQ, uint32_t sRing, uint32_t sBar,
                                             int lane, volatile int32_t* abort_flag) {
    using C = DCfg;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    auto wait = [&](int b, uint32_t parity) {
        return __all_sync(0xFFFFFFFFu, bounded_wait(bar(b), parity, abort_flag, p.status, kWaitLimitNs));
    };
    constexpr int kSlots = kIsV ? C::kVSlots : C::kKSlots;
    constexpr int kFull = kIsV ? C::kBarVFull : C::kBarKFull;
    constexpr int kEmpty = kIsV ? C::kBarVEmpty : C::kBarKEmpty;
    const uint64_t once = ptx::policy_evict_first();  // every K/V byte is read once
    const bool paged = p.block_table != nullptr;
    const int page_rows = 1 << p.page_shift;
    const int pages_per_tile = paged ? kTile >> p.page_shift : 0;
    uint32_t slot = 0, par = 0, issued = 0, items = 0;
    uint32_t q_issued[2] = {0u, 0u};
    bool aborted = false;
    for (int ui = ubeg; ui < uend && !aborted; ++ui) {
        const DecUnit u = p.units[ui];
        if (u.n_tiles <= 0) continue;
        if (!kIsV) {
            const int qb = static_cast<int>(items & 1u);
            if (!wait(C::kBarQEmpty + qb, (q_issued[qb] & 1u) ^ 1u)) {
                aborted = true;
                break;
            }
            if (lane == 0) {
                ptx::mbar_arrive_expect_tx(bar(C::kBarQFull + qb), C::kQBytes);
#pragma unroll
                for (int b = 0; b < 2; ++b)
                    ptx::tma_load_3d(sQ + qb * C::kQBytes + b * (NC * 128), tmQ, bar(C::kBarQFull + qb), b * 64,
                                     u.kvh * p.G, u.q_tok0);
            }
            ++q_issued[qb];
            ++items;
        }
        const int last_page = paged ? (u.Lk - 1) >> p.page_shift : 0;
        const int32_t* table = paged ? p.block_table + static_cast<int64_t>(u.seq) * p.max_blocks : nullptr;
        for (int j = 0; j < u.n_tiles; ++j) {
            if (!wait(kEmpty + slot, par ^ 1u)) {
                aborted = true;
                break;
            }
            const uint32_t dst = sRing + slot * C::kSlotBytes;
            if (lane == 0) ptx::mbar_arrive_expect_tx(bar(kFull + slot), C::kSlotBytes);
            __syncwarp();
            if (!paged) {
                if (lane == 0) {
                    const int row = u.k_row0 + (u.tile0 + j) * kTile;
#pragma unroll
                    for (int b = 0; b < 2; ++b)
                        ptx::tma_load_3d_hint(dst + b * (kTile * 128), tmKV, bar(kFull + slot), b * 64, u.kvh, row,
                                              once);
                }
            } else if (lane < pages_per_tile) {
                const int page_idx = min(((u.tile0 + j) * kTile >> p.page_shift) + lane, last_page);
                // A bad page id only moves the box out of the cache, where TMA reads zeros.
                const int row = static_cast<int>(static_cast<uint32_t>(table[page_idx]) << p.page_shift);
#pragma unroll
                for (int b = 0; b < 2; ++b)
                    ptx::tma_load_3d_hint(dst + b * (kTile * 128) + lane * (page_rows * 128), tmKV, bar(kFull + slot),
                                          b * 64, u.kvh, row, once);
            }
            ++issued;
            if (++slot == kSlots) { slot = 0; par ^= 1u; }
        }
    }
    if (aborted && lane == 0) {
        // Let every copy still in flight land before the CTA exits: at most
        // one outstanding tile per slot and per Q buffer (the latest).
        for (uint32_t s = 0; s < static_cast<uint32_t>(kSlots); ++s)
            if (issued > s) {
                const uint32_t uses = (issued - s + kSlots - 1) / kSlots;
                drain_wait(bar(kFull + s), (uses - 1u) & 1u, kDrainLimitNs);
            }
        if (!kIsV)
            for (int i = 0; i < 2; ++i)
                if (q_issued[i] > 0) drain_wait(bar(C::kBarQFull + i), (q_issued[i] - 1u) & 1u, kDrainLimitNs);
    }
    __syncwarp();
}

__device__ __forceinline__ void dec_mma(const DParams& p, int ubeg, int uend, uint32_t tmem, uint32_t sQ,
                                        uint32_t sK, uint32_t sV, uint32_t sP, uint32_t sBar,
                                        volatile int32_t* abort_flag) {
    using C = DCfg;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    auto wait = [&](int b, uint32_t parity) {
        return __all_sync(0xFFFFFFFFu, bounded_wait(bar(b), parity, abort_flag, p.status, kWaitLimitNs));
    };
    uint32_t kslot = 0, kpar = 0, vslot = 0, vpar = 0, items = 0, g = 0;
    uint32_t sbuf = 0;  // S buffer of the next S MMA (tiles are scored in order)
    uint32_t q_uses[2] = {0u, 0u};
    bool ok = true;
    if ((p.flags & kFlagForceTimeout) || ((p.flags & kFlagForceTimeoutFirstCta) && blockIdx.x == 0))
        ok = __all_sync(0xFFFFFFFFu, bounded_wait(bar(C::kBarNever), 0u, abort_flag, p.status, kForcedLimitNs));

    for (int ui = ubeg; ui < uend && ok; ++ui) {
        const DecUnit u = p.units[ui];
        const int n = u.n_tiles;
        if (n <= 0) continue;
        const int qb = static_cast<int>(items & 1u);
        if (!(ok = wait(C::kBarQFull + qb, q_uses[qb] & 1u))) break;
        ++q_uses[qb];
        ++items;
        const uint32_t qaddr = sQ + qb * C::kQBytes;
        // S = K . Q^T from the next K slot into the next S buffer.
        auto issue_s = [&]() -> bool {
            if (!wait(C::kBarKFull + kslot, kpar)) return false;
            ptx::tc_fence_after();
            const uint32_t kaddr = sK + kslot * C::kSlotBytes;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                const uint32_t aoff = (ks >> 2) * (kTile * 128) + (ks & 3) * 32;
                const uint32_t boff = (ks >> 2) * (NC * 128) + (ks & 3) * 32;
                ptx::mma_ss_warp(tmem + C::kColS + 32u * sbuf, ptx::sdesc_sw128(kaddr + aoff, 16, 1024),
                                 ptx::sdesc_sw128(qaddr + boff, 16, 1024), C::kIdescS, ks > 0 ? 1u : 0u);
            }
            ptx::tc_commit_warp(bar(C::kBarSFull + static_cast<int>(sbuf)));
            ptx::tc_commit_warp(bar(C::kBarKEmpty + kslot));
            if (++kslot == C::kKSlots) { kslot = 0; kpar ^= 1u; }
            if (++sbuf == C::kSBufs) sbuf = 0;
            return true;
        };
        const int pre = n < C::kSBufs ? n : C::kSBufs;
        for (int i = 0; i < pre && ok; ++i) ok = issue_s();
        if (!ok) break;
        if (n <= C::kSBufs) ptx::tc_commit_warp(bar(C::kBarQEmpty + qb));
        for (int j = 0; j < n; ++j) {
            const uint32_t gj = g + static_cast<uint32_t>(j);
            const int pb = static_cast<int>(gj & 1u);
            if (!(ok = wait(C::kBarPFull + pb, (gj >> 1) & 1u))) break;
            if (!(ok = wait(C::kBarVFull + vslot, vpar))) break;
            ptx::tc_fence_after();
            const uint32_t vaddr = sV + vslot * C::kSlotBytes;
            const uint32_t paddr = sP + pb * C::kPBytes;
#pragma unroll
            for (int ks = 0; ks < kTile / 16; ++ks) {
                // V tile is [keys][d]: read channel-major, 16 keys per step,
                // 64-channel blocks kTile * 128 bytes apart, 8-key groups 1024 apart.
                const uint32_t boff = (ks >> 2) * (NC * 128) + (ks & 3) * 32;
                ptx::mma_ss_warp(tmem + C::kColO, ptx::sdesc_sw128(vaddr + ks * (16 * 128), kTile * 128, 1024),
                                 ptx::sdesc_sw128(paddr + boff, 16, 1024), C::kIdescPV,
                                 (j > 0 || ks > 0) ? 1u : 0u);
            }
            ptx::tc_commit_warp(bar(C::kBarPVDone + pb));
            ptx::tc_commit_warp(bar(C::kBarVEmpty + vslot));
            if (++vslot == C::kVSlots) { vslot = 0; vpar ^= 1u; }
            if (j + C::kSBufs < n) {
                if (!(ok = issue_s())) break;
                if (j + C::kSBufs + 1 == n) ptx::tc_commit_warp(bar(C::kBarQEmpty + qb));
            }
        }
        g += static_cast<uint32_t>(n);
    }
    // Every MMA this warp issued must finish before TMEM is released.
    ptx::tc_commit_warp(bar(C::kBarDrain));
    drain_wait(bar(C::kBarDrain), 0u, kDrainLimitNs);
}

// Reduces v[c] over the 128 threads of a softmax warpgroup for each of its
// NCOL columns and gives every thread all NCOL results.  Within a warp, lanes
// 8, 16, ... apart are first combined column by column until NCOL lanes are
// left per column; the columns are then halved with butterfly exchanges, so
// lane l ends with column l mod NCOL.  The four warps combine through shared
// memory.
template <int NCOL, bool kMax>
__device__ __forceinline__ void wg_reduce(const float* v, float* out, float* red, int warp, int lane,
                                          uint32_t bar_id) {
    float x[NCOL];
#pragma unroll
    for (int c = 0; c < NCOL; ++c) x[c] = v[c];
#pragma unroll
    for (int o = 16; o >= NCOL; o >>= 1) {
#pragma unroll
        for (int c = 0; c < NCOL; ++c) {
            const float y = __shfl_xor_sync(0xFFFFFFFFu, x[c], o);
            x[c] = kMax ? fmaxf(x[c], y) : x[c] + y;
        }
    }
#pragma unroll
    for (int o = NCOL / 2; o >= 1; o >>= 1) {  // o = number of columns kept
        const bool upper = (lane & o) != 0;
#pragma unroll
        for (int i = 0; i < o; ++i) {
            const float send = upper ? x[i] : x[i + o];
            const float keep = upper ? x[i + o] : x[i];
            const float recv = __shfl_xor_sync(0xFFFFFFFFu, send, o);
            x[i] = kMax ? fmaxf(keep, recv) : keep + recv;
        }
    }
    static_assert(NCOL <= 16, "one warpgroup reduces at most 16 columns");
    if (lane < NCOL) red[warp * 16 + lane] = x[0];
    ptx::bar_sync(bar_id, kWGThreads);
    const int col = lane & (NCOL - 1);
    float t = red[col];
#pragma unroll
    for (int w = 1; w < 4; ++w) t = kMax ? fmaxf(t, red[w * 16 + col]) : t + red[w * 16 + col];
#pragma unroll
    for (int c = 0; c < NCOL; ++c) out[c] = __shfl_sync(0xFFFFFFFFu, t, c);
}

__device__ __forceinline__ uint16_t f32_to_bf16_bits(float x) {
    return static_cast<uint16_t>(ptx::pack_bf16x2(x, 0.f) & 0xFFFFu);
}

__device__ __forceinline__ int64_t out_row(const DParams& p, const DecUnit& u, int c) {
    return static_cast<int64_t>(u.q_tok0 + (c >> p.g_shift)) * p.Hq + u.kvh * p.G + (c & (p.G - 1));
}

// Softmax warpgroup `wg` (0 or 1).  NCOL (4, 8 or 16) is the number of
// S^T / O^T columns each warpgroup processes: half the largest G * Lq of the
// batch, rounded up.  Columns beyond a unit's own G * Lq are masked and never
// written to P^T (zero there).  `tid` is the thread's index in its
// warpgroup, which is also its TMEM lane and the key of the tile it scores.
template <int NCOL>
__device__ __forceinline__ void dec_softmax(const DParams& p, int ubeg, int uend, uint32_t tmem, uint32_t sP,
                                            float* sRed, uint32_t sBar, int wg, int tid, uint32_t epoch,
                                            volatile int32_t* abort_flag) {
    using C = DCfg;
    auto bar = [&](int i) { return sBar + 8u * static_cast<uint32_t>(i); };
    const int warp = tid >> 5, lane = tid & 31;
    const uint32_t kBarWG = kBarWG0 + static_cast<uint32_t>(wg);
    const int col0 = wg * NCOL;  // first column of this warpgroup
    const uint32_t lane_off = static_cast<uint32_t>(warp * 32) << 16;
    const uint32_t tS = tmem + lane_off + C::kColS + static_cast<uint32_t>(col0);
    const uint32_t tO = tmem + lane_off + C::kColO + static_cast<uint32_t>(col0);
    sRed += wg * 128;
    const float cl = p.scale_log2;
    const int gs = p.g_shift;
    // P^T element (column c, key tid): 64-key block, row c, 16-byte chunk swizzled by c mod 8.
    // A lane pair (keys 2i, 2i + 1) writes one 32-bit word per column.
    const uint32_t p_pair = static_cast<uint32_t>((tid >> 6) * (NC * 128) + col0 * 128 + ((tid & 6) << 1));
    const uint32_t p_chunk = static_cast<uint32_t>((tid & 63) >> 3);
    uint32_t g = 0;
    uint32_t sbuf = 0, spar = 0;  // S buffer of tile g (g mod 3) and its phase parity
    int red_buf = 0;
    auto red_ptr = [&]() {
        float* r = sRed + red_buf * 64;
        red_buf ^= 1;
        return r;
    };
    auto warp_wait = [&](int b, uint32_t parity) {
        return __all_sync(0xFFFFFFFFu, bounded_wait(bar(b), parity, abort_flag, p.status, kWaitLimitNs));
    };
    // A wait's outcome is made uniform over the warpgroup before anyone acts
    // on it, so no warp leaves while the others sit in a named barrier.
    auto wg_wait = [&](int b, uint32_t parity) { return ptx::bar_red_and(kBarWG, kWGThreads, warp_wait(b, parity)); };

    for (int ui = ubeg; ui < uend; ++ui) {
        const DecUnit u = p.units[ui];
        const int ncols = u.nq << gs;
        if (u.n_tiles <= 0) {  // the sequence has no key: O = 0, LSE = -inf
#pragma unroll
            for (int c = 0; c < NCOL; ++c) {
                if (col0 + c >= ncols) break;
                const int64_t row = out_row(p, u, col0 + c);
                p.o[row * D + tid] = 0;
                if (tid == c) p.lse[row] = -INFINITY;
            }
            continue;
        }
        const int lim0 = u.Lk - u.nq;  // column c sees keys 0 .. lim0 + c / G
        if (col0 >= ncols) {
            // No column of this unit is ours: keep the P arrivals in step.
            // Waiting for PV(g - 2) keeps an arrival from landing in the
            // previous phase of P buffer b.
            for (int j = 0; j < u.n_tiles; ++j) {
                const uint32_t b = g & 1u;
                const bool ok = g < 2u || warp_wait(C::kBarPVDone + static_cast<int>(b), ((g - 2u) >> 1) & 1u);
                if (!ptx::bar_red_and(kBarWG, kWGThreads, ok)) return;
                ptx::mbar_arrive(bar(C::kBarPFull + static_cast<int>(b)));
                ++g;
                if (++sbuf == C::kSBufs) { sbuf = 0; spar ^= 1u; }
            }
            continue;
        }
        const bool all_used = col0 + NCOL <= ncols;
        float base[NCOL], l[NCOL], lh[NCOL];
#pragma unroll
        for (int c = 0; c < NCOL; ++c) {
            base[c] = -INFINITY;
            l[c] = 0.f;
            lh[c] = 0.f;
        }
        for (int j = 0; j < u.n_tiles; ++j) {
            const uint32_t b = g & 1u;
            // S(g) ready, and P buffer b free (last read by PV(g - 2)).
            bool ok = warp_wait(C::kBarSFull + static_cast<int>(sbuf), spar);
            if (ok && g >= 2u) ok = warp_wait(C::kBarPVDone + static_cast<int>(b), ((g - 2u) >> 1) & 1u);
            // Fast path: past the chunk's first tile (bases set), every key
            // of the tile visible to every column, all columns in use.
            const bool fast = j > 0 && all_used && (u.tile0 + j + 1) * kTile - 1 <= lim0;
            uint32_t sr[NCOL];
            float x[NCOL];  // exponent s - base per column (-inf where masked)
            float s[NCOL];  // scaled scores, -inf where masked (slow path and rebase)
            bool need = j == 0;
            if (ok) {
                ptx::tc_fence_after();
                ptx::tmem_ld_n<NCOL>(tS + 32u * sbuf, sr);
                ptx::tmem_wait_ld();
                ptx::tmem_ld_fence<NCOL>(sr);
                if (fast) {
                    const uint64_t cc = ptx::f32x2(cl, cl);
                    float xm = -INFINITY;
#pragma unroll
                    for (int c = 0; c < NCOL; c += 2) {
                        ptx::f32x2_split(ptx::fma_f32x2(ptx::f32x2(__uint_as_float(sr[c]), __uint_as_float(sr[c + 1])),
                                                        cc, ptx::f32x2(-base[c], -base[c + 1])),
                                         x[c], x[c + 1]);
                        xm = ptx::max3f(xm, x[c], x[c + 1]);
                    }
                    need = xm > kRebaseSlack;
                } else {
                    const int key = (u.tile0 + j) * kTile + tid;
#pragma unroll
                    for (int c = 0; c < NCOL; ++c) {
                        const bool vis = col0 + c < ncols && key <= lim0 + ((col0 + c) >> gs);
                        s[c] = vis ? __uint_as_float(sr[c]) * cl : -INFINITY;
                        need |= s[c] - base[c] > kRebaseSlack;
                    }
                }
            }
            // One warpgroup barrier per tile in the common case: it carries
            // both "some column needs a new base" and "some wait failed".
            const bool rebase = ptx::bar_red_or(kBarWG, kWGThreads, need || !ok);
            if (rebase) {
                if (!ptx::bar_red_and(kBarWG, kWGThreads, ok)) return;
                if (fast) {
#pragma unroll
                    for (int c = 0; c < NCOL; ++c) s[c] = __uint_as_float(sr[c]) * cl;
                }
                float tmax[NCOL];
                wg_reduce<NCOL, true>(s, tmax, red_ptr(), warp, lane, kBarWG);
                bool scaled = false;
                float alpha[NCOL];
#pragma unroll
                for (int c = 0; c < NCOL; ++c) {
                    const float nb = fmaxf(base[c], tmax[c]);
                    alpha[c] = nb == base[c] ? 1.f : (base[c] == -INFINITY ? 0.f : ptx::ex2_approx(base[c] - nb));
                    base[c] = nb;
                    l[c] *= alpha[c];
                    lh[c] *= alpha[c];
                    scaled |= alpha[c] != 1.f;
                }
                // base and tmax are the same in every thread, so is `scaled`.
                if (j > 0 && scaled) {
                    // O holds PV of the earlier tiles on the old bases; the
                    // latest of them, PV(g - 1), must be complete.
                    const uint32_t gp = g - 1u;
                    if (!wg_wait(C::kBarPVDone + static_cast<int>(gp & 1u), (gp >> 1) & 1u)) return;
                    ptx::tc_fence_after();
                    uint32_t ov[NCOL];
                    ptx::tmem_ld_n<NCOL>(tO, ov);
                    ptx::tmem_wait_ld();
                    ptx::tmem_ld_fence<NCOL>(ov);
#pragma unroll
                    for (int c = 0; c < NCOL; ++c) ov[c] = __float_as_uint(__uint_as_float(ov[c]) * alpha[c]);
                    ptx::tmem_st_n<NCOL>(tO, ov);
                    ptx::tmem_wait_st();
                }
            }
            if (rebase || !fast) {
#pragma unroll
                for (int c = 0; c < NCOL; ++c) x[c] = s[c] - (base[c] == -INFINITY ? 0.f : base[c]);
            }
            // Probabilities two columns (c, c ^ kPair) at a time, packed into
            // one bf16x2 word, and the P^T stores as 32-bit words of two
            // adjacent keys: after one exchange the even lane of a pair
            // writes column c, the odd lane column c ^ kPair.  With kPair = 4
            // the two rows a warp writes land in opposite halves of the
            // banks (the swizzle moves row c's chunks by c mod 8), so a warp
            // stores 128 bytes with no conflict.  Masked columns hold p = 0.
            constexpr int kPair = NCOL >= 8 ? 4 : 1;
            const bool odd = (lane & 1) != 0;
            const uint32_t prow = sP + b * C::kPBytes + p_pair;
#pragma unroll
            for (int c = 0; c < NCOL; ++c) {
                if (c & kPair) continue;
                const int c2 = c | kPair;
                const float p0 = ptx::ex2_approx(x[c]);
                const float p1 = ptx::ex2_approx(x[c2]);
                const uint32_t pk = ptx::pack_bf16x2(p0, p1);  // column c low, column c2 high
                l[c] += p0;
                l[c2] += p1;
                lh[c] = ptx::add_bf16lo(lh[c], pk);
                lh[c2] = ptx::add_bf16hi(lh[c2], pk);
                const uint32_t recv = __shfl_xor_sync(0xFFFFFFFFu, pk, 1);
                const uint32_t word = odd ? __byte_perm(pk, recv, 0x3276) : __byte_perm(pk, recv, 0x5410);
                const int cw = odd ? c2 : c;  // column this lane writes
                ptx::st_shared_u32(prow + cw * 128 + ((p_chunk ^ ((col0 + cw) & 7)) << 4), word);
            }
            ptx::fence_proxy_async_smem();
            ptx::tc_fence_before();
            ptx::mbar_arrive(bar(C::kBarPFull + static_cast<int>(b)));
            ++g;
            if (++sbuf == C::kSBufs) { sbuf = 0; spar ^= 1u; }
        }
        // epilogue: wait for the unit's last PV
        const uint32_t gl = g - 1u;
        if (!wg_wait(C::kBarPVDone + static_cast<int>(gl & 1u), (gl >> 1) & 1u)) return;
        ptx::tc_fence_after();
        uint32_t ov[NCOL];
        ptx::tmem_ld_n<NCOL>(tO, ov);
        ptx::tmem_wait_ld();
        ptx::tmem_ld_fence<NCOL>(ov);
        float L[NCOL], LH[NCOL];
        wg_reduce<NCOL, false>(l, L, red_ptr(), warp, lane, kBarWG);
        wg_reduce<NCOL, false>(lh, LH, red_ptr(), warp, lane, kBarWG);
        if (u.part < 0) {
            // O is normalised by the sum of the rounded weights the PV MMA
            // used (a weighted mean of V rows); LSE uses the unrounded sum.
#pragma unroll
            for (int c = 0; c < NCOL; ++c) {
                if (col0 + c >= ncols) break;
                const int64_t row = out_row(p, u, col0 + c);
                const float inv = LH[c] > 0.f ? 1.f / LH[c] : 0.f;
                p.o[row * D + tid] = f32_to_bf16_bits(__uint_as_float(ov[c]) * inv);
                if (tid == c) p.lse[row] = L[c] > 0.f ? (base[c] + log2f(L[c])) * kLn2Dec : -INFINITY;
            }
            continue;
        }
        // split key range: partial (normalised O, log2-domain LSE)
        float* po = p.part_o + static_cast<int64_t>(u.part) * NC * D;
#pragma unroll
        for (int c = 0; c < NCOL; ++c) {
            if (col0 + c >= ncols) break;
            po[(col0 + c) * D + tid] = LH[c] > 0.f ? __uint_as_float(ov[c]) / LH[c] : 0.f;
            if (tid == c) p.part_lse[u.part * NC + col0 + c] = L[c] > 0.f ? base[c] + log2f(L[c]) : -INFINITY;
        }
        __threadfence();
        ptx::bar_sync(kBarWG, kWGThreads);
        bool last = false;
        // Each warpgroup counts the chunks of its own columns; the chunk that
        // brings its counter to n_chunks in this launch's epoch merges.
        if (tid == 0) last = count_arrival(p.counters + 2 * u.group + wg, epoch) == static_cast<uint32_t>(u.n_chunks);
        last = ptx::bar_red_or(kBarWG, kWGThreads, last);
        if (!last) continue;
        // This unit finished last: merge the (sequence, kv head)'s partials,
        // O = sum_k 2^(lse_k - lse) O_k with lse = log2 sum_k 2^lse_k, in one
        // online pass over the chunks.  The loads of kMergeBatch chunks (every
        // column's partial LSE and O) are issued together before any of them
        // is used, so a batch of chunks costs one L2 round trip.  Up to 64
        // loaded values per thread; at 16 columns one chunk's 32 already fill
        // the registers the softmax leaves free.
        __threadfence();
        const int part0 = u.part - u.chunk;
        constexpr int kMergeBatch = NCOL >= 16 ? 1 : 32 / NCOL;
        float m[NCOL], acc[NCOL], wsum[NCOL];
#pragma unroll
        for (int c = 0; c < NCOL; ++c) {
            m[c] = -INFINITY;
            acc[c] = 0.f;
            wsum[c] = 0.f;
        }
        auto merge_chunk = [&](const float (&lk)[NCOL], const float (&ok)[NCOL]) {
#pragma unroll
            for (int c = 0; c < NCOL; ++c) {
                if (lk[c] == -INFINITY) continue;  // this chunk saw no key of column c (or is past the last)
                const float nm = fmaxf(m[c], lk[c]);
                const float a = m[c] == -INFINITY ? 0.f : ptx::ex2_approx(m[c] - nm);
                const float w = ptx::ex2_approx(lk[c] - nm);
                acc[c] = acc[c] * a + w * ok[c];
                wsum[c] = wsum[c] * a + w;
                m[c] = nm;
            }
        };
        if constexpr (kMergeBatch == 1) {
            for (int k = 0; k < u.n_chunks; ++k) {
                const float* plse = p.part_lse + (part0 + k) * NC + col0;
                const float* po_k = p.part_o + (static_cast<int64_t>(part0 + k) * NC + col0) * D + tid;
                float lk[NCOL], ok[NCOL];
#pragma unroll
                for (int c = 0; c < NCOL; ++c) {
                    const bool used = col0 + c < ncols;
                    lk[c] = used ? __ldcg(plse + c) : -INFINITY;
                    ok[c] = used ? __ldcg(po_k + c * D) : 0.f;
                }
                merge_chunk(lk, ok);
            }
        } else {
        for (int k0 = 0; k0 < u.n_chunks; k0 += kMergeBatch) {
            float lk[kMergeBatch][NCOL], ok[kMergeBatch][NCOL];
#pragma unroll
            for (int i = 0; i < kMergeBatch; ++i) {
                const int k = k0 + i;
                const bool have = k < u.n_chunks;
                const float* plse = p.part_lse + static_cast<int64_t>(part0 + (have ? k : 0)) * NC + col0;
                const float* po_k = p.part_o + (static_cast<int64_t>(part0 + (have ? k : 0)) * NC + col0) * D + tid;
#pragma unroll
                for (int c = 0; c < NCOL; ++c) {
                    const bool used = have && col0 + c < ncols;
                    lk[i][c] = used ? __ldcg(plse + c) : -INFINITY;
                    ok[i][c] = used ? __ldcg(po_k + c * D) : 0.f;
                }
            }
#pragma unroll
            for (int i = 0; i < kMergeBatch; ++i) merge_chunk(lk[i], ok[i]);
        }
        }
#pragma unroll
        for (int c = 0; c < NCOL; ++c) {
            if (col0 + c >= ncols) break;
            const int64_t row = out_row(p, u, col0 + c);
            p.o[row * D + tid] = f32_to_bf16_bits(wsum[c] > 0.f ? acc[c] / wsum[c] : 0.f);
            if (tid == 0) p.lse[row] = wsum[c] > 0.f ? (m[c] + log2f(wsum[c])) * kLn2Dec : -INFINITY;
        }
    }
}

template <int NCOL>
__global__ void __launch_bounds__(kThreadsDec, 1)
    opattn_decode_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                         const __grid_constant__ CUtensorMap tmV, const DParams p) {
    using C = DCfg;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    const uint32_t raw = ptx::smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* gbase = smem_raw + (base - raw);
    const uint32_t sQ = base + C::kQOff;
    const uint32_t sK = base + C::kKOff;
    const uint32_t sV = base + C::kVOff;
    const uint32_t sP = base + C::kPOff;
    const uint32_t sBar = base + C::kBarOff;
    float* sRed = reinterpret_cast<float*>(gbase + C::kRedOff);
    volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(gbase + C::kMiscOff);
    volatile int32_t* abort_flag = reinterpret_cast<volatile int32_t*>(gbase + C::kMiscOff + 4);
    volatile uint32_t* epoch_slot = reinterpret_cast<volatile uint32_t*>(gbase + C::kMiscOff + 8);

    const int tid = threadIdx.x;
    const int warp = tid >> 5;
    const int lane = tid & 31;

    if (tid == 0) {
        for (int i = 0; i < C::kKSlots; ++i) {
            ptx::mbar_init(sBar + 8u * (C::kBarKFull + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarKEmpty + i), 1);
        }
        for (int i = 0; i < C::kVSlots; ++i) {
            ptx::mbar_init(sBar + 8u * (C::kBarVFull + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarVEmpty + i), 1);
        }
        for (int i = 0; i < C::kSBufs; ++i) ptx::mbar_init(sBar + 8u * (C::kBarSFull + i), 1);
        for (int i = 0; i < 2; ++i) {
            ptx::mbar_init(sBar + 8u * (C::kBarQFull + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarQEmpty + i), 1);
            ptx::mbar_init(sBar + 8u * (C::kBarPFull + i), 2 * kWGThreads);
            ptx::mbar_init(sBar + 8u * (C::kBarPVDone + i), 1);
        }
        ptx::mbar_init(sBar + 8u * C::kBarDrain, 1);
        ptx::mbar_init(sBar + 8u * C::kBarNever, 1);
        *abort_flag = 0;
        *epoch_slot = run_epoch(p.run);
        ptx::fence_mbar_init();
    }
    if (tid < static_cast<int>(2 * kWGThreads)) {
        // Columns a unit does not use are never written: start them finite.
        constexpr int kPer = 2 * C::kPBytes / (2 * static_cast<int>(kWGThreads));
        const uint32_t dst = sP + static_cast<uint32_t>(tid) * kPer;
#pragma unroll
        for (int i = 0; i < kPer; i += 16) ptx::st_shared_v4(dst + i, 0u, 0u, 0u, 0u);
        ptx::fence_proxy_async_smem();
    }
    if (warp == kWarpMmaDec) {
        ptx::tmem_alloc(ptx::smem_addr(const_cast<uint32_t*>(tmem_slot)), C::kTmemCols);
        ptx::tmem_relinquish();
    }
    if (warp == kWarpProducerDec && lane == 0) {
        ptx::prefetch_tmap(&tmQ);
        ptx::prefetch_tmap(&tmK);
    }
    if (warp == kWarpProducerVDec && lane == 0) ptx::prefetch_tmap(&tmV);
    ptx::tc_fence_before();
    __syncthreads();
    ptx::tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t epoch = *epoch_slot;
    const int ubeg = p.cta_off[blockIdx.x];
    const int uend = p.cta_off[blockIdx.x + 1];

    if (warp < 8) {
        dec_softmax<NCOL>(p, ubeg, uend, tmem, sP, sRed, sBar, warp >> 2, tid & 127, epoch, abort_flag);
    } else if (warp == kWarpProducerDec) {
        dec_producer<false>(&tmQ, &tmK, p, ubeg, uend, sQ, sK, sBar, lane, abort_flag);
    } else if (warp == kWarpProducerVDec) {
        dec_producer<true>(&tmQ, &tmV, p, ubeg, uend, sQ, sV, sBar, lane, abort_flag);
    } else if (warp == kWarpMmaDec) {
        dec_mma(p, ubeg, uend, tmem, sQ, sK, sV, sP, sBar, abort_flag);
    }

    ptx::tc_fence_before();
    __syncthreads();
    if (warp == kWarpMmaDec) {
        ptx::tc_fence_after();
        ptx::tmem_dealloc(tmem, C::kTmemCols);
    }
    if (tid == 0) run_exit(p.run, epoch);
}

template <int NCOL>
int launch_ncol(const DecodeLaunchArgs& a, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                const DParams& kp, cudaStream_t stream) {
    using C = DCfg;
    static std::mutex mu;
    static bool attr_done[128] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    {
        std::lock_guard<std::mutex> lk(mu);
        if (dev < 0 || dev >= 128 || !attr_done[dev]) {
            e = cudaFuncSetAttribute(opattn_decode_kernel<NCOL>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     C::kSmemBytes);
            if (e != cudaSuccess) return e;
            if (dev >= 0 && dev < 128) attr_done[dev] = true;
        }
    }
    opattn_decode_kernel<NCOL><<<a.n_cta, kThreadsDec, C::kSmemBytes, stream>>>(tq, tk, tv, kp);
    return cudaGetLastError();
}

}  // namespace

int launch_decode(const DecodeLaunchArgs& a, cudaStream_t stream) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return -1;
    const int G = a.Hq / a.Hkv;
    if (G <= 0 || NC % G != 0 || a.max_cols <= 0 || a.max_cols > NC) return -5;
    int g_shift = 0;
    while ((1 << g_shift) < G) ++g_shift;
    CUtensorMap tq, tk, tv;
    const bool paged = a.block_table != nullptr;
    int page_shift = 0;
    if (paged) {
        while ((1 << page_shift) < a.block_size) ++page_shift;
        if ((1 << page_shift) != a.block_size || a.block_size < 8 || a.block_size > kTile) return -5;
    }
    // With no keys at all no unit visits a key tile; the K/V maps then only
    // need to be well formed, so they describe one row of q.
    const uint64_t cache_rows = paged ? static_cast<uint64_t>(a.num_blocks) * static_cast<uint64_t>(a.block_size)
                                      : static_cast<uint64_t>(a.total_k);
    const void* kb = cache_rows > 0 ? a.k : a.q;
    const void* vb = cache_rows > 0 ? a.v : a.q;
    const uint64_t krows = cache_rows > 0 ? cache_rows : 1;
    const uint32_t box_rows = paged ? static_cast<uint32_t>(a.block_size) : static_cast<uint32_t>(kTile);
    if (!encode_3d(fn, &tq, a.q, D, a.Hq, a.total_q, G, NC / G)) return -2;
    if (!encode_3d(fn, &tk, kb, D, a.Hkv, krows, 1, box_rows)) return -3;
    if (!encode_3d(fn, &tv, vb, D, a.Hkv, krows, 1, box_rows)) return -4;
    DParams kp;
    kp.units = a.units;
    kp.cta_off = a.cta_off;
    kp.o = static_cast<uint16_t*>(a.o);
    kp.lse = a.lse;
    kp.Hq = a.Hq;
    kp.G = G;
    kp.g_shift = g_shift;
    kp.scale_log2 = a.scale * kLog2eDec;
    kp.counters = a.counters;
    kp.run = a.run;
    kp.part_o = a.part_o;
    kp.part_lse = a.part_lse;
    kp.status = a.status;
    kp.flags = a.flags;
    kp.block_table = a.block_table;
    kp.max_blocks = a.max_blocks;
    kp.page_shift = page_shift;
    // columns per softmax warpgroup
    if (a.max_cols <= 8) return launch_ncol<4>(a, tq, tk, tv, kp, stream);
    if (a.max_cols <= 16) return launch_ncol<8>(a, tq, tk, tv, kp, stream);
    return launch_ncol<16>(a, tq, tk, tv, kp, stream);
}

}  // namespace opattn
