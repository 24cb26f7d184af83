// opattn_api.cpp -- host runtime of libopattn: argument validation, the
// longest-first ragged work-list scheduler, pinned staging for the work
// list, reusable plans and the C-ABI entry points declared in opattn.h.
#include "opattn.h"

#include <cuda_runtime.h>

#include <algorithm>
#include <array>
#include <chrono>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <functional>
#include <mutex>
#include <queue>
#include <utility>
#include <vector>

#include "opattn_internal.h"

namespace opattn {
namespace {

constexpr int32_t kVersion = 10100;  // 1.1.0

struct Geometry {
    int32_t n_seq, Hq, Hkv, d, G, TPB;
    int64_t total_q, total_k;
};

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Checks that do not touch tensor pointers.
opattn_status check_geometry(const int32_t* cu_q, const int32_t* cu_k, int32_t n_seq, int32_t Hq, int32_t Hkv,
                             int32_t d, Geometry* g) {
    if (n_seq < 0 || Hq <= 0 || Hkv <= 0) return OPATTN_ERR_INVALID_ARG;
    if (n_seq > 0 && (!cu_q || !cu_k)) return OPATTN_ERR_INVALID_ARG;
    if (Hq % Hkv != 0) return OPATTN_ERR_INVALID_ARG;
    if (d != 64 && d != 128) return OPATTN_ERR_UNSUPPORTED;
    const int32_t G = Hq / Hkv;
    if (G > kRowsPerTile) return OPATTN_ERR_UNSUPPORTED;
    if (n_seq > 0) {
        if (cu_q[0] != 0 || cu_k[0] != 0) return OPATTN_ERR_INVALID_ARG;
        for (int32_t s = 0; s < n_seq; ++s)
            if (cu_q[s + 1] < cu_q[s] || cu_k[s + 1] < cu_k[s]) return OPATTN_ERR_INVALID_ARG;
    }
    g->n_seq = n_seq;
    g->Hq = Hq;
    g->Hkv = Hkv;
    g->d = d;
    g->G = G;
    g->TPB = tokens_per_tile(G);
    g->total_q = n_seq > 0 ? cu_q[n_seq] : 0;
    g->total_k = n_seq > 0 ? cu_k[n_seq] : 0;
    // Packed row indices (token * heads + head) must fit the 32-bit unit
    // fields and the 32-bit TMA coordinates.
    if (g->total_q * static_cast<int64_t>(Hq) >= (int64_t{1} << 31)) return OPATTN_ERR_UNSUPPORTED;
    if (g->total_k * static_cast<int64_t>(Hkv) >= (int64_t{1} << 31)) return OPATTN_ERR_UNSUPPORTED;
    return OPATTN_OK;
}

opattn_status check_tensors(const void* q, const void* k, const void* v, const void* o, const float* lse,
                            float scale, const Geometry& g) {
    if (!(std::isfinite(scale) && scale > 0.f)) return OPATTN_ERR_INVALID_ARG;
    if (!q || !o || !lse) return OPATTN_ERR_INVALID_ARG;
    if (g.total_k > 0 && (!k || !v)) return OPATTN_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(o, 16) || !aligned(lse, 4)) return OPATTN_ERR_MISALIGNED;
    if (g.total_k > 0 && (!aligned(k, 16) || !aligned(v, 16))) return OPATTN_ERR_MISALIGNED;
    return OPATTN_OK;
}

// ------------------------------------------------------------- scheduler

struct Schedule {
    std::vector<UnitRec> units;    // grouped by CTA, in the order each CTA runs them
    std::vector<int32_t> cta_off;  // n_cta + 1
    int32_t n_cta = 0;
    int32_t n_groups = 0;          // split units (kUnitWarps merge counters each)
    int32_t n_parts = 0;           // pieces of split units (one partial slot each)
};

// K/V bytes of the (sequence, kv head) pairs whose units run together: small
// enough that their K/V stays in L2 (129 MB) while all their q-blocks read it.
constexpr int64_t kL2GroupBytes = 48ll << 20;

// Greedy list scheduling in the given order: each unit goes to the CTA with
// the least cost so far (ties: lower CTA index); a CTA's units keep the
// order.  Makespan within mean load + largest unit.
//
// The least-loaded CTA comes from a bucket queue: loads only grow, the least
// load only grows, and every load lies within the largest unit cost C of the
// least one, so C + 1 circular buckets indexed by load hold every CTA
// without collisions.  Each bucket is a bitset of CTAs; its lowest set bit is
// the lowest CTA index at that load, which is the order of (load, index)
// pairs.  Batches whose buckets would take more than kMaxBucketWords words
// use a heap of (load, index) pairs instead.
// The units are taken in the order order[0], order[1], ... (indices into `all`).
// The working arrays are kept per host thread and reused, so that a call
// allocates (and page-faults in) nothing once the thread has scheduled a
// batch as large.
template <class U, class CostFn>
void list_pack(const std::vector<U>& all, const std::vector<uint32_t>& order, int32_t max_ctas, CostFn cost,
               std::vector<U>* units, std::vector<int32_t>* cta_off, int32_t* n_cta_out) {
    auto ordered = [&](int64_t i) -> const U& { return all[order[static_cast<size_t>(i)]]; };
    const int64_t n = static_cast<int64_t>(order.size());
    cta_off->clear();
    *n_cta_out = 0;
    if (n == 0) {
        units->clear();
        return;
    }
    const int32_t n_cta = static_cast<int32_t>(std::min<int64_t>(std::max<int32_t>(max_ctas, 1), n));
    thread_local std::vector<int32_t> owner, per_cta, costs, count, fill;
    thread_local std::vector<uint64_t> bits;
    thread_local std::vector<int64_t> load;
    owner.resize(static_cast<size_t>(n));
    costs.resize(static_cast<size_t>(n));
    per_cta.assign(static_cast<size_t>(n_cta), 0);
    int64_t max_cost = 1;
    for (int64_t i = 0; i < n; ++i) {
        const int64_t c = cost(ordered(i));
        costs[static_cast<size_t>(i)] = static_cast<int32_t>(c);
        max_cost = std::max<int64_t>(max_cost, c);
    }
    const size_t words = (static_cast<size_t>(n_cta) + 63) / 64;
    constexpr size_t kMaxBucketWords = size_t{1} << 20;
    const size_t n_buckets = static_cast<size_t>(max_cost) + 1;
    if (n_buckets * words <= kMaxBucketWords) {
        bits.assign(n_buckets * words, 0);
        count.assign(n_buckets, 0);
        load.assign(static_cast<size_t>(n_cta), 0);
        for (int32_t c = 0; c < n_cta; ++c) bits[static_cast<size_t>(c) >> 6] |= uint64_t{1} << (c & 63);
        count[0] = n_cta;
        int64_t least = 0;  // least load of any CTA
        size_t b = 0;       // its bucket, least mod n_buckets
        for (int64_t i = 0; i < n; ++i) {
            while (count[b] == 0) {
                ++least;
                if (++b == n_buckets) b = 0;
            }
            uint64_t* row = bits.data() + b * words;
            size_t wi = 0;
            while (row[wi] == 0) ++wi;
            const int32_t c = static_cast<int32_t>(wi * 64 + static_cast<size_t>(__builtin_ctzll(row[wi])));
            row[wi] &= row[wi] - 1;
            --count[b];
            owner[static_cast<size_t>(i)] = c;
            ++per_cta[static_cast<size_t>(c)];
            const int64_t nl = load[static_cast<size_t>(c)] + costs[static_cast<size_t>(i)];
            load[static_cast<size_t>(c)] = nl;
            // c came from bucket b (load `least`) and costs are below n_buckets
            size_t nb = b + static_cast<size_t>(costs[static_cast<size_t>(i)]);
            if (nb >= n_buckets) nb -= n_buckets;
            bits[nb * words + (static_cast<size_t>(c) >> 6)] |= uint64_t{1} << (c & 63);
            ++count[nb];
        }
    } else {
        using Slot = std::pair<int64_t, int32_t>;
        std::priority_queue<Slot, std::vector<Slot>, std::greater<Slot>> heap;
        for (int32_t c = 0; c < n_cta; ++c) heap.push({0, c});
        for (int64_t i = 0; i < n; ++i) {
            Slot sl = heap.top();
            heap.pop();
            owner[static_cast<size_t>(i)] = sl.second;
            ++per_cta[static_cast<size_t>(sl.second)];
            sl.first += costs[static_cast<size_t>(i)];
            heap.push(sl);
        }
    }
    cta_off->assign(static_cast<size_t>(n_cta) + 1, 0);
    for (int32_t c = 0; c < n_cta; ++c)
        (*cta_off)[static_cast<size_t>(c) + 1] = (*cta_off)[static_cast<size_t>(c)] + per_cta[static_cast<size_t>(c)];
    fill.assign(cta_off->begin(), cta_off->end() - 1);
    units->resize(static_cast<size_t>(n));
    for (int64_t i = 0; i < n; ++i) {
        const int32_t c = owner[static_cast<size_t>(i)];
        (*units)[static_cast<size_t>(fill[static_cast<size_t>(c)]++)] = ordered(i);
    }
    *n_cta_out = n_cta;
}

// Split-KV for units over long key ranges.  When a batch has few units for
// the grid (one prompt chunk over a long cached prefix, say), the longest
// unit sets the list schedule's makespan however the rest are placed.  The
// stream-K cut takes the key tiles of all units in pair order and cuts them
// into one equal stretch per CTA; a unit that falls into several stretches
// becomes pieces on consecutive CTAs, each over its own run of key tiles,
// and the piece that finishes last merges the pieces' partial results.  A
// piece costs its tiles, one for its Q load and epilogue, and one more for
// writing its partial result and its share of the merge.
constexpr int64_t kPieceOverhead = 2;
// The cut replaces the list schedule only when its makespan (in those costs)
// is below this fraction of the list schedule's, and only when a CTA's
// stretch is at least kMinStretchTiles key tiles: below that the batch is
// small enough that launch and load latency, not the makespan, set its time.
constexpr double kSplitGain = 0.85;
constexpr int64_t kMinStretchTiles = 4;

int64_t max_cta_load(const std::vector<UnitRec>& units, const std::vector<int32_t>& cta_off) {
    int64_t mx = 0;
    for (size_t c = 0; c + 1 < cta_off.size(); ++c) {
        int64_t load = 0;
        for (int32_t i = cta_off[c]; i < cta_off[c + 1]; ++i) {
            const UnitRec& u = units[static_cast<size_t>(i)];
            load += u.n_tiles + 1 + (u.part >= 0 ? kPieceOverhead : 0);
        }
        mx = std::max(mx, load);
    }
    return mx;
}

// The stream-K cut of `all` (units in pair order) over at most max_ctas CTAs.
// Units without key tiles are spread over the CTAs round robin.
void stream_k_prefill(const std::vector<UnitRec>& all, int32_t max_ctas, Schedule* out) {
    int64_t total = 0;
    for (const UnitRec& u : all) total += u.n_tiles;
    out->units.clear();
    out->cta_off.clear();
    out->n_groups = 0;
    out->n_parts = 0;
    const int32_t n_cta = static_cast<int32_t>(std::max<int64_t>(1, std::min<int64_t>(max_ctas, total)));
    std::vector<std::vector<UnitRec>> per_cta(static_cast<size_t>(n_cta));
    auto bound = [&](int64_t c) { return c * total / n_cta; };  // first tile of CTA c's stretch
    int64_t pos = 0;
    int32_t rr = 0;
    for (const UnitRec& u : all) {
        if (u.n_tiles <= 0) {
            per_cta[static_cast<size_t>(rr)].push_back(u);
            rr = (rr + 1) % n_cta;
            continue;
        }
        int64_t c = std::min<int64_t>(n_cta - 1, pos * n_cta / total);
        while (c > 0 && bound(c) > pos) --c;
        while (c + 1 < n_cta && bound(c + 1) <= pos) ++c;
        const int64_t end = pos + u.n_tiles;
        std::vector<std::array<int64_t, 3>> pieces;  // (CTA, first tile, tiles)
        for (int64_t t = pos; t < end; ++c) {
            const int64_t stop = std::min<int64_t>(end, bound(c + 1));
            if (stop > t) pieces.push_back({c, t - pos, stop - t});
            t = stop;
        }
        const int32_t k = static_cast<int32_t>(pieces.size());
        for (int32_t i = 0; i < k; ++i) {
            UnitRec p = u;
            p.tile0 = static_cast<int32_t>(pieces[static_cast<size_t>(i)][1]);
            p.n_tiles = static_cast<int32_t>(pieces[static_cast<size_t>(i)][2]);
            p.part = k > 1 ? out->n_parts + i : -1;
            p.group = k > 1 ? out->n_groups : -1;
            p.chunk = i;
            p.n_chunks = k;
            per_cta[static_cast<size_t>(pieces[static_cast<size_t>(i)][0])].push_back(p);
        }
        if (k > 1) {
            out->n_parts += k;
            ++out->n_groups;
        }
        pos = end;
    }
    out->cta_off.assign(static_cast<size_t>(n_cta) + 1, 0);
    for (int32_t c = 0; c < n_cta; ++c) {
        const auto& v = per_cta[static_cast<size_t>(c)];
        out->cta_off[static_cast<size_t>(c) + 1] = out->cta_off[static_cast<size_t>(c)] + static_cast<int32_t>(v.size());
        out->units.insert(out->units.end(), v.begin(), v.end());
    }
    out->n_cta = n_cta;
}

// Replaces the list schedule in `out` by the stream-K cut of `all` when the
// cut's makespan is below kSplitGain of the list schedule's.  A quick bound
// first: the cut cannot beat mean load + 2 pieces' overhead, so batches whose
// list schedule is already within that are left alone.
void split_if_faster(const std::vector<UnitRec>& all, int32_t max_ctas, Schedule* out) {
    if (out->n_cta <= 0 || all.empty()) return;
    int64_t total = 0, tiles = 0;
    for (const UnitRec& u : all) {
        total += u.n_tiles + 1;
        tiles += u.n_tiles;
    }
    const int32_t cap = std::max<int32_t>(max_ctas, 1);
    if (tiles < kMinStretchTiles * cap) return;
    const int64_t lpt = max_cta_load(out->units, out->cta_off);
    const double floor = static_cast<double>(total) / cap;
    if (static_cast<double>(lpt) * kSplitGain <= floor) return;
    Schedule sk;
    stream_k_prefill(all, cap, &sk);
    if (static_cast<double>(max_cta_load(sk.units, sk.cta_off)) < kSplitGain * static_cast<double>(lpt)) *out = sk;
}

// Units are (sequence, kv head, block of 2 * TPB query tokens).  Cost is the
// number of key tiles the block visits after whole tiles above the causal
// diagonal are skipped, plus one for the Q load and the epilogue.  Pairs
// (sequence, kv head) are taken in order and gathered into groups of at most
// kL2GroupBytes of K/V; the units are assigned group by group, longest first
// within a group, each to the CTA with the least cost so far.  A CTA runs its
// units in that order, so at any time the CTAs work on one group and each
// K/V tile comes from HBM about once; across the whole list the greedy
// assignment keeps the makespan within mean load + largest unit.  The
// longest-first order within a group is a stable counting sort on the tile
// count (O(units + tiles) per group).  The working arrays are kept per host
// thread and reused (see list_pack).
void build_schedule(const int32_t* cu_q, const int32_t* cu_k, const Geometry& g, int32_t max_ctas, Schedule* out,
                    bool allow_split = true) {
    const int32_t tpu = 2 * g.TPB;
    int64_t n_units = 0;
    for (int32_t s = 0; s < g.n_seq; ++s) n_units += (static_cast<int64_t>(cu_q[s + 1] - cu_q[s]) + tpu - 1) / tpu;
    n_units *= g.Hkv;
    thread_local std::vector<UnitRec> all;
    thread_local std::vector<size_t> group_start;  // index in `all` of each group's first unit
    thread_local std::vector<int32_t> group_max;   // most key tiles of a unit in the group
    thread_local std::vector<uint32_t> order;
    thread_local std::vector<size_t> slot;
    all.resize(static_cast<size_t>(n_units));
    group_start.clear();
    group_max.clear();
    int64_t group_bytes = 0;
    const int64_t pair_row_bytes = 2 * static_cast<int64_t>(g.d) * 2;  // K and V, bf16
    size_t n = 0;
    for (int32_t s = 0; s < g.n_seq; ++s) {
        const int32_t Lq = cu_q[s + 1] - cu_q[s];
        const int32_t Lk = cu_k[s + 1] - cu_k[s];
        const int32_t delta = Lk - Lq;
        if (Lq == 0) continue;
        // the units of kv head 0; the other heads' differ only in the head
        const size_t first = n;
        int32_t seq_max = 0;
        for (int32_t t0 = 0; t0 < Lq; t0 += tpu) {
            const int32_t n_tok = std::min(tpu, Lq - t0);
            const int32_t qlim0 = t0 + delta;
            const int32_t last_key = std::min(qlim0 + n_tok - 1, Lk - 1);
            const int32_t n_tiles = last_key < 0 ? 0 : last_key / kBlockN + 1;
            seq_max = std::max(seq_max, n_tiles);
            UnitRec& u = all[n++];
            u.q_tok0 = cu_q[s] + t0;
            u.n_tok = n_tok;
            u.k_row0 = cu_k[s];
            u.Lk = Lk;
            u.qlim0 = qlim0;
            u.kvh = 0;
            u.n_tiles = n_tiles;
            u.seq = s;
            u.tile0 = 0;
            u.part = -1;
            u.group = -1;
            u.chunk = 0;
            u.n_chunks = 1;
        }
        const size_t per_head = n - first;
        const int64_t pair_bytes = static_cast<int64_t>(Lk) * pair_row_bytes;
        for (int32_t h = 0; h < g.Hkv; ++h) {
            if (group_start.empty() || (group_bytes > 0 && group_bytes + pair_bytes > kL2GroupBytes)) {
                group_start.push_back(first + static_cast<size_t>(h) * per_head);
                group_max.push_back(0);
                group_bytes = 0;
            }
            group_bytes += pair_bytes;
            group_max.back() = std::max(group_max.back(), seq_max);
            if (h == 0) continue;
            UnitRec* dst = all.data() + first + static_cast<size_t>(h) * per_head;
            std::memcpy(dst, all.data() + first, per_head * sizeof(UnitRec));
            for (size_t i = 0; i < per_head; ++i) dst[i].kvh = h;
        }
        n = first + static_cast<size_t>(g.Hkv) * per_head;
    }
    // group by group, longest first within a group (stable counting sort of indices)
    order.resize(all.size());
    group_start.push_back(all.size());
    for (size_t gi = 0; gi + 1 < group_start.size(); ++gi) {
        const size_t b = group_start[gi], e = group_start[gi + 1];
        const int32_t mx = group_max[gi];
        slot.assign(static_cast<size_t>(mx) + 2, 0);
        for (size_t i = b; i < e; ++i) ++slot[static_cast<size_t>(mx - all[i].n_tiles) + 1];  // rank 0 = most tiles
        slot[0] = b;
        for (size_t r = 1; r < slot.size(); ++r) slot[r] += slot[r - 1];
        for (size_t i = b; i < e; ++i) order[slot[static_cast<size_t>(mx - all[i].n_tiles)]++] = static_cast<uint32_t>(i);
    }
    list_pack(all, order, max_ctas, [](const UnitRec& u) { return u.n_tiles + 1; }, &out->units, &out->cta_off,
              &out->n_cta);
    out->n_groups = 0;
    out->n_parts = 0;
    if (allow_split) split_if_faster(all, max_ctas, out);
}

// Device work area: [cta_off (n_cta + 1) | pad to 32 B | units | merge
// counters (kUnitWarps per split unit, 8 bytes each) | run words | status |
// pad 256 | part_lse (n_parts x kUnitRows fp32) | part_o (n_parts x
// kUnitRows x d fp32)].  The counters, run words and status word are
// contiguous: the one-shot calls zero them with the work-list upload, a plan
// once when it is created (the counters carry the launch epoch, RunWords).
struct WorkLayout {
    size_t off_units, off_counters, off_run, off_status, off_part_lse, off_part_o, bytes, upload_bytes, zero_bytes;
};
WorkLayout work_layout(const Schedule& s, int32_t d) {
    WorkLayout w;
    w.off_units = (s.cta_off.size() * sizeof(int32_t) + 31) / 32 * 32;
    w.off_counters = (w.off_units + s.units.size() * sizeof(UnitRec) + 15) / 16 * 16;
    w.off_run = w.off_counters + static_cast<size_t>(s.n_groups) * kUnitWarps * sizeof(unsigned long long);
    w.off_status = w.off_run + sizeof(RunWords);
    w.upload_bytes = w.off_counters;
    w.zero_bytes = w.off_status + sizeof(int32_t) - w.off_counters;
    w.off_part_lse = (w.off_status + sizeof(int32_t) + 255) / 256 * 256;
    w.off_part_o = w.off_part_lse + (static_cast<size_t>(s.n_parts) * kUnitRows * sizeof(float) + 255) / 256 * 256;
    w.bytes = w.off_part_o + static_cast<size_t>(s.n_parts) * kUnitRows * static_cast<size_t>(d) * sizeof(float);
    return w;
}
// Writes each byte of the upload once: the offsets, the units and zeros in
// the two alignment gaps.
void pack_upload(const Schedule& s, const WorkLayout& w, uint8_t* dst) {
    const size_t off_bytes = s.cta_off.size() * sizeof(int32_t);
    const size_t end_units = w.off_units + s.units.size() * sizeof(UnitRec);
    std::memcpy(dst, s.cta_off.data(), off_bytes);
    std::memset(dst + off_bytes, 0, w.off_units - off_bytes);
    std::memcpy(dst + w.off_units, s.units.data(), s.units.size() * sizeof(UnitRec));
    std::memset(dst + end_units, 0, w.upload_bytes - end_units);
}

// ------------------------------------------------------ OPATTN_LOG=1
// With OPATTN_LOG set to anything but "0" in the environment, every schedule
// the library builds prints one line on stderr: work units, CTAs, the largest
// and mean CTA load and the largest unit (in the scheduler's cost, key tiles
// + 1 per unit for prefill, key tiles for decode), and the host time from the
// call's entry to the finished list.
bool log_enabled() {
    static const bool on = [] {
        const char* e = std::getenv("OPATTN_LOG");
        return e != nullptr && e[0] != '\0' && !(e[0] == '0' && e[1] == '\0');
    }();
    return on;
}
using Clock = std::chrono::steady_clock;
double us_since(Clock::time_point t0) {
    return std::chrono::duration<double, std::micro>(Clock::now() - t0).count();
}
template <class U, class CostFn>
void log_schedule(const char* what, const std::vector<U>& units, const std::vector<int32_t>& cta_off, CostFn cost,
                  double host_us, const char* extra = "") {
    if (!log_enabled()) return;
    const size_t n_cta = cta_off.empty() ? 0 : cta_off.size() - 1;
    int64_t total = 0, max_load = 0, max_unit = 0;
    for (size_t c = 0; c < n_cta; ++c) {
        int64_t load = 0;
        for (int32_t i = cta_off[c]; i < cta_off[c + 1]; ++i) {
            const int64_t u = cost(units[static_cast<size_t>(i)]);
            load += u;
            max_unit = std::max(max_unit, u);
        }
        total += load;
        max_load = std::max(max_load, load);
    }
    std::fprintf(stderr,
                 "opattn: %s: %zu units on %zu CTAs; CTA load max %lld mean %.1f (max/mean %.3f); largest unit %lld;"
                 "%s host %.1f us\n",
                 what, units.size(), n_cta, static_cast<long long>(max_load),
                 n_cta ? static_cast<double>(total) / static_cast<double>(n_cta) : 0.0,
                 total > 0 ? static_cast<double>(max_load) * static_cast<double>(n_cta) / static_cast<double>(total) : 0.0,
                 static_cast<long long>(max_unit), extra, host_us);
}
int64_t prefill_cost(const UnitRec& u) { return u.n_tiles + 1; }

// ---------------------------------------------------- pinned staging pool
// The work list is built in mapped pinned memory and read from there by the
// upload kernel (opattn_upload.cu); a staging buffer is reused only after
// the event recorded behind that read has completed.  Where the memory
// cannot be mapped, an asynchronous copy moves it instead.  The pool grows
// while every buffer is in flight, up to kMaxStaging buffers; beyond that a
// call waits for the upload of the oldest buffer (the host is then that many
// calls ahead of the GPU) instead of pinning more memory.  A call needing a
// larger buffer than any free one still gets a new one.
struct Staging {
    void* host = nullptr;
    void* dev = nullptr;  // device address of the mapped buffer, or null
    size_t cap = 0;
    cudaEvent_t done = nullptr;
    bool busy = false;
    uint64_t seq = 0;     // release order: the smallest is the oldest upload
};
constexpr size_t kMaxStaging = 32;
std::mutex g_stage_mu;
std::vector<Staging*> g_stage_pool;
uint64_t g_stage_seq = 0;

Staging* staging_acquire(size_t bytes) {
    Staging* oldest = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_stage_mu);
        for (Staging* s : g_stage_pool) {
            if (s->busy || s->cap < bytes) continue;
            if (cudaEventQuery(s->done) == cudaSuccess) {
                s->busy = true;
                return s;
            }
            (void)cudaGetLastError();  // cudaErrorNotReady is not an error here
            if (!oldest || s->seq < oldest->seq) oldest = s;
        }
        if (oldest && g_stage_pool.size() >= kMaxStaging)
            oldest->busy = true;
        else
            oldest = nullptr;
    }
    if (oldest) {
        if (cudaEventSynchronize(oldest->done) != cudaSuccess) (void)cudaGetLastError();
        return oldest;
    }
    Staging* s = new Staging;
    size_t cap = 4096;
    while (cap < bytes) cap *= 2;
    if (cudaHostAlloc(&s->host, cap, cudaHostAllocPortable | cudaHostAllocMapped) == cudaSuccess) {
        if (cudaHostGetDevicePointer(&s->dev, s->host, 0) != cudaSuccess) {
            (void)cudaGetLastError();
            s->dev = nullptr;
        }
    } else {
        (void)cudaGetLastError();
        if (cudaHostAlloc(&s->host, cap, cudaHostAllocPortable) != cudaSuccess) {
            delete s;
            return nullptr;
        }
    }
    if (cudaEventCreateWithFlags(&s->done, cudaEventDisableTiming) != cudaSuccess) {
        cudaFreeHost(s->host);
        delete s;
        return nullptr;
    }
    s->cap = cap;
    s->busy = true;
    std::lock_guard<std::mutex> lk(g_stage_mu);
    g_stage_pool.push_back(s);
    return s;
}
void staging_release(Staging* s, cudaStream_t stream) {
    std::lock_guard<std::mutex> lk(g_stage_mu);
    cudaEventRecord(s->done, stream);
    s->seq = ++g_stage_seq;
    s->busy = false;
}
// Moves the first `bytes` of a staged work list to `dst` and zeroes the
// `zero_bytes` at `zero` (a multiple of 4), in stream order on `stream`.
bool upload_staged(const Staging* s, void* dst, size_t bytes, void* zero, size_t zero_bytes, cudaStream_t stream) {
    if (s->dev)
        return launch_upload(s->dev, dst, bytes, static_cast<int32_t*>(zero), zero_bytes / sizeof(int32_t),
                             stream) == 0;
    return cudaMemcpyAsync(dst, s->host, bytes, cudaMemcpyHostToDevice, stream) == cudaSuccess &&
           cudaMemsetAsync(zero, 0, zero_bytes, stream) == cudaSuccess;
}

// Stream-ordered scratch of the one-shot calls comes from a memory pool the
// library creates per device.  It keeps up to kPoolKeepBytes of freed scratch
// mapped across synchronizations, where the device's default pool (release
// threshold 0 unless its owner raises it) hands freed memory back to the
// system at every synchronization and maps it again on the next call.  If
// the pool cannot be created the default pool serves the calls.
constexpr uint64_t kPoolKeepBytes = 64ull << 20;
constexpr int kMaxPoolDevices = 64;

cudaMemPool_t scratch_pool() {
    static std::mutex mu;
    static cudaMemPool_t pools[kMaxPoolDevices] = {};
    static bool tried[kMaxPoolDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxPoolDevices) {
        (void)cudaGetLastError();
        return nullptr;
    }
    std::lock_guard<std::mutex> lk(mu);
    if (!tried[dev]) {
        tried[dev] = true;
        cudaMemPoolProps props;
        std::memset(&props, 0, sizeof props);
        props.allocType = cudaMemAllocationTypePinned;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        cudaMemPool_t pool = nullptr;
        if (cudaMemPoolCreate(&pool, &props) == cudaSuccess) {
            uint64_t keep = kPoolKeepBytes;
            if (cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep) == cudaSuccess) {
                pools[dev] = pool;
            } else {
                cudaMemPoolDestroy(pool);
            }
        }
        (void)cudaGetLastError();
    }
    return pools[dev];
}

// cudaMallocAsync from the library's pool (or the default pool).
cudaError_t scratch_alloc(void** ptr, size_t bytes, cudaStream_t stream) {
    cudaMemPool_t pool = scratch_pool();
    return pool ? cudaMallocFromPoolAsync(ptr, bytes, pool, stream) : cudaMallocAsync(ptr, bytes, stream);
}

int device_sm_count() {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    return sms;
}

LaunchArgs make_args(const void* q, const void* k, const void* v, void* o, float* lse, const Geometry& g,
                     float scale, const uint8_t* work, const WorkLayout& w, const Schedule& sch, uint32_t flags) {
    const int32_t n_cta = sch.n_cta;
    LaunchArgs a;
    a.q = q;
    a.k = k;
    a.v = v;
    a.o = o;
    a.lse = lse;
    a.total_q = g.total_q;
    a.total_k = g.total_k;
    a.Hq = g.Hq;
    a.Hkv = g.Hkv;
    a.d = g.d;
    a.scale = scale;
    a.units = reinterpret_cast<const UnitRec*>(work + w.off_units);
    a.cta_off = reinterpret_cast<const int32_t*>(work);
    a.n_cta = n_cta;
    a.status = reinterpret_cast<int32_t*>(const_cast<uint8_t*>(work) + w.off_status);
    a.flags = flags;
    if (sch.n_groups > 0) {
        uint8_t* wb = const_cast<uint8_t*>(work);
        a.counters = reinterpret_cast<unsigned long long*>(wb + w.off_counters);
        a.run = reinterpret_cast<RunWords*>(wb + w.off_run);
        a.part_lse = reinterpret_cast<float*>(wb + w.off_part_lse);
        a.part_o = reinterpret_cast<float*>(wb + w.off_part_o);
    }
    return a;
}

// Paged caches: the packed offsets the scheduler works on are built from the
// per-sequence key counts; checks the paging arguments that need no device.
struct PagedGeometry {
    std::vector<int32_t> cu_k;
    int32_t block_size = 0, max_blocks = 0;
};
opattn_status check_paged(const int32_t* seqlens_k, int32_t n_seq, int32_t block_size, int32_t max_blocks,
                          PagedGeometry* pg) {
    if (n_seq < 0) return OPATTN_ERR_INVALID_ARG;
    if (n_seq > 0 && !seqlens_k) return OPATTN_ERR_INVALID_ARG;
    if (block_size < 8 || block_size > kBlockN || (block_size & (block_size - 1)) != 0) return OPATTN_ERR_UNSUPPORTED;
    if (max_blocks < 1) return OPATTN_ERR_INVALID_ARG;
    pg->cu_k.assign(static_cast<size_t>(n_seq) + 1, 0);
    int64_t acc = 0;
    for (int32_t s = 0; s < n_seq; ++s) {
        const int32_t lk = seqlens_k[s];
        if (lk < 0) return OPATTN_ERR_INVALID_ARG;
        if ((static_cast<int64_t>(lk) + block_size - 1) / block_size > max_blocks) return OPATTN_ERR_INVALID_ARG;
        acc += lk;
        if (acc >= (int64_t{1} << 31)) return OPATTN_ERR_UNSUPPORTED;
        pg->cu_k[static_cast<size_t>(s) + 1] = static_cast<int32_t>(acc);
    }
    pg->block_size = block_size;
    pg->max_blocks = max_blocks;
    return OPATTN_OK;
}
opattn_status check_paged_tensors(const void* k_cache, const void* v_cache, const int32_t* block_table,
                                  int64_t num_blocks, const Geometry& g, int32_t block_size) {
    if (g.total_k == 0) return OPATTN_OK;
    if (!k_cache || !v_cache || !block_table || num_blocks < 1) return OPATTN_ERR_INVALID_ARG;
    if (!aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(block_table, 4)) return OPATTN_ERR_MISALIGNED;
    if (num_blocks * block_size * static_cast<int64_t>(g.Hkv) >= (int64_t{1} << 31)) return OPATTN_ERR_UNSUPPORTED;
    return OPATTN_OK;
}

struct PagedArgs {
    const int32_t* block_table = nullptr;
    int64_t num_blocks = 0;
    int32_t block_size = 0, max_blocks = 0;
};

// One-shot path shared by opattn_prefill and opattn_prefill_checked.
opattn_status prefill_impl(const void* q, const void* k, const void* v, void* o, float* lse, const int32_t* cu_q,
                           const int32_t* cu_k, int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                           cudaStream_t stream, uint32_t flags, bool checked, const PagedArgs* paged = nullptr) {
    const Clock::time_point t_entry = Clock::now();
    Geometry g;
    opattn_status st = check_geometry(cu_q, cu_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    if (g.total_q == 0) return OPATTN_OK;
    if (paged) {
        Geometry gq = g;
        gq.total_k = 0;  // k/v are checked as caches below
        st = check_tensors(q, nullptr, nullptr, o, lse, scale, gq);
        if (st == OPATTN_OK)
            st = check_paged_tensors(k, v, paged->block_table, paged->num_blocks, g, paged->block_size);
    } else {
        st = check_tensors(q, k, v, o, lse, scale, g);
    }
    if (st != OPATTN_OK) return st;
    const int sms = device_sm_count();
    if (sms <= 0) return OPATTN_ERR_CUDA;

    // Reused by the thread's next call: the list is copied into the staging
    // buffer below before this call returns.
    thread_local Schedule sch;
    build_schedule(cu_q, cu_k, g, sms, &sch);
    log_schedule("prefill", sch.units, sch.cta_off, prefill_cost, us_since(t_entry));
    const WorkLayout w = work_layout(sch, g.d);
    Staging* stg = staging_acquire(w.upload_bytes);
    if (!stg) return OPATTN_ERR_CUDA;
    pack_upload(sch, w, static_cast<uint8_t*>(stg->host));

    void* work = nullptr;
    if (scratch_alloc(&work, w.bytes, stream) != cudaSuccess) {
        staging_release(stg, stream);
        return OPATTN_ERR_CUDA;
    }
    bool ok = upload_staged(stg, work, w.upload_bytes, static_cast<uint8_t*>(work) + w.off_counters, w.zero_bytes,
                            stream);
    staging_release(stg, stream);
    int32_t dev_status = 0;
    if (ok) {
        LaunchArgs a = make_args(q, k, v, o, lse, g, scale, static_cast<uint8_t*>(work), w, sch, flags);
        if (paged) {
            a.block_table = paged->block_table;
            a.max_blocks = paged->max_blocks;
            a.block_size = paged->block_size;
            a.num_blocks = paged->num_blocks;
        }
        ok = launch_prefill(a, stream) == 0;
    }
    if (ok && checked) {
        ok = cudaMemcpyAsync(&dev_status, static_cast<uint8_t*>(work) + w.off_status, sizeof(int32_t),
                             cudaMemcpyDeviceToHost, stream) == cudaSuccess;
        ok = ok && cudaStreamSynchronize(stream) == cudaSuccess;
    }
    cudaFreeAsync(work, stream);
    if (!ok) return OPATTN_ERR_CUDA;
    if (checked && dev_status != kDevOk) return OPATTN_ERR_TIMEOUT;
    return OPATTN_OK;
}

static_assert(kNoAllocMaxUnits == OPATTN_NOALLOC_MAX_UNITS, "opattn.h and the scratch size disagree");

// Work units of a batch without building the schedule (same enumeration
// as build_schedule).
int64_t count_units(const int32_t* cu_q, const Geometry& g) {
    const int64_t tpu = 2 * g.TPB;
    int64_t n = 0;
    for (int32_t s = 0; s < g.n_seq; ++s) n += (static_cast<int64_t>(cu_q[s + 1] - cu_q[s]) + tpu - 1) / tpu;
    return n * g.Hkv;
}

// Same computation as prefill_impl with the work list in the library's
// fixed device array: nothing is allocated on the device.
opattn_status prefill_noalloc_impl(const void* q, const void* k, const void* v, void* o, float* lse,
                                   const int32_t* cu_q, const int32_t* cu_k, int32_t n_seq, int32_t Hq,
                                   int32_t Hkv, int32_t d, float scale, cudaStream_t stream) {
    const Clock::time_point t_entry = Clock::now();
    Geometry g;
    opattn_status st = check_geometry(cu_q, cu_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    if (g.total_q == 0) return OPATTN_OK;
    st = check_tensors(q, k, v, o, lse, scale, g);
    if (st != OPATTN_OK) return st;
    if (count_units(cu_q, g) > kNoAllocMaxUnits) return OPATTN_ERR_CAPACITY;
    // The list is copied from heap memory freed on return, which a captured
    // graph could not replay.
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const cudaError_t ce = cudaStreamIsCapturing(stream, &cs);
    if (ce != cudaSuccess) {
        (void)cudaGetLastError();
        return ce == cudaErrorStreamCaptureImplicit ? OPATTN_ERR_INVALID_ARG : OPATTN_ERR_CUDA;
    }
    if (cs != cudaStreamCaptureStatusNone) return OPATTN_ERR_INVALID_ARG;
    const int sms = device_sm_count();
    if (sms <= 0) return OPATTN_ERR_CUDA;

    Schedule sch;
    // No split-KV here: the fixed array has no room for the pieces' partials.
    build_schedule(cu_q, cu_k, g, std::min(sms, kNoAllocMaxCtas), &sch, /*allow_split=*/false);
    log_schedule("prefill (no-alloc)", sch.units, sch.cta_off, prefill_cost, us_since(t_entry));
    const WorkLayout w = work_layout(sch, g.d);
    void* scratch = nullptr;
    size_t scratch_bytes = 0;
    if (noalloc_scratch(&scratch, &scratch_bytes) != 0) return OPATTN_ERR_CUDA;
    if (w.bytes > scratch_bytes) return OPATTN_ERR_CAPACITY;
    // The list is copied from ordinary (pageable) host memory: the runtime
    // stages it before cudaMemcpyAsync returns, so the vector may go away.
    std::vector<uint8_t> host(w.upload_bytes);
    pack_upload(sch, w, host.data());
    uint8_t* work = static_cast<uint8_t*>(scratch);
    if (cudaMemcpyAsync(work, host.data(), w.upload_bytes, cudaMemcpyHostToDevice, stream) != cudaSuccess)
        return OPATTN_ERR_CUDA;
    // The array keeps the previous call's contents: the status word must
    // start at zero.
    if (cudaMemsetAsync(work + w.off_status, 0, sizeof(int32_t), stream) != cudaSuccess) return OPATTN_ERR_CUDA;
    const LaunchArgs a = make_args(q, k, v, o, lse, g, scale, work, w, sch, 0u);
    return launch_prefill(a, stream) == 0 ? OPATTN_OK : OPATTN_ERR_CUDA;
}

// ------------------------------------------------------------------ decode

// Additional checks of the decode kernel: d = 128, G divides kDecCols, and
// every sequence's G * Lq query (token, head) pairs fit the kDecCols columns.
opattn_status check_decode_geometry(const int32_t* cu_q, const Geometry& g) {
    if (g.d != kDecHeadDim) return OPATTN_ERR_UNSUPPORTED;
    if (kDecCols % g.G != 0) return OPATTN_ERR_UNSUPPORTED;
    for (int32_t s = 0; s < g.n_seq; ++s)
        if (static_cast<int64_t>(cu_q[s + 1] - cu_q[s]) * g.G > kDecCols) return OPATTN_ERR_UNSUPPORTED;
    return OPATTN_OK;
}

struct DecodeSchedule {
    std::vector<DecUnit> units;    // grouped by CTA, in pair order within a CTA, then zero-tile units
    std::vector<int32_t> cta_off;  // n_cta + 1
    int32_t n_cta = 0;
    int32_t n_groups = 0;          // split (sequence, kv head) pairs: one merge counter each
    int32_t n_parts = 0;           // partial (O, LSE) slots
    int32_t chunk_tiles = 0;       // key tiles per CTA (rounded up)
    int32_t max_cols = 0;          // largest G * Lq over the batch
};

struct DecPair {
    int32_t s, h, n_t;  // sequence, kv head, key tiles
};

// Appends pair `pr` cut into `pieces` (CTA, first tile, tiles) to the per-CTA
// unit lists; a pair in several pieces gets a merge counter and contiguous
// partial slots.
void add_pair_units(const DecPair& pr, const std::vector<std::array<int64_t, 3>>& pieces, const int32_t* cu_q,
                    const int32_t* cu_k, DecodeSchedule* out, std::vector<std::vector<DecUnit>>* per_cta) {
    const int32_t n_chunks = static_cast<int32_t>(pieces.size());
    const int32_t group = n_chunks > 1 ? out->n_groups++ : -1;
    const int32_t part0 = n_chunks > 1 ? out->n_parts : -1;
    if (n_chunks > 1) out->n_parts += n_chunks;
    for (int32_t i = 0; i < n_chunks; ++i) {
        DecUnit u;
        u.q_tok0 = cu_q[pr.s];
        u.nq = cu_q[pr.s + 1] - cu_q[pr.s];
        u.k_row0 = cu_k[pr.s];
        u.Lk = cu_k[pr.s + 1] - cu_k[pr.s];
        u.kvh = pr.h;
        u.tile0 = static_cast<int32_t>(pieces[static_cast<size_t>(i)][1]);
        u.n_tiles = static_cast<int32_t>(pieces[static_cast<size_t>(i)][2]);
        u.part = n_chunks > 1 ? part0 + i : -1;
        u.group = group;
        u.chunk = i;
        u.n_chunks = n_chunks;
        u.seq = pr.s;
        (*per_cta)[static_cast<size_t>(pieces[static_cast<size_t>(i)][0])].push_back(u);
    }
}

// Stream-K cut: the key tiles of all pairs, taken in order, are cut into
// n_cta equal stretches, one per CTA, so every CTA streams the same number of
// tiles to within one; a pair whose tiles fall into several stretches is
// split into chunks there.
void stream_k_cut(const std::vector<DecPair>& pairs, int64_t total_tiles, int32_t n_cta, const int32_t* cu_q,
                  const int32_t* cu_k, DecodeSchedule* out, std::vector<std::vector<DecUnit>>* per_cta) {
    auto bound = [&](int64_t c) { return c * total_tiles / n_cta; };  // first tile of CTA c's stretch
    int64_t pos = 0;  // global index of the pair's first tile
    for (const DecPair& pr : pairs) {
        if (pr.n_t == 0) continue;
        // CTAs whose stretch meets [pos, pos + n_t)
        int64_t c = std::min<int64_t>(n_cta - 1, pos * n_cta / total_tiles);
        while (c > 0 && bound(c) > pos) --c;
        while (c + 1 < n_cta && bound(c + 1) <= pos) ++c;
        std::vector<std::array<int64_t, 3>> pieces;
        int64_t t = pos;
        const int64_t end = pos + pr.n_t;
        while (t < end) {
            const int64_t stop = std::min<int64_t>(end, bound(c + 1));
            if (stop > t) pieces.push_back({c, t - pos, stop - t});
            t = stop;
            ++c;
        }
        add_pair_units(pr, pieces, cu_q, cu_k, out, per_cta);
        pos = end;
    }
}

// Pair-aligned cut, for at most n_cta pairs with keys: the smallest chunk
// size M such that sum_p ceil(t_p / M) chunks fit the grid; pair p is cut
// into ceil(t_p / M) nearly equal chunks, one CTA each.  Every CTA then holds
// one chunk, where a stream-K stretch can hold the end of one split pair and
// the start of the next.  Returns the CTAs used.
int32_t pair_aligned_cut(const std::vector<DecPair>& pairs, int32_t n_cta, const int32_t* cu_q, const int32_t* cu_k,
                         DecodeSchedule* out, std::vector<std::vector<DecUnit>>* per_cta) {
    int32_t hi = 1;
    for (const DecPair& pr : pairs) hi = std::max(hi, pr.n_t);
    auto need = [&](int32_t m) {
        int64_t n = 0;
        for (const DecPair& pr : pairs) n += (pr.n_t + m - 1) / m;
        return n;
    };
    int32_t lo = 1;  // smallest m with need(m) <= n_cta; need(hi) = pairs with keys <= n_cta
    while (lo < hi) {
        const int32_t mid = lo + (hi - lo) / 2;
        if (need(mid) <= n_cta) hi = mid; else lo = mid + 1;
    }
    per_cta->assign(static_cast<size_t>(need(lo)), {});
    int64_t c = 0;
    for (const DecPair& pr : pairs) {
        if (pr.n_t == 0) continue;
        const int32_t k = (pr.n_t + lo - 1) / lo;
        std::vector<std::array<int64_t, 3>> pieces;
        for (int32_t i = 0; i < k; ++i) {
            const int64_t t0 = static_cast<int64_t>(pr.n_t) * i / k;
            const int64_t t1 = static_cast<int64_t>(pr.n_t) * (i + 1) / k;
            pieces.push_back({c++, t0, t1 - t0});
        }
        add_pair_units(pr, pieces, cu_q, cu_k, out, per_cta);
    }
    return static_cast<int32_t>(per_cta->size());
}

// Model of a decode launch's time, in key-tile times, from its per-CTA unit
// lists (fitted to plan-run latencies of small batches on GB300: ~0.8 us per
// key tile of a CTA's chain, ~3.8 us per extra unit in the chain; HBM is
// saturated by about 96 CTAs streaming at once).
double decode_schedule_cost(const std::vector<std::vector<DecUnit>>& per_cta, int64_t total_tiles) {
    int64_t max_tiles = 0, max_units = 0;
    bool split = false;
    for (const auto& us : per_cta) {
        int64_t t = 0, n = 0;
        for (const DecUnit& u : us) {
            if (u.n_tiles <= 0) continue;
            t += u.n_tiles;
            ++n;
            split = split || u.n_chunks > 1;
        }
        max_tiles = std::max(max_tiles, t);
        max_units = std::max(max_units, n);
    }
    return std::max(static_cast<double>(total_tiles) / 96.0, static_cast<double>(max_tiles)) + 5.0 * max_units +
           (split ? 2.0 : 0.0);
}

// Units are (sequence, kv head, range of key tiles); a pair split into chunks
// is merged later by the last chunk to finish.  The default cut is stream-K
// (stream_k_cut).  With fit_grid (the default grid of a one-shot call or a
// plan without an SM budget) a uniform batch takes a grid that splits no
// pair, and a batch with no more pairs than CTAs takes the pair-aligned cut
// (pair_aligned_cut) when the cost model says it is faster.  Pairs with no
// keys become zero-tile units spread over the CTAs.
void build_decode_schedule(const int32_t* cu_q, const int32_t* cu_k, const Geometry& g, int32_t max_ctas,
                           DecodeSchedule* out, bool fit_grid = false) {
    std::vector<DecPair> pairs;
    int64_t total_tiles = 0;
    int64_t n_pairs = 0;  // pairs with keys
    for (int32_t s = 0; s < g.n_seq; ++s) {
        if (cu_q[s + 1] == cu_q[s]) continue;
        const int32_t n_t = (cu_k[s + 1] - cu_k[s] + kBlockN - 1) / kBlockN;
        for (int32_t h = 0; h < g.Hkv; ++h) pairs.push_back({s, h, n_t});
        total_tiles += static_cast<int64_t>(n_t) * g.Hkv;
        if (n_t > 0) n_pairs += g.Hkv;
    }
    out->units.clear();
    out->cta_off.clear();
    out->n_cta = 0;
    out->n_groups = 0;
    out->n_parts = 0;
    int32_t max_cols = 1;
    for (int32_t s = 0; s < g.n_seq; ++s) max_cols = std::max(max_cols, (cu_q[s + 1] - cu_q[s]) * g.G);
    out->max_cols = max_cols;
    if (pairs.empty()) return;
    const int32_t cap = std::max<int32_t>(max_ctas, 1);
    int32_t n_sk = cap;
    // When every (sequence, kv head) pair has the same number of key tiles,
    // a grid of n CTAs splits no pair if n divides the pair count, and splits
    // every pair into equal chunks if the pair count divides n (and n / pairs
    // divides a pair's tiles).  A split pair costs its chunks a partial write
    // and its last chunk a merge (2-9% of such batches, measured), so with
    // fit_grid the largest such grid down to 4/5 of the cap is taken.
    if (fit_grid && cap > 1) {
        int32_t tp = -1;
        bool uniform = true;
        for (const DecPair& pr : pairs) {
            if (pr.n_t == 0) continue;
            if (tp < 0) tp = pr.n_t;
            uniform = uniform && pr.n_t == tp;
        }
        if (uniform && n_pairs > 0) {
            const int32_t lo = (cap * 4 + 4) / 5;
            for (int32_t n = cap; n >= lo; --n) {
                const bool whole = n_pairs % n == 0;
                const bool equal = n % n_pairs == 0 && tp % (n / n_pairs) == 0;
                if (whole || equal) {
                    n_sk = n;
                    break;
                }
            }
        }
    }
    n_sk = static_cast<int32_t>(std::max<int64_t>(1, std::min<int64_t>(n_sk, std::max<int64_t>(total_tiles, 1))));
    std::vector<std::vector<DecUnit>> per_cta(static_cast<size_t>(n_sk));
    DecodeSchedule sk = *out;
    if (total_tiles > 0) stream_k_cut(pairs, total_tiles, n_sk, cu_q, cu_k, &sk, &per_cta);
    if (fit_grid && n_pairs > 0 && n_pairs <= cap) {
        std::vector<std::vector<DecUnit>> pa_cta;
        DecodeSchedule pa = *out;
        pair_aligned_cut(pairs, cap, cu_q, cu_k, &pa, &pa_cta);
        if (decode_schedule_cost(pa_cta, total_tiles) <= decode_schedule_cost(per_cta, total_tiles)) {
            per_cta.swap(pa_cta);
            sk = pa;
        }
    }
    out->n_groups = sk.n_groups;
    out->n_parts = sk.n_parts;
    const int32_t n_cta = static_cast<int32_t>(per_cta.size());
    int32_t zero_rr = 0;
    for (const DecPair& pr : pairs) {
        if (pr.n_t != 0) continue;
        add_pair_units(pr, {{zero_rr, 0, 0}}, cu_q, cu_k, out, &per_cta);
        zero_rr = (zero_rr + 1) % n_cta;
    }
    out->cta_off.assign(static_cast<size_t>(n_cta) + 1, 0);
    for (int32_t c = 0; c < n_cta; ++c) {
        out->cta_off[static_cast<size_t>(c) + 1] =
            out->cta_off[static_cast<size_t>(c)] + static_cast<int32_t>(per_cta[static_cast<size_t>(c)].size());
        out->units.insert(out->units.end(), per_cta[static_cast<size_t>(c)].begin(), per_cta[static_cast<size_t>(c)].end());
    }
    out->n_cta = n_cta;
    out->chunk_tiles = static_cast<int32_t>((total_tiles + n_cta - 1) / n_cta);
}

// Device work area: [cta_off | pad 32 | units | counters (2 per group: one per
// softmax warpgroup, 8 bytes each) | run words (epoch, exits) | status | pad 256 |
// part_lse (n_parts x kDecCols) | part_o (n_parts x kDecCols x d)].  The
// counters, the run words and the status word are contiguous.  One-shot calls
// zero them with the work-list upload; a plan zeroes them once when it is
// created.  Counters are tagged with the launch epoch, which the kernel
// advances itself (RunWords), so plan runs need no memset, and a run that
// stopped early leaves no count that a later run would take for its own.
struct DecodeLayout {
    size_t off_units, off_counters, off_run, off_status, off_part_lse, off_part_o, bytes, upload_bytes, zero_bytes;
};
DecodeLayout decode_layout(const DecodeSchedule& s) {
    DecodeLayout w;
    w.off_units = (s.cta_off.size() * sizeof(int32_t) + 31) / 32 * 32;
    w.off_counters = w.off_units + s.units.size() * sizeof(DecUnit);  // a multiple of 16
    w.off_run = w.off_counters + 2 * static_cast<size_t>(s.n_groups) * sizeof(unsigned long long);
    w.off_status = w.off_run + sizeof(RunWords);
    w.upload_bytes = w.off_counters;
    w.zero_bytes = w.off_status + sizeof(int32_t) - w.off_counters;
    w.off_part_lse = (w.off_status + sizeof(int32_t) + 255) / 256 * 256;
    w.off_part_o = w.off_part_lse + (static_cast<size_t>(s.n_parts) * kDecCols * sizeof(float) + 255) / 256 * 256;
    w.bytes = w.off_part_o + static_cast<size_t>(s.n_parts) * kDecCols * kDecHeadDim * sizeof(float);
    return w;
}
void pack_decode_upload(const DecodeSchedule& s, const DecodeLayout& w, uint8_t* dst) {
    const size_t off_bytes = s.cta_off.size() * sizeof(int32_t);
    const size_t end_units = w.off_units + s.units.size() * sizeof(DecUnit);
    std::memcpy(dst, s.cta_off.data(), off_bytes);
    std::memset(dst + off_bytes, 0, w.off_units - off_bytes);
    std::memcpy(dst + w.off_units, s.units.data(), s.units.size() * sizeof(DecUnit));
    std::memset(dst + end_units, 0, w.upload_bytes - end_units);
}
DecodeLaunchArgs make_decode_args(const void* q, const void* k, const void* v, void* o, float* lse,
                                  const Geometry& g, float scale, uint8_t* work, const DecodeLayout& w,
                                  int32_t n_cta, int32_t max_cols, uint32_t flags) {
    DecodeLaunchArgs a;
    a.q = q;
    a.k = k;
    a.v = v;
    a.o = o;
    a.lse = lse;
    a.total_q = g.total_q;
    a.total_k = g.total_k;
    a.Hq = g.Hq;
    a.Hkv = g.Hkv;
    a.scale = scale;
    a.units = reinterpret_cast<const DecUnit*>(work + w.off_units);
    a.cta_off = reinterpret_cast<const int32_t*>(work);
    a.n_cta = n_cta;
    a.max_cols = max_cols;
    a.counters = reinterpret_cast<unsigned long long*>(work + w.off_counters);
    a.run = reinterpret_cast<RunWords*>(work + w.off_run);
    a.part_lse = reinterpret_cast<float*>(work + w.off_part_lse);
    a.part_o = reinterpret_cast<float*>(work + w.off_part_o);
    a.status = reinterpret_cast<int32_t*>(work + w.off_status);
    a.flags = flags;
    a.block_table = nullptr;
    a.max_blocks = 0;
    a.block_size = 0;
    a.num_blocks = 0;
    return a;
}

void log_decode_schedule(const char* what, const DecodeSchedule& s, double host_us) {
    if (!log_enabled()) return;
    char extra[96];
    std::snprintf(extra, sizeof extra, " %d split pairs, %d partials;", s.n_groups, s.n_parts);
    log_schedule(what, s.units, s.cta_off, [](const DecUnit& u) { return static_cast<int64_t>(u.n_tiles); }, host_us,
                 extra);
}

opattn_status decode_impl(const void* q, const void* k, const void* v, void* o, float* lse, const int32_t* cu_q,
                          const int32_t* cu_k, int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, float scale,
                          cudaStream_t stream, uint32_t flags, bool checked, const PagedArgs* paged = nullptr) {
    const Clock::time_point t_entry = Clock::now();
    Geometry g;
    opattn_status st = check_geometry(cu_q, cu_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    st = check_decode_geometry(cu_q, g);
    if (st != OPATTN_OK) return st;
    if (g.total_q == 0) return OPATTN_OK;
    if (paged) {
        Geometry gq = g;
        gq.total_k = 0;  // k/v are checked as caches below
        st = check_tensors(q, nullptr, nullptr, o, lse, scale, gq);
        if (st == OPATTN_OK)
            st = check_paged_tensors(k, v, paged->block_table, paged->num_blocks, g, paged->block_size);
    } else {
        st = check_tensors(q, k, v, o, lse, scale, g);
    }
    if (st != OPATTN_OK) return st;
    const int sms = device_sm_count();
    if (sms <= 0) return OPATTN_ERR_CUDA;

    DecodeSchedule sch;
    build_decode_schedule(cu_q, cu_k, g, sms, &sch, /*fit_grid=*/true);
    log_decode_schedule("decode", sch, us_since(t_entry));
    const DecodeLayout w = decode_layout(sch);
    Staging* stg = staging_acquire(w.upload_bytes);
    if (!stg) return OPATTN_ERR_CUDA;
    pack_decode_upload(sch, w, static_cast<uint8_t*>(stg->host));
    void* work = nullptr;
    if (scratch_alloc(&work, w.bytes, stream) != cudaSuccess) {
        staging_release(stg, stream);
        return OPATTN_ERR_CUDA;
    }
    uint8_t* wb = static_cast<uint8_t*>(work);
    bool ok = upload_staged(stg, wb, w.upload_bytes, wb + w.off_counters, w.zero_bytes, stream);
    staging_release(stg, stream);
    int32_t dev_status = 0;
    if (ok) {
        DecodeLaunchArgs a = make_decode_args(q, k, v, o, lse, g, scale, wb, w, sch.n_cta, sch.max_cols, flags);
        if (paged) {
            a.block_table = paged->block_table;
            a.max_blocks = paged->max_blocks;
            a.block_size = paged->block_size;
            a.num_blocks = paged->num_blocks;
        }
        ok = launch_decode(a, stream) == 0;
    }
    if (ok && checked) {
        ok = cudaMemcpyAsync(&dev_status, wb + w.off_status, sizeof(int32_t), cudaMemcpyDeviceToHost, stream) ==
             cudaSuccess;
        ok = ok && cudaStreamSynchronize(stream) == cudaSuccess;
    }
    cudaFreeAsync(work, stream);
    if (!ok) return OPATTN_ERR_CUDA;
    if (checked && dev_status != kDevOk) return OPATTN_ERR_TIMEOUT;
    return OPATTN_OK;
}

}  // namespace
}  // namespace opattn

using namespace opattn;

struct opattn_plan {
    Geometry g;
    bool decode = false;
    Schedule sch;          // prefill plans
    WorkLayout w;
    DecodeSchedule dsch;   // decode plans
    DecodeLayout dw;
    int32_t block_size = 0;  // paged decode plans (0: packed K/V)
    int32_t max_blocks = 0;
    int device = 0;
    void* work = nullptr;
};

extern "C" {

int32_t opattn_version(void) { return kVersion; }

const char* opattn_status_string(int32_t status) {
    switch (status) {
        case OPATTN_OK: return "ok";
        case OPATTN_ERR_INVALID_ARG: return "invalid argument";
        case OPATTN_ERR_UNSUPPORTED:
            return "unsupported configuration (prefill: head dim 64 or 128, Hq/Hkv <= 128; decode: head dim 128, "
                   "Hq/Hkv divides 32, Lq * Hq/Hkv <= 32 per sequence)";
        case OPATTN_ERR_MISALIGNED: return "misaligned pointer (q/k/v/o need 16 bytes, lse 4 bytes)";
        case OPATTN_ERR_CUDA: return "CUDA runtime error";
        case OPATTN_ERR_TIMEOUT: return "device wait timed out";
        case OPATTN_ERR_CAPACITY: return "output array too small";
        default: return "unknown status";
    }
}

opattn_status opattn_prefill(const void* q, const void* k, const void* v, void* o, float* lse,
                             const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq, int32_t Hq,
                             int32_t Hkv, int32_t d, float scale, void* stream) {
    return prefill_impl(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, scale,
                        static_cast<cudaStream_t>(stream), 0u, false);
}

opattn_status opattn_prefill_noalloc(const void* q, const void* k, const void* v, void* o, float* lse,
                                     const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq,
                                     int32_t Hq, int32_t Hkv, int32_t d, float scale, void* stream) {
    return prefill_noalloc_impl(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, scale,
                                static_cast<cudaStream_t>(stream));
}

opattn_status opattn_prefill_checked(const void* q, const void* k, const void* v, void* o, float* lse,
                                     const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq,
                                     int32_t Hq, int32_t Hkv, int32_t d, float scale, void* stream,
                                     uint32_t flags) {
    if (flags & ~(OPATTN_FLAG_TEST_FORCE_TIMEOUT | OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA))
        return OPATTN_ERR_INVALID_ARG;
    const uint32_t kflags = ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT) ? kFlagForceTimeout : 0u) |
                            ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA) ? kFlagForceTimeoutFirstCta : 0u);
    return prefill_impl(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, scale,
                        static_cast<cudaStream_t>(stream), kflags, true);
}

opattn_status opattn_plan_create(opattn_plan** plan, const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k,
                                 int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, int32_t max_ctas) {
    if (!plan) return OPATTN_ERR_INVALID_ARG;
    *plan = nullptr;
    if (max_ctas < 0) return OPATTN_ERR_INVALID_ARG;
    Geometry g;
    opattn_status st = check_geometry(cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    opattn_plan* p = new opattn_plan;
    p->g = g;
    if (cudaGetDevice(&p->device) != cudaSuccess) {
        delete p;
        return OPATTN_ERR_CUDA;
    }
    if (g.total_q > 0) {
        const int sms = device_sm_count();
        if (sms <= 0) {
            delete p;
            return OPATTN_ERR_CUDA;
        }
        const int32_t cap = max_ctas > 0 ? std::min(max_ctas, sms) : sms;
        const Clock::time_point t0 = Clock::now();
        build_schedule(cu_seqlens_q, cu_seqlens_k, g, cap, &p->sch);
        log_schedule("prefill plan", p->sch.units, p->sch.cta_off, prefill_cost, us_since(t0));
        p->w = work_layout(p->sch, g.d);
        // the work list, then the counters, run words and status word at zero
        const size_t init_bytes = p->w.off_counters + p->w.zero_bytes;
        std::vector<uint8_t> host(init_bytes, 0);
        pack_upload(p->sch, p->w, host.data());
        if (cudaMalloc(&p->work, p->w.bytes) != cudaSuccess) {
            delete p;
            return OPATTN_ERR_CUDA;
        }
        if (cudaMemcpy(p->work, host.data(), init_bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
            cudaFree(p->work);
            delete p;
            return OPATTN_ERR_CUDA;
        }
    }
    *plan = p;
    return OPATTN_OK;
}

}  // extern "C"

namespace {
// Launch of a packed-K/V plan with kernel flags (0 for opattn_plan_run).
opattn_status plan_launch(const opattn_plan* plan, const void* q, const void* k, const void* v, void* o, float* lse,
                          float scale, cudaStream_t stream, uint32_t kflags) {
    opattn_status st = check_tensors(q, k, v, o, lse, scale, plan->g);
    if (st != OPATTN_OK) return st;
    if (plan->block_size > 0) return OPATTN_ERR_INVALID_ARG;  // paged plans run with opattn_plan_run_paged
    uint8_t* work = static_cast<uint8_t*>(plan->work);
    if (plan->decode) {
        const DecodeLaunchArgs a = make_decode_args(q, k, v, o, lse, plan->g, scale, work, plan->dw, plan->dsch.n_cta,
                                                    plan->dsch.max_cols, kflags);
        return launch_decode(a, stream) == 0 ? OPATTN_OK : OPATTN_ERR_CUDA;
    }
    const LaunchArgs a = make_args(q, k, v, o, lse, plan->g, scale, work, plan->w, plan->sch, kflags);
    return launch_prefill(a, stream) == 0 ? OPATTN_OK : OPATTN_ERR_CUDA;
}
}  // namespace

extern "C" {

opattn_status opattn_plan_run(const opattn_plan* plan, const void* q, const void* k, const void* v, void* o,
                              float* lse, float scale, void* stream) {
    if (!plan) return OPATTN_ERR_INVALID_ARG;
    if (plan->g.total_q == 0) return OPATTN_OK;
    return plan_launch(plan, q, k, v, o, lse, scale, static_cast<cudaStream_t>(stream), 0u);
}

opattn_status opattn_plan_run_checked(const opattn_plan* plan, const void* q, const void* k, const void* v, void* o,
                                      float* lse, float scale, void* stream, uint32_t flags) {
    if (!plan) return OPATTN_ERR_INVALID_ARG;
    if (flags & ~(OPATTN_FLAG_TEST_FORCE_TIMEOUT | OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA))
        return OPATTN_ERR_INVALID_ARG;
    if (plan->block_size > 0) return OPATTN_ERR_INVALID_ARG;
    if (plan->g.total_q == 0) return OPATTN_OK;
    const uint32_t kflags = ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT) ? kFlagForceTimeout : 0u) |
                            ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA) ? kFlagForceTimeoutFirstCta : 0u);
    const cudaStream_t st_ = static_cast<cudaStream_t>(stream);
    int32_t* status = reinterpret_cast<int32_t*>(static_cast<uint8_t*>(plan->work) +
                                                 (plan->decode ? plan->dw.off_status : plan->w.off_status));
    if (cudaMemsetAsync(status, 0, sizeof(int32_t), st_) != cudaSuccess) return OPATTN_ERR_CUDA;
    opattn_status st = plan_launch(plan, q, k, v, o, lse, scale, st_, kflags);
    if (st != OPATTN_OK) return st;
    int32_t dev_status = 0;
    if (cudaMemcpyAsync(&dev_status, status, sizeof(int32_t), cudaMemcpyDeviceToHost, st_) != cudaSuccess ||
        cudaStreamSynchronize(st_) != cudaSuccess)
        return OPATTN_ERR_CUDA;
    return dev_status == kDevOk ? OPATTN_OK : OPATTN_ERR_TIMEOUT;
}

opattn_status opattn_plan_destroy(opattn_plan* plan) {
    if (!plan) return OPATTN_OK;
    opattn_status st = OPATTN_OK;
    if (plan->work) {
        int prev = 0;
        cudaGetDevice(&prev);
        cudaSetDevice(plan->device);
        if (cudaDeviceSynchronize() != cudaSuccess) st = OPATTN_ERR_CUDA;
        if (cudaFree(plan->work) != cudaSuccess) st = OPATTN_ERR_CUDA;
        cudaSetDevice(prev);
    }
    delete plan;
    return st;
}

opattn_status opattn_plan_info(const opattn_plan* plan, int64_t* n_units, int32_t* n_ctas) {
    if (!plan) return OPATTN_ERR_INVALID_ARG;
    if (n_units) *n_units = static_cast<int64_t>(plan->decode ? plan->dsch.units.size() : plan->sch.units.size());
    if (n_ctas) *n_ctas = plan->decode ? plan->dsch.n_cta : plan->sch.n_cta;
    return OPATTN_OK;
}

opattn_status opattn_schedule(const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq, int32_t Hq,
                              int32_t Hkv, int32_t d, int32_t n_ctas, int32_t* units, int64_t unit_capacity,
                              int32_t* cta_offsets, int64_t* n_units_out, int32_t* n_ctas_used) {
    if (n_ctas <= 0 || !n_units_out || !n_ctas_used) return OPATTN_ERR_INVALID_ARG;
    Geometry g;
    opattn_status st = check_geometry(cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    thread_local Schedule sch;  // copied out below; reused by the thread's next call
    const Clock::time_point t0 = Clock::now();
    build_schedule(cu_seqlens_q, cu_seqlens_k, g, n_ctas, &sch);
    log_schedule("prefill schedule", sch.units, sch.cta_off, prefill_cost, us_since(t0));
    *n_units_out = static_cast<int64_t>(sch.units.size());
    *n_ctas_used = sch.n_cta;
    if (static_cast<int64_t>(sch.units.size()) > unit_capacity) return OPATTN_ERR_CAPACITY;
    if (!sch.units.empty() && (!units || !cta_offsets)) return OPATTN_ERR_INVALID_ARG;
    if (!sch.units.empty()) {
        std::memcpy(units, sch.units.data(), sch.units.size() * sizeof(UnitRec));
        std::memcpy(cta_offsets, sch.cta_off.data(), sch.cta_off.size() * sizeof(int32_t));
    }
    return OPATTN_OK;
}

opattn_status opattn_decode(const void* q, const void* k, const void* v, void* o, float* lse,
                            const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq, int32_t Hq,
                            int32_t Hkv, int32_t d, float scale, void* stream) {
    return decode_impl(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, scale,
                       static_cast<cudaStream_t>(stream), 0u, false);
}

opattn_status opattn_decode_checked(const void* q, const void* k, const void* v, void* o, float* lse,
                                    const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq,
                                    int32_t Hq, int32_t Hkv, int32_t d, float scale, void* stream, uint32_t flags) {
    if (flags & ~(OPATTN_FLAG_TEST_FORCE_TIMEOUT | OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA))
        return OPATTN_ERR_INVALID_ARG;
    const uint32_t kflags = ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT) ? kFlagForceTimeout : 0u) |
                            ((flags & OPATTN_FLAG_TEST_FORCE_TIMEOUT_FIRST_CTA) ? kFlagForceTimeoutFirstCta : 0u);
    return decode_impl(q, k, v, o, lse, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, scale,
                       static_cast<cudaStream_t>(stream), kflags, true);
}

}  // extern "C"

namespace {
opattn_status decode_plan_create(opattn_plan** plan, const int32_t* cu_q, const int32_t* cu_k, int32_t n_seq,
                                 int32_t Hq, int32_t Hkv, int32_t d, int32_t max_ctas, int32_t block_size,
                                 int32_t max_blocks) {
    if (!plan) return OPATTN_ERR_INVALID_ARG;
    *plan = nullptr;
    if (max_ctas < 0) return OPATTN_ERR_INVALID_ARG;
    Geometry g;
    opattn_status st = check_geometry(cu_q, cu_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    st = check_decode_geometry(cu_q, g);
    if (st != OPATTN_OK) return st;
    opattn_plan* p = new opattn_plan;
    p->g = g;
    p->decode = true;
    p->block_size = block_size;
    p->max_blocks = max_blocks;
    if (cudaGetDevice(&p->device) != cudaSuccess) {
        delete p;
        return OPATTN_ERR_CUDA;
    }
    if (g.total_q > 0) {
        const int sms = device_sm_count();
        if (sms <= 0) {
            delete p;
            return OPATTN_ERR_CUDA;
        }
        const int32_t cap = max_ctas > 0 ? std::min(max_ctas, sms) : sms;
        // an explicit SM budget is kept exactly; the default grid may shrink
        // a little so that a uniform batch splits no pair
        const Clock::time_point t0 = Clock::now();
        build_decode_schedule(cu_q, cu_k, g, cap, &p->dsch, /*fit_grid=*/max_ctas == 0);
        log_decode_schedule("decode plan", p->dsch, us_since(t0));
        p->dw = decode_layout(p->dsch);
        // the work list, then the counters and the status word at zero
        const size_t init_bytes = p->dw.off_counters + p->dw.zero_bytes;
        std::vector<uint8_t> host(init_bytes, 0);
        pack_decode_upload(p->dsch, p->dw, host.data());
        if (cudaMalloc(&p->work, p->dw.bytes) != cudaSuccess) {
            delete p;
            return OPATTN_ERR_CUDA;
        }
        if (cudaMemcpy(p->work, host.data(), init_bytes, cudaMemcpyHostToDevice) != cudaSuccess) {
            cudaFree(p->work);
            delete p;
            return OPATTN_ERR_CUDA;
        }
    }
    *plan = p;
    return OPATTN_OK;
}
}  // namespace

extern "C" {

opattn_status opattn_decode_plan_create(opattn_plan** plan, const int32_t* cu_seqlens_q,
                                        const int32_t* cu_seqlens_k, int32_t n_seq, int32_t Hq, int32_t Hkv,
                                        int32_t d, int32_t max_ctas) {
    return decode_plan_create(plan, cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, max_ctas, 0, 0);
}

opattn_status opattn_prefill_paged(const void* q, const void* k_cache, const void* v_cache,
                                   const int32_t* block_table, int64_t num_blocks, int32_t block_size,
                                   int32_t max_blocks, void* o, float* lse, const int32_t* cu_seqlens_q,
                                   const int32_t* seqlens_k, int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d,
                                   float scale, void* stream) {
    PagedGeometry pg;
    opattn_status st = check_paged(seqlens_k, n_seq, block_size, max_blocks, &pg);
    if (st != OPATTN_OK) return st;
    PagedArgs pa;
    pa.block_table = block_table;
    pa.num_blocks = num_blocks;
    pa.block_size = block_size;
    pa.max_blocks = max_blocks;
    return prefill_impl(q, k_cache, v_cache, o, lse, cu_seqlens_q, pg.cu_k.data(), n_seq, Hq, Hkv, d, scale,
                        static_cast<cudaStream_t>(stream), 0u, false, &pa);
}

opattn_status opattn_prefill_paged_plan_create(opattn_plan** plan, const int32_t* cu_seqlens_q,
                                               const int32_t* seqlens_k, int32_t n_seq, int32_t Hq, int32_t Hkv,
                                               int32_t d, int32_t block_size, int32_t max_blocks, int32_t max_ctas) {
    if (plan) *plan = nullptr;
    PagedGeometry pg;
    opattn_status st = check_paged(seqlens_k, n_seq, block_size, max_blocks, &pg);
    if (st != OPATTN_OK) return st;
    st = opattn_plan_create(plan, cu_seqlens_q, pg.cu_k.data(), n_seq, Hq, Hkv, d, max_ctas);
    if (st != OPATTN_OK) return st;
    (*plan)->block_size = block_size;
    (*plan)->max_blocks = max_blocks;
    return OPATTN_OK;
}

opattn_status opattn_decode_paged(const void* q, const void* k_cache, const void* v_cache, const int32_t* block_table,
                                  int64_t num_blocks, int32_t block_size, int32_t max_blocks, void* o, float* lse,
                                  const int32_t* cu_seqlens_q, const int32_t* seqlens_k, int32_t n_seq, int32_t Hq,
                                  int32_t Hkv, int32_t d, float scale, void* stream) {
    PagedGeometry pg;
    opattn_status st = check_paged(seqlens_k, n_seq, block_size, max_blocks, &pg);
    if (st != OPATTN_OK) return st;
    PagedArgs pa;
    pa.block_table = block_table;
    pa.num_blocks = num_blocks;
    pa.block_size = block_size;
    pa.max_blocks = max_blocks;
    return decode_impl(q, k_cache, v_cache, o, lse, cu_seqlens_q, pg.cu_k.data(), n_seq, Hq, Hkv, d, scale,
                       static_cast<cudaStream_t>(stream), 0u, false, &pa);
}

opattn_status opattn_decode_paged_plan_create(opattn_plan** plan, const int32_t* cu_seqlens_q,
                                              const int32_t* seqlens_k, int32_t n_seq, int32_t Hq, int32_t Hkv,
                                              int32_t d, int32_t block_size, int32_t max_blocks, int32_t max_ctas) {
    if (plan) *plan = nullptr;
    PagedGeometry pg;
    opattn_status st = check_paged(seqlens_k, n_seq, block_size, max_blocks, &pg);
    if (st != OPATTN_OK) return st;
    return decode_plan_create(plan, cu_seqlens_q, pg.cu_k.data(), n_seq, Hq, Hkv, d, max_ctas, block_size,
                              max_blocks);
}

opattn_status opattn_plan_run_paged(const opattn_plan* plan, const void* q, const void* k_cache,
                                    const void* v_cache, const int32_t* block_table, int64_t num_blocks, void* o,
                                    float* lse, float scale, void* stream) {
    if (!plan || plan->block_size == 0) return OPATTN_ERR_INVALID_ARG;
    if (plan->g.total_q == 0) return OPATTN_OK;
    Geometry gq = plan->g;
    gq.total_k = 0;
    opattn_status st = check_tensors(q, nullptr, nullptr, o, lse, scale, gq);
    if (st != OPATTN_OK) return st;
    st = check_paged_tensors(k_cache, v_cache, block_table, num_blocks, plan->g, plan->block_size);
    if (st != OPATTN_OK) return st;
    uint8_t* work = static_cast<uint8_t*>(plan->work);
    const cudaStream_t st_ = static_cast<cudaStream_t>(stream);
    if (!plan->decode) {
        LaunchArgs a = make_args(q, k_cache, v_cache, o, lse, plan->g, scale, work, plan->w, plan->sch, 0u);
        a.block_table = block_table;
        a.max_blocks = plan->max_blocks;
        a.block_size = plan->block_size;
        a.num_blocks = num_blocks;
        return launch_prefill(a, st_) == 0 ? OPATTN_OK : OPATTN_ERR_CUDA;
    }
    DecodeLaunchArgs a = make_decode_args(q, k_cache, v_cache, o, lse, plan->g, scale, work, plan->dw,
                                          plan->dsch.n_cta, plan->dsch.max_cols, 0u);
    a.block_table = block_table;
    a.max_blocks = plan->max_blocks;
    a.block_size = plan->block_size;
    a.num_blocks = num_blocks;
    return launch_decode(a, st_) == 0 ? OPATTN_OK : OPATTN_ERR_CUDA;
}

}  // extern "C"

namespace {
opattn_status decode_schedule_out(const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq,
                                  int32_t Hq, int32_t Hkv, int32_t d, int32_t n_ctas, bool fit_grid, int32_t* units,
                                  int64_t unit_capacity, int32_t* cta_offsets, int64_t* n_units_out,
                                  int32_t* n_ctas_used) {
    if (n_ctas <= 0 || !n_units_out || !n_ctas_used) return OPATTN_ERR_INVALID_ARG;
    Geometry g;
    opattn_status st = check_geometry(cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, &g);
    if (st != OPATTN_OK) return st;
    st = check_decode_geometry(cu_seqlens_q, g);
    if (st != OPATTN_OK) return st;
    DecodeSchedule sch;
    build_decode_schedule(cu_seqlens_q, cu_seqlens_k, g, n_ctas, &sch, fit_grid);
    *n_units_out = static_cast<int64_t>(sch.units.size());
    *n_ctas_used = sch.n_cta;
    if (static_cast<int64_t>(sch.units.size()) > unit_capacity) return OPATTN_ERR_CAPACITY;
    if (!sch.units.empty() && (!units || !cta_offsets)) return OPATTN_ERR_INVALID_ARG;
    if (!sch.units.empty()) {
        std::memcpy(units, sch.units.data(), sch.units.size() * sizeof(DecUnit));
        std::memcpy(cta_offsets, sch.cta_off.data(), sch.cta_off.size() * sizeof(int32_t));
    }
    return OPATTN_OK;
}
}  // namespace

extern "C" {

opattn_status opattn_decode_schedule(const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k, int32_t n_seq,
                                     int32_t Hq, int32_t Hkv, int32_t d, int32_t n_ctas, int32_t* units,
                                     int64_t unit_capacity, int32_t* cta_offsets, int64_t* n_units_out,
                                     int32_t* n_ctas_used) {
    return decode_schedule_out(cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, n_ctas, false, units, unit_capacity,
                               cta_offsets, n_units_out, n_ctas_used);
}

opattn_status opattn_decode_schedule_default(const int32_t* cu_seqlens_q, const int32_t* cu_seqlens_k,
                                             int32_t n_seq, int32_t Hq, int32_t Hkv, int32_t d, int32_t sms,
                                             int32_t* units, int64_t unit_capacity, int32_t* cta_offsets,
                                             int64_t* n_units_out, int32_t* n_ctas_used) {
    return decode_schedule_out(cu_seqlens_q, cu_seqlens_k, n_seq, Hq, Hkv, d, sms, true, units, unit_capacity,
                               cta_offsets, n_units_out, n_ctas_used);
}

}  // extern "C"
