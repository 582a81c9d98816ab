// Plan evaluation in shared memory (rows a3-a11).
//
// Deterministic plans (pc_kernel): a CTA plays 16 plans as a three-stage warp
// pipeline over 16 dispatch positions at a time.  Producer warps turn each
// (plan, position) into a unit record (Eq. 3-4 chain, write list, release
// slot); two residency warps settle LRU model residency under capacity
// (Eq. 11) with four lanes per plan, each playing its own devices' units;
// one timing warp plays releases, loads, starts and finishes (Eq. 2, 5, 7,
// 10) with lane = plan.  Records pass through a ring of four buffers guarded
// by named barriers.  Per-plan state lives in shared memory:
//   - finish-time slots (u32 microseconds) assigned statically from the DAG
//     (wf_slots.cpp) instead of one word per activation, [slot][plan];
//   - per device: free time [device][plan]; resident weights, count and LRU
//     queue [device row][residency lane].
// Status bits (Eq. 8-10) come first from status_kernel, a warp per plan.
//
// Stochastic latencies (stoch_kernel): one plan per CTA, the same pipeline
// with one producer warp, residency settled once for all samples, and 64
// timing lanes, one per sample.
//
// Times: the deterministic sweep first plays u32 times and lists a plan whose
// times reach 2^32 us; a second instantiation with u64 times plays the listed
// plans, with 16, 6 or 3 plans per CTA by occupancy and finish slots of 40
// bits (a u32 word and a byte) while no time can reach 2^40 us.  Once a
// context has seen most plans leave 32 bits, a third instantiation (Rel32)
// plays the whole batch on u32 times counted from a per-plan base that rises
// with the plan's devices' free times, and lists for the u64 sweep only what
// leaves 32 bits even so.  Only a unit whose summed run time saturates 32
// bits goes on to the exact int64 path in wf_eval.cu, as does a stochastic
// plan whose times leave 32 bits.
//
// A compile-time variant (kPhi) also returns the window terms of Eq. 12's
// ranking key: residency marks a reload (a model its device held before) in
// bit 31 of the record's load word, and timing counts the timely prefetches
// and sums each unit's load delay plus its reload time.
#include <algorithm>
#include <mutex>
#include <utility>
#include <vector>

#include "wf_internal.cuh"

namespace {

__host__ __device__ __forceinline__ uint32_t round16(uint32_t x) { return (x + 15u) & ~15u; }

// Resident models of one device as a queue of 4-bit model ids, least
// recently used in nibble 0; nibbles at and above the count are zero.  A
// 32-bit word holds up to 8 models, a 64-bit word up to 16.
template <typename Q>
struct Lru;

template <>
struct Lru<uint32_t> {
    static constexpr uint32_t kOnes = 0x11111111u, kHigh = 0x88888888u;
    static constexpr int kSlots = 8;
    __device__ static __forceinline__ int32_t find(uint32_t q, uint32_t n, uint32_t m)
    {
        const uint32_t x = q ^ (kOnes * m);
        const uint32_t t = (x - kOnes) & ~x & kHigh;  // lowest zero nibble
        const int32_t k = t ? (__ffs((int)t) - 1) >> 2 : kSlots;
        return k < (int32_t)n ? k : (int32_t)n;
    }
    __device__ static __forceinline__ uint32_t remove(uint32_t q, int32_t k)
    {
        const uint32_t low = q & ((1u << (4 * k)) - 1u);
        const uint32_t high = k < kSlots - 1 ? ((q >> (4 * k + 4)) << (4 * k)) : 0u;
        return low | high;
    }
};

template <>
struct Lru<uint64_t> {
    static constexpr uint64_t kOnes = 0x1111111111111111ull, kHigh = 0x8888888888888888ull;
    static constexpr int kSlots = 16;
    __device__ static __forceinline__ int32_t find(uint64_t q, uint32_t n, uint32_t m)
    {
        const uint64_t x = q ^ (kOnes * m);
        const uint64_t t = (x - kOnes) & ~x & kHigh;
        const int32_t k = t ? (__ffsll((long long)t) - 1) >> 2 : kSlots;
        return k < (int32_t)n ? k : (int32_t)n;
    }
    __device__ static __forceinline__ uint64_t remove(uint64_t q, int32_t k)
    {
        const uint64_t low = k ? (q & ((1ull << (4 * k)) - 1)) : 0ull;
        const uint64_t high = k < kSlots - 1 ? ((q >> (4 * k + 4)) << (4 * k)) : 0ull;
        return low | high;
    }
};

__device__ __forceinline__ uint32_t bit_of_g(const uint32_t *row, int32_t n)
{
    return (__ldg(row + (n >> 5)) >> (n & 31)) & 1u;
}

// CTA shape, a three-stage pipeline over kChunk dispatch positions at a time:
// the last kProducers warps prepare the unit records of kP plans (lane =
// position) into a ring of kBuffers buffers; warps 1..kRes settle model
// residency (lane = plan and device group: hits, reclamations, occupancy
// changes); warp 0 plays the timing (lane = plan: releases, starts,
// finishes, slots).  With u32 times and 16 plans per CTA, four CTAs share an
// SM at 2,000 activations; the u64 variant holds fewer plans per CTA when its
// slots need the room.
constexpr int kChunk = 16;
constexpr int kPlansPerIter = 32 / kChunk;  // plans a producer warp covers per iteration
constexpr int kPlans32 = 16;                // plans per CTA of the u32 sweep
// Record buffers of the ring: four, or three under reclamation by next use,
// whose seventh record word would otherwise cost a CTA per SM at 2,000
// activations.  Named barriers: kFullP + b (producers -> residency), kFullR +
// b (residency -> timing), kEmpty + b (timing -> producers) for buffer b;
// kOpen (residency -> timing, once at the end).
template <int kReclaim>
struct Ring {
    static constexpr int kBuffers = kReclaim ? 3 : 4;
    static constexpr int kFullP = 1, kFullR = kFullP + kBuffers, kEmpty = kFullR + kBuffers, kOpen = kEmpty + kBuffers;
    static_assert(kOpen < 16, "named barriers");
};
constexpr int kRecWords = 6;

// The ring holds a record as word pairs (8-byte shared-memory accesses):
// (w0, w2) for timing, (w1, w3) read and rewritten by residency, (w4, w5)
// for timing, and under reclamation by next use (the unit's next use, 0).
template <int kReclaim>
struct RecPairs {
    static constexpr int kPairs = 3 + kReclaim;
};

template <int kP>
struct PcShape {
    static constexpr int kProducers = kP >= 32 ? 8 : kP >= 16 ? 4 : kP >= 6 ? 3 : 2;
    static constexpr int kRes = kP >= 32 ? 4 : kP >= 16 ? 2 : 1;  // residency warps
    static constexpr int kWarps = 1 + kRes + kProducers;
    // Four 16-plan CTAs share an SM (shared memory allows it at 2,000
    // activations), which bounds the registers per thread.
    static constexpr int kMinBlocks = kP >= 32 ? 2 : kP >= 16 ? 4 : 1;
    // Elements (8-byte word pairs) per (pair, position) row of the ring.  A
    // producer store covers 16 positions x 2 plans in two halves of 16
    // lanes; an odd pitch puts each half's 16 pairs on 32 distinct banks, and
    // the consumers' plan-major loads are contiguous.
    static constexpr int kPitch = kP | 1;
    static_assert(kChunk == 16 && kP >= 1 && kP <= 32, "ring pitch assumes 16 positions per chunk");
};

// Unit record (one per plan and dispatch position):
//   w0 run time of the unit (sum over the fused chain, Eq. 4) plus the grant,
//      saturated at 2^32 - 1 (a saturated unit sends its plan to the int64 path)
//   w1 KV admission of the unit (largest on the chain, Eq. 4); the residency
//      stage overwrites it with the load time the unit waits for (0 on a hit)
//   w2 arrival time of the unit's session
//   w3 device | model << 5 | prefetch << 9 | reclaim << 10 | writes << 11 | skip << 14
//      | first write code << 16; the residency stage clears the prefetch bit
//      on a hit and sets kWasEmpty (bit 10) and kEmptied (bit 15) for timing
//   w4 second write code | third write code << 16
//   w5 the unit's last member | release slot code << 16 (bit 31: accumulator;
//      0xFFFF: none); in the batched producer's records the low half holds
//      the fourth write code instead when the unit writes exactly four (with
//      five or more, the timing stage reads the last member's list)
constexpr uint32_t kSkip = 1u << 14;
constexpr uint32_t kPrefetch = 1u << 9;
constexpr uint32_t kWasEmpty = 1u << 10;   // after residency: a miss on an empty device
constexpr uint32_t kEmptied = 1u << 15;    // after residency: the unit's reclaim empties the device
constexpr uint32_t kRunCap = 0xFFFFFFFFu;  // saturation of w0
// A plan's open word in shared memory: the devices still occupied at its end
// (residency, low bits) and, from bit kOpenBad, the placement status bits
// (WF_ST_DEVICE, WF_ST_CAPACITY) its producers found.
constexpr int kOpenBad = 24;

// Residency lanes per plan: a device group each (d = g mod kG), or one lane
// for every device under reclamation by next use.
// A lane's state for its t-th device (d = g + t kG) sits at [t][lane]: the
// lanes of a warp touch consecutive words.
template <int kP, int kReclaim>
struct PcGroups {
    static constexpr int kG = kReclaim ? 1 : (32 * PcShape<kP>::kRes) / kP;
    static constexpr int kLanes = kG == 1 ? kP : 32 * PcShape<kP>::kRes;  // row length of the state
    static_assert(kG >= 1 && kG * kP <= 32 * PcShape<kP>::kRes, "residency lanes");
    __host__ __device__ static int32_t rows(int32_t D) { return (D + kG - 1) / kG; }
};

// Storage of the finish-time slots, [slot][plan]: TT words, or (Split40, for
// u64 times whose every value stays below 2^40 us) a 32-bit low word per
// slot and an 8-bit high byte in an array of its own: 5 bytes instead of 8,
// so more plans fit an SM.
struct Split40 {};

// Relative 32-bit times (slot storage Rel32, with TT = uint32_t): every time
// the timing stage keeps (finish slots, device free times, the plan's end)
// counts from a per-plan base B, which it raises now and then to one below
// the smallest device free time.  That is exact: every later unit starts at
// or after its device's free time, so a stored finish or arrival below B can
// be read as B without changing any start (Eq. 2, 5, 7).  A session slot
// that would fall below B keeps its exact value in global memory instead,
// for the p95.
struct Rel32 {};
template <typename ST>
struct IsRel {
    static constexpr bool value = false;
};
template <>
struct IsRel<Rel32> {
    static constexpr bool value = true;
};
constexpr uint32_t kRebaseAt = 3u << 30;   // a plan's end above this raises its base ...
constexpr uint32_t kRebaseMin = 1u << 28;  // ... by at least this much, else not at all

// Up to this many sessions the timing lane selects its plan's p95 itself;
// beyond, a warp per plan does after the sweep (warp_select).
constexpr int32_t kLaneSelect = 32;

template <typename ST>
struct SlotBytes {
    static constexpr uint32_t kLo = sizeof(ST), kHi = 0;
};
template <>
struct SlotBytes<Split40> {
    static constexpr uint32_t kLo = 4, kHi = 1;
};
template <>
struct SlotBytes<Rel32> {
    static constexpr uint32_t kLo = 4, kHi = 0;
};

template <typename TT, typename ST, int kS>
struct SlotArr {  // plain words
    TT *v;
    __device__ __forceinline__ TT get(uint32_t i) const { return v[i * kS]; }
    __device__ __forceinline__ void set(uint32_t i, TT x) const { v[i * kS] = x; }
};
template <int kS>
struct SlotArr<uint64_t, Split40, kS> {
    uint32_t *lo;
    uint8_t *hi;
    __device__ __forceinline__ uint64_t get(uint32_t i) const
    {
        return ((uint64_t)hi[i * kS] << 32) | lo[i * kS];
    }
    __device__ __forceinline__ void set(uint32_t i, uint64_t x) const
    {
        lo[i * kS] = (uint32_t)x;
        hi[i * kS] = (uint8_t)(x >> 32);
    }
};

// Slots 2i and 2i + 1 of a 32-bit slot array read as one 64-bit value i (the
// relative sweep's session latencies at the end of a plan).
template <int kS>
struct PairArr {
    uint32_t *v;
    __device__ __forceinline__ uint64_t get(uint32_t i) const
    {
        return ((uint64_t)v[(2 * i + 1) * kS] << 32) | v[2 * i * kS];
    }
    __device__ __forceinline__ void set(uint32_t i, uint64_t x) const
    {
        v[2 * i * kS] = (uint32_t)x;
        v[(2 * i + 1) * kS] = (uint32_t)(x >> 32);
    }
};

struct PcLayout {
    uint32_t weight, cap, load, arr, ring, slots, slots_hi, tfree, used, queue, nres, open, flag, nuse, rcnt, gmask,
        everl, total;
};

// Shared memory of a CTA of kP plans with TT times and NS slots per plan;
// with reclamation by next use (kReclaim) the ring carries a seventh record
// word and each plan keeps per (device, model) the next use of the resident
// copy and per model the number of devices holding it; with the window terms
// of Eq. 12 (kPhi) each residency lane keeps per device the models it ever
// held.
template <int kP, typename TT, int kReclaim = 0, bool kPhi = false, typename ST = TT>
__host__ __device__ inline PcLayout pc_layout(int32_t D, int32_t M, int32_t W, int32_t NS)
{
    constexpr uint32_t t = sizeof(TT);
    PcLayout l;
    uint32_t o = 0;
    l.weight = o; o += round16(4u * M);
    l.cap = o; o += round16(4u * D);
    l.load = o; o += round16(4u * M * D);
    l.arr = o; o += round16(4u * W);
    l.ring = o; o += round16(8u * Ring<kReclaim>::kBuffers * RecPairs<kReclaim>::kPairs * kChunk * PcShape<kP>::kPitch);
    l.slots = o; o += round16(SlotBytes<ST>::kLo * (uint32_t)NS * kP);
    l.slots_hi = o; o += round16(SlotBytes<ST>::kHi * (uint32_t)NS * kP);
    l.tfree = o; o += round16(t * D * kP);
    const uint32_t rs = (uint32_t)(PcGroups<kP, kReclaim>::rows(D) * PcGroups<kP, kReclaim>::kLanes);
    l.used = o; o += round16(4u * rs);
    l.queue = o; o += round16((M <= 8 ? 4u : 8u) * rs);  // Lru<uint32_t> or Lru<uint64_t>
    l.nres = o; o += round16(rs);
    l.open = o; o += round16(4u * kP);
    l.flag = o; o += 16;
    l.nuse = o; o += kReclaim ? round16(2u * D * M * kP) : 0u;
    l.rcnt = o; o += kReclaim ? round16((uint32_t)M * kP) : 0u;
    l.gmask = o; o += round16(4u * Ring<kReclaim>::kBuffers * PcGroups<kP, kReclaim>::kG * kP);
    l.everl = o; o += kPhi ? round16(2u * rs) : 0u;
    l.total = o;
    return l;
}


__device__ __forceinline__ void named_sync(int id, int threads)
{
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

__device__ __forceinline__ void named_arrive(int id, int threads)
{
    asm volatile("bar.arrive %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// The r-th smallest (0-based) of slots 0 .. n-1 of a slot array (one thread).
template <typename TT, typename SA>
__device__ TT select_slots(const SA &v, int32_t n, int32_t r)
{
    int32_t lo = 0, hi = n - 1;
    while (lo < hi) {
        const TT pivot = v.get(lo + (hi - lo) / 2);
        int32_t i = lo, j = hi;
        while (i <= j) {
            while (v.get(i) < pivot) ++i;
            while (v.get(j) > pivot) --j;
            if (i <= j) { const TT t = v.get(i); v.set(i, v.get(j)); v.set(j, t); ++i; --j; }
        }
        if (r <= j) hi = j;
        else if (r >= i) lo = i;
        else return v.get(r);
    }
    return v.get(r);
}

// The same by a whole warp.  The p95's rank is near the top (the
// (n - r)-th largest: 4th of 64, 13th of 256), so the warp takes maxima: the
// largest value below the last maximum and how many equal it, until the
// count reaches n - r.  For a rank further down, a radix selection from the
// highest bit set in any value, each bit decided by a ballot.  Up to 32
// kCache values are read once into registers (a column of the slot array is
// a strided read with bank conflicts); more are read again for every step.
template <int kCache, typename SA, typename F>
__device__ __forceinline__ void each_value(const SA &a, int32_t n, bool cached, const uint64_t (&c)[kCache], F &&f)
{
    const int lane = threadIdx.x & 31;
    if (cached) {
#pragma unroll
        for (int j = 0; j < kCache; ++j)
            if (32 * j < n) f(c[j], 32 * j + lane < n);
    } else {
        for (int32_t i0 = 0; i0 < n; i0 += 32) {
            const int32_t i = i0 + lane;
            f(i < n ? (uint64_t)a.get(i) : 0ull, i < n);
        }
    }
}

template <typename SA>
__device__ uint64_t warp_select(const SA &a, int32_t n, int32_t r)
{
    constexpr int kCache = 8;
    constexpr int32_t kMaxSteps = 32;
    const int lane = threadIdx.x & 31;
    const bool cached = n <= 32 * kCache;
    uint64_t c[kCache];  // the values, 0 beyond n (never above the answer when taking maxima)
#pragma unroll
    for (int j = 0; j < kCache; ++j) {
        const int32_t i = 32 * j + lane;
        c[j] = cached && i < n ? (uint64_t)a.get(i) : 0ull;
    }
    if (n - r <= kMaxSteps) {
        int32_t need = n - r;  // the need-th largest of the values below thr
        uint64_t thr = ~0ull;
        for (;;) {
            uint64_t mx = 0;
            each_value(a, n, cached, c, [&](uint64_t v, bool) {
                if (v < thr) mx = max(mx, v);
            });
            const uint32_t hi = __reduce_max_sync(0xFFFFFFFFu, (uint32_t)(mx >> 32));
            const uint32_t lo = __reduce_max_sync(0xFFFFFFFFu, (uint32_t)(mx >> 32) == hi ? (uint32_t)mx : 0u);
            const uint64_t m = ((uint64_t)hi << 32) | lo;
            int32_t cnt = 0;
            each_value(a, n, cached, c, [&](uint64_t v, bool in) {
                cnt += __popc(__ballot_sync(0xFFFFFFFFu, in && v == m));
            });
            if (cnt >= need) return m;
            need -= cnt;
            thr = m;
        }
    }
    uint64_t any = 0;
    each_value(a, n, cached, c, [&](uint64_t v, bool) { any |= v; });
    any = ((uint64_t)__reduce_or_sync(0xFFFFFFFFu, (uint32_t)(any >> 32)) << 32) |
          __reduce_or_sync(0xFFFFFFFFu, (uint32_t)any);
    uint64_t prefix = 0;
    for (int bit = any ? 63 - __clzll((long long)any) : -1; bit >= 0; --bit) {
        int32_t zeros = 0;  // values that match prefix above bit and have a 0 there
        each_value(a, n, cached, c, [&](uint64_t v, bool in) {
            zeros += __popc(__ballot_sync(0xFFFFFFFFu, in && ((v ^ prefix) >> bit) == 0));
        });
        if (r >= zeros) {
            r -= zeros;
            prefix |= 1ull << bit;
        }
    }
    return prefix;
}

// Two extra slots follow a plan's nslots slots: a sink that absorbs writes
// with no reader (index nslots) and a slot that always holds 0 (nslots + 1),
// the release slot of a node without predecessors.  With them every unit
// reads one release slot and writes its first two codes without branching;
// the host encodes both into the per-node records (hrec).

// Row pointers of one plan.
struct PlanPtrs {
    const uint8_t *place;
    const uint16_t *order;
    const uint32_t *fuse, *prefetch, *retain;
};

// Producer: the unit record of dispatch position i of a plan.  One 16-byte
// gather (hrec) gives a node's links, release slot, model, write codes and
// arrival; the chain walk reads the members' records, whose last one holds
// the unit's write codes.
__device__ __forceinline__ void produce(const wf_dev_problem &dp, const PlanPtrs &r, int32_t i,
                                        uint32_t rec[kRecWords], int32_t *head = nullptr)
{
    const int32_t D = dp.D;
    const int32_t h = __ldg(r.order + i);
    if (head) *head = h;
    // Loads that depend on h alone go out together, ahead of any branch.
    const int32_t d = __ldg(r.place + h);
    const uint4 hr = __ldg(dp.hrec + h);
    const uint32_t fw = __ldg(r.fuse + (h >> 5));
    const uint32_t pw = __ldg(r.prefetch + (h >> 5));
    const uint32_t fp = hr.x & 0xFFFFu;
    if (fp != 0xFFFFu && ((fw >> (h & 31)) & 1u) && __ldg(r.place + fp) == d) {  // runs inside its head's unit
        rec[3] = kSkip;
        return;
    }
    const int2 lk0 = __ldg(dp.lk + h * D + d);
    uint32_t run = (uint32_t)lk0.x + (uint32_t)dp.grant, ovf = 0;  // both < 2^31: no wrap
    int32_t kv = lk0.y, tail = h;
    uint32_t ty = hr.y, tw = hr.w;  // the tail's write codes
    for (uint32_t s = hr.x >> 16; s != 0xFFFFu;) {  // Eq. 3 chain
        if (!bit_of_g(r.fuse, s) || __ldg(r.place + s) != d) break;
        const int2 lk = __ldg(dp.lk + s * D + d);
        const uint4 sr = __ldg(dp.hrec + s);
        const uint32_t r2 = run + (uint32_t)lk.x;
        ovf |= r2 < run;
        run = r2;
        kv = max(kv, lk.y);
        tail = (int32_t)s;
        ty = sr.y;
        tw = sr.w;
        s = sr.x >> 16;
    }
    const uint32_t nwl = (ty >> 20) & 7u;
    const uint32_t c2 = __ldg(dp.wc23 + tail) & 0xFFFFu;
    const uint32_t pf = (pw >> (h & 31)) & 1u;
    const uint32_t reclaim = r.retain ? !bit_of_g(r.retain, tail) : 0u;
    rec[0] = ovf ? kRunCap : run;
    rec[1] = (uint32_t)kv;
    rec[2] = hr.z;
    rec[3] = (uint32_t)d | (((hr.y >> 16) & 15u) << 5) | (pf << 9) | (reclaim << 10) | (nwl << 11) |
             (tw << 16);
    rec[4] = (tw >> 16) | (c2 << 16);
    rec[5] = (uint32_t)tail | (hr.y << 16);
}

// Row of one plan for the batched producer: placement and dispatch rows, and
// the byte offset of its fusion / prefetch / retain bit rows.
struct RowPtrs {
    const uint8_t *place;
    const uint16_t *order;
    int64_t boff;
};

__device__ __forceinline__ const uint32_t *bits_row(const uint32_t *base, int64_t boff)
{
    return (const uint32_t *)((const uint8_t *)base + boff);
}

// Bulk prefetch of [p, p + bytes) into L2 (p 16-byte aligned, bytes a
// multiple of 16); no completion to wait for.
__device__ __forceinline__ void l2_prefetch(const void *p, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

// The records of kI (plan, position) pairs at once, with the gathers of all
// pairs issued together in three dependent rounds: the head's own tables
// (placement, node record, fusion / prefetch / retain words, third and
// fourth write codes); then its run time and KV on its device and the placement and fusion
// bit of its fusible neighbours; then the rare fused chain, walked as in
// produce().  Each record goes to the ring as soon as it is complete; act[j]
// false leaves a skip record.  dev[j] is the unit's device (all ones for a
// skip record).
template <int kI, int kPitch>
__device__ __forceinline__ void produce_batch(const wf_dev_problem &dp, const wf_plans &pl, const RowPtrs *rp,
                                              const bool *act, const int32_t *hh, uint2 *rb, int pos,
                                              const int *qq, uint32_t *dev, uint32_t *open)
{
    const int32_t D = dp.D;
    uint32_t d[kI], fw[kI], pw[kI], rw[kI], c2[kI], bad[kI];
    uint4 hr[kI];
#pragma unroll
    for (int j = 0; j < kI; ++j) {
        const int32_t h = hh[j];
        d[j] = act[j] ? __ldg(rp[j].place + h) : 0u;
        hr[j] = act[j] ? __ldg(dp.hrec + h) : make_uint4(0xFFFFFFFFu, 0, 0, 0);
        fw[j] = act[j] ? __ldg(bits_row(pl.fuse, rp[j].boff) + (h >> 5)) : 0u;
        pw[j] = act[j] ? __ldg(bits_row(pl.prefetch, rp[j].boff) + (h >> 5)) : 0u;
        rw[j] = act[j] && pl.retain ? __ldg(bits_row(pl.retain, rp[j].boff) + (h >> 5)) : 0xFFFFFFFFu;
        c2[j] = act[j] ? __ldg(dp.wc23 + h) : 0u;
    }
    // Placement and fit (Eq. 8) of every position's activation: a device
    // index beyond D here, a device it does not fit (KV entry -1 in lk) with
    // the next gathers.  A plan with either gets the status bits, and the
    // record a skip, so no later stage indexes by it.
#pragma unroll
    for (int j = 0; j < kI; ++j) {
        bad[j] = act[j] && d[j] >= (uint32_t)D ? (uint32_t)WF_ST_DEVICE : 0u;
        if (bad[j]) d[j] = 0u;
    }
    int2 lk0[kI];
    uint32_t pprev[kI], fnx[kI], pnx[kI];
#pragma unroll
    for (int j = 0; j < kI; ++j) {
        const uint32_t fp = hr[j].x & 0xFFFFu, s = hr[j].x >> 16;
        lk0[j] = act[j] ? __ldg(dp.lk + hh[j] * D + (int32_t)d[j]) : make_int2(0, 0);
        pprev[j] = act[j] && fp != 0xFFFFu ? __ldg(rp[j].place + fp) : 0xFFFFFFFFu;  // never a device
        fnx[j] = act[j] && s != 0xFFFFu ? __ldg(bits_row(pl.fuse, rp[j].boff) + (s >> 5)) : 0u;
        pnx[j] = act[j] && s != 0xFFFFu ? __ldg(rp[j].place + s) : 0xFFFFFFFFu;
    }
#pragma unroll
    for (int j = 0; j < kI; ++j) {
        dev[j] = 0xFFFFFFFFu;
        if (qq[j] < 0) continue;  // a lane beyond the CTA's plans
        uint2 *dst = rb + pos * kPitch + qq[j];
        const int32_t h = hh[j];
        const uint32_t s0 = hr[j].x >> 16;
        if (act[j] && !bad[j] && lk0[j].y < 0) bad[j] = (uint32_t)WF_ST_CAPACITY;  // (d was cleared for a bad device)
        if (bad[j]) atomicOr(open + qq[j], bad[j] << kOpenBad);
        if (!act[j] || bad[j] || (((fw[j] >> (h & 31)) & 1u) && pprev[j] == d[j])) {  // no unit, or inside its head's
            dst[0] = make_uint2(0u, 0u);
            dst[1 * kChunk * kPitch] = make_uint2(0u, kSkip);
            dst[2 * kChunk * kPitch] = make_uint2(0u, 0u);
            continue;
        }
        uint32_t run = (uint32_t)lk0[j].x + (uint32_t)dp.grant, ovf = 0;  // both < 2^31: no wrap
        int32_t kv = lk0[j].y, tail = h;
        uint32_t ty = hr[j].y, tw = hr[j].w, c2t = c2[j], rwt = rw[j];
        uint32_t cbad = 0;  // a member that does not fit the head's device
        if (s0 != 0xFFFFu && ((fnx[j] >> (s0 & 31)) & 1u) && pnx[j] == d[j]) {  // Eq. 3 chain
            const uint32_t *fuse = bits_row(pl.fuse, rp[j].boff);
            for (uint32_t s = s0; s != 0xFFFFu;) {
                if (s != s0 && (!bit_of_g(fuse, s) || __ldg(rp[j].place + s) != d[j])) break;
                const int2 lk = __ldg(dp.lk + s * D + d[j]);
                cbad |= lk.y < 0;
                const uint4 sr = __ldg(dp.hrec + s);
                const uint32_t r2 = run + (uint32_t)lk.x;
                ovf |= r2 < run;
                run = r2;
                kv = max(kv, lk.y);
                tail = (int32_t)s;
                ty = sr.y;
                tw = sr.w;
                s = sr.x >> 16;
            }
            c2t = __ldg(dp.wc23 + tail);
            rwt = pl.retain ? __ldg(bits_row(pl.retain, rp[j].boff) + (tail >> 5)) : 0xFFFFFFFFu;
        }
        if (cbad) {  // (the member's own position flags the plan as well)
            atomicOr(open + qq[j], (uint32_t)WF_ST_CAPACITY << kOpenBad);
            dst[0] = make_uint2(0u, 0u);
            dst[1 * kChunk * kPitch] = make_uint2(0u, kSkip);
            dst[2 * kChunk * kPitch] = make_uint2(0u, 0u);
            continue;
        }
        const uint32_t nwl = (ty >> 20) & 7u;
        const uint32_t pf = (pw[j] >> (h & 31)) & 1u;
        const uint32_t reclaim = ((rwt >> (tail & 31)) & 1u) ^ 1u;
        dst[0] = make_uint2(ovf ? kRunCap : run, hr[j].z);
        dst[1 * kChunk * kPitch] = make_uint2(
            (uint32_t)kv, d[j] | (((hr[j].y >> 16) & 15u) << 5) | (pf << 9) | (reclaim << 10) | (nwl << 11) | (tw << 16));
        dst[2 * kChunk * kPitch] = make_uint2((tw >> 16) | (c2t << 16),
                                              (nwl == 4 ? c2t >> 16 : (uint32_t)tail) | (hr[j].y << 16));
        dev[j] = d[j];
    }
}

// One unit on its device under least-recently-used reclamation (Eq. 11,
// Section 3.5): q / n / u_d are the device's queue, resident count and
// resident weights.  The unit's own model leaves the queue first; the
// victims are then exactly the queue's first entries (least recently used
// first), and the unit's model goes back in as the most recently used.
// Returns the record's rewritten (w1, w3): the load the unit waits for (none
// on a hit, Eq. 5) and the occupancy changes of section 4.3.
template <typename Q>
__device__ __forceinline__ uint2 settle_lru(Q &q, uint32_t &n, uint32_t &u_d, uint32_t capd, uint32_t r1,
                                            uint32_t r3, const int32_t *weight, const int32_t *load, int32_t D,
                                            int *err, bool &missed)
{
    const int32_t d = (int32_t)(r3 & 31u);
    const uint32_t m = (r3 >> 5) & 15u;
    const uint32_t wm = (uint32_t)weight[m];
    const bool was_empty = n == 0;
    const int32_t kq = Lru<Q>::find(q, n, m);
    const bool hit = kq < (int32_t)n;
    missed = !hit;
    q = hit ? Lru<Q>::remove(q, hit ? kq : 0) : q;  // (an index below the queue length)
    n -= hit ? 1u : 0u;
    const uint32_t need = hit ? r1 : wm + r1;  // used + need <= cap + peak < 2^32
    uint32_t e = 0;
    while (u_d + need > capd && e < n) {
        u_d -= (uint32_t)weight[(uint32_t)(q >> (4 * e)) & 15u];
        ++e;
    }
    if (u_d + need > capd) atomicExch(err, 2);  // unreachable for a valid plan
    q = e < (uint32_t)Lru<Q>::kSlots ? (q >> (4 * e)) : (Q)0;
    n -= e;
    q |= (Q)m << (4 * n);
    n += 1;
    u_d += hit ? 0u : wm;
    uint32_t emptied = 0;
    if ((r3 >> 10) & 1u) {  // retain bit 0: reclaim at the end of the unit
        q &= ~((Q)0xF << (4 * (n - 1)));
        n -= 1;
        u_d -= wm;
        emptied = n == 0;
    }
    return make_uint2(hit ? 0u : (uint32_t)load[m * D + d],
                      (r3 & ~(kPrefetch | kWasEmpty)) | (hit ? 0u : (r3 & kPrefetch)) |
                          (was_empty ? kWasEmpty : 0u) | (emptied ? kEmptied : 0u));
}

// A finish time into a slot: an accumulator keeps the latest of its
// writers, any other slot takes the value.
template <typename TT, typename SA>
__device__ __forceinline__ void publish(const SA &slots, uint32_t code, TT c)
{
    const uint32_t i = code & 0x7FFFu;
    slots.set(i, (code & 0x8000u) ? max(slots.get(i), c) : c);
}

// The sweep of groups of kP plans: every plan of the batch (in_list NULL, plan
// = group * kP + q) or the listed ones (plan = in_list[group * kP + q] below
// *in_count).  CTA b plays groups b, b + gridDim.x, ...  TT = uint32_t: a plan whose times leave 32 bits is appended to
// ovf_list; once every plan of a CTA has, its stages run on without loads.
// TT = uint64_t: only a unit whose summed run time reaches 2^32 - 1 sends its
// plan to ovf_list.
template <typename Q, typename TT, int kP, int kReclaim, bool kPhi, typename ST>
__global__ void __launch_bounds__(32 * PcShape<kP>::kWarps, PcShape<kP>::kMinBlocks)
pc_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, const int32_t *in_list, const int32_t *in_count,
          int32_t *ovf_list, int32_t *ovf_count)
{
    constexpr int kRW = RecPairs<kReclaim>::kPairs;  // word pairs per record in the ring
    using S = PcShape<kP>;
    constexpr int kPitch = S::kPitch;
    constexpr int kProdThreads = 32 * S::kProducers;
    constexpr int kResThreads = 32 * S::kRes;
    constexpr bool kNarrow = sizeof(TT) == 4;
    constexpr bool kRel = IsRel<ST>::value;  // relative 32-bit times
    static_assert(!kRel || (kNarrow && kReclaim == 0 && !kPhi), "relative times: u32, least recently used");
    constexpr int kG = PcGroups<kP, kReclaim>::kG;  // residency lanes per plan
    using RG = Ring<kReclaim>;
    constexpr int kBuffers = RG::kBuffers, kFullP = RG::kFullP, kFullR = RG::kFullR, kEmpty = RG::kEmpty,
                  kOpen = RG::kOpen;
    extern __shared__ __align__(128) uint8_t sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W;
    const int32_t rank = (int32_t)((95 * (int64_t)W + 99) / 100 - 1);  // the p95's nearest rank (Section 4.2)
    const PcLayout L = pc_layout<kP, TT, kReclaim, kPhi, ST>(D, M, W, dp.nslots + 2);
    const int64_t total = in_list ? (int64_t)*in_count : pl.P;
    if ((int64_t)blockIdx.x * kP >= total) return;  // the whole CTA: no plan
    uint2 *ring = (uint2 *)(sm + L.ring);
    const int32_t chunks = (N + kChunk - 1) / kChunk;
    volatile uint32_t *gave_up = (volatile uint32_t *)(sm + L.flag);

    int32_t *weight = (int32_t *)(sm + L.weight);
    int32_t *cap = (int32_t *)(sm + L.cap);
    int32_t *load = (int32_t *)(sm + L.load);
    uint32_t *arrival = (uint32_t *)(sm + L.arr);
    uint32_t *open = (uint32_t *)(sm + L.open);
    uint32_t *gmask = (uint32_t *)(sm + L.gmask);  // [buffer][device group][plan]
    for (int32_t k = threadIdx.x; k < M; k += blockDim.x) weight[k] = __ldg(dp.weight + k);
    for (int32_t k = threadIdx.x; k < D; k += blockDim.x) cap[k] = __ldg(dp.cap + k);
    for (int32_t k = threadIdx.x; k < M * D; k += blockDim.x) load[k] = __ldg(dp.load + k);
    for (int32_t k = threadIdx.x; k < W; k += blockDim.x) arrival[k] = (uint32_t)__ldg(dp.arrival + k);
    // (each role's first __syncthreads below publishes these tables)

  for (int64_t j0 = (int64_t)blockIdx.x * kP; j0 < total; j0 += (int64_t)gridDim.x * kP) {
    const int ng = (int)(total - j0 < kP ? total - j0 : kP);
    if (threadIdx.x == 0) *gave_up = 0;
    if (threadIdx.x < kP) open[threadIdx.x] = 0;

    if (warp > S::kRes) {
        // ---------------- producers: lane = dispatch position ----------------
        __syncthreads();
        const int pw = warp - 1 - S::kRes;
        const int pos = lane % kChunk, sub = lane / kChunk;
        // The plans this lane serves, fixed for the whole sweep: row pointers
        // and whether the plan is live, resolved once.
        constexpr int kStep = S::kProducers * kPlansPerIter;
        constexpr int kIters = (kP + kStep - 1) / kStep;
        RowPtrs rp[kIters];
        bool okq[kIters];
        int qq[kIters];
        int64_t qplan[kIters];
#pragma unroll
        for (int j = 0; j < kIters; ++j) {
            const int q = pw * kPlansPerIter + j * kStep + sub;
            qq[j] = q < kP ? q : -1;
            okq[j] = q < kP && q < ng;
            qplan[j] = 0;
            rp[j].place = nullptr;
            rp[j].order = nullptr;
            rp[j].boff = 0;
            if (okq[j]) {
                const int64_t pq = in_list ? (int64_t)__ldg(in_list + j0 + q) : j0 + q;
                qplan[j] = pq;
                okq[j] = __ldg(out.status + pq) == 0;
                rp[j].place = pl.place + pq * pl.place_stride;
                rp[j].order = (const uint16_t *)((const uint8_t *)pl.order + pq * pl.order_stride);
                rp[j].boff = pq * pl.bits_stride;
            }
        }
        // The node-indexed rows (placement, fusion and prefetch bits) are
        // gathered all through the sweep; one bulk L2 prefetch per row up
        // front streams them in rather than sector by sector.  (Rows are
        // 16-byte aligned, and their 16-byte-rounded sizes fit the strides.)
        const uint32_t place_bytes = (uint32_t)((N + 15) & ~15), bits_bytes = (uint32_t)((((N + 31) >> 5) * 4 + 15) & ~15);
#pragma unroll
        for (int j = 0; j < kIters; ++j)
            if (pos == 0 && okq[j]) {
                l2_prefetch(rp[j].place, place_bytes);
                l2_prefetch(bits_row(pl.fuse, rp[j].boff), bits_bytes);
                l2_prefetch(bits_row(pl.prefetch, rp[j].boff), bits_bytes);
            }
        // Dispatch entries are read one chunk ahead of their use.
        int32_t h0[kIters];
#pragma unroll
        for (int j = 0; j < kIters; ++j) h0[j] = okq[j] && pos < N ? __ldg(rp[j].order + pos) : 0;
        // The timing stage's give-up flag, read a chunk before it is used so
        // that no load of this chunk waits for it.
        bool quit = false;
        for (int32_t c = 0; c < chunks; ++c) {
            const int b = c % kBuffers;
            if (c >= kBuffers) named_sync(kEmpty + b, kProdThreads + 32);  // timing released buffer b
            uint2 *rb = ring + b * kRW * kChunk * kPitch;
            const int32_t i = c * kChunk + pos;
            int32_t h1[kIters];
            bool act[kIters];
#pragma unroll
            for (int j = 0; j < kIters; ++j) {
                h1[j] = okq[j] && i + kChunk < N && !quit ? __ldg(rp[j].order + i + kChunk) : 0;
                act[j] = okq[j] && i < N && !quit;
                if (kReclaim && qq[j] >= 0)  // the next use of this unit's model on its device
                    rb[(3 * kChunk + pos) * kPitch + qq[j]] =
                        make_uint2(act[j] ? (uint32_t)__ldg(dp.nextuse + qplan[j] * (int64_t)N + i) : 0xFFFFu, 0u);
            }
            uint32_t dev[kIters];
            produce_batch<kIters, kPitch>(dp, pl, rp, act, h0, rb, pos, qq, dev, open);
            // For each residency lane, the chunk's units on its devices: one
            // ballot per device group; each half-warp holds one plan.
#pragma unroll
            for (int j = 0; j < kIters; ++j) {
                const uint32_t key = dev[j] == 0xFFFFFFFFu ? (uint32_t)kG : dev[j] % kG;
#pragma unroll
                for (int gg = 0; gg < kG; ++gg) {
                    const uint32_t bal = __ballot_sync(0xFFFFFFFFu, key == (uint32_t)gg);
                    if (pos == gg && qq[j] >= 0) gmask[(b * kG + gg) * kP + qq[j]] = (bal >> (kChunk * sub)) & 0xFFFFu;
                }
            }
#pragma unroll
            for (int j = 0; j < kIters; ++j) h0[j] = h1[j];
            quit = kNarrow && *gave_up;
            named_arrive(kFullP + b, kProdThreads + kResThreads);  // buffer b is full
        }
        // Match the timing stage's releases of the last buffers.
        for (int32_t c = chunks; c < chunks + kBuffers; ++c)
            if (c >= kBuffers) named_sync(kEmpty + c % kBuffers, kProdThreads + 32);
    } else if (warp >= 1) {
        // ---------------- residency (Eq. 11, Section 3.5) ----------------
        // Lane (plan, device group): kG lanes per plan, and lane g plays the
        // plan's units on the devices d = g (mod kG) in dispatch order;
        // under least-recently-used reclamation devices do not interact.
        // Reclamation by next use counts a model's copies over all devices,
        // so there one lane per plan plays every device.  The producers
        // leave each lane's units of the chunk as a mask (gmask).
        const int rl = (warp - 1) * 32 + lane;
        const int qp = rl / kG, g = rl % kG;
        const bool rmine = qp < kP;
        const int64_t p = (rmine && qp < ng) ? (in_list ? (int64_t)in_list[j0 + qp] : j0 + qp) : 0;
        const bool live = rmine && qp < ng && out.status[p] == 0;
        constexpr int kRow = PcGroups<kP, kReclaim>::kLanes;
        uint32_t *used = (uint32_t *)(sm + L.used) + rl;  // [device / kG][lane]
        Q *queue = (Q *)(sm + L.queue) + rl;
        uint8_t *nres = sm + L.nres + rl;
        uint16_t *nuse = (uint16_t *)(sm + L.nuse) + qp;  // [device][model][plan]
        uint8_t *rcnt = sm + L.rcnt + qp;                 // [model][plan]
        uint16_t *everl = (uint16_t *)(sm + L.everl) + rl;  // [device / kG][lane], bit m: m was held (kPhi)
        if (rmine) {
            for (int32_t t = 0; t * kG + g < D; ++t) {
                used[t * kRow] = 0; queue[t * kRow] = 0; nres[t * kRow] = 0;
                if (kPhi) everl[t * kRow] = 0;
            }
            if (kReclaim)
                for (int32_t k = 0; k < M; ++k) rcnt[k * kP] = 0;
        }
        __syncthreads();
        for (int32_t c = 0; c < chunks; ++c) {
            const int b = c % kBuffers;
            named_sync(kFullP + b, kProdThreads + kResThreads);
            uint2 *rb = ring + b * kRW * kChunk * kPitch + qp;
            uint32_t todo = live ? gmask[(b * kG + g) * kP + qp] : 0u;
            // The ring words of the lane's next unit are read while this one
            // plays (pair 1: w1 | w3).
            int32_t k = todo ? __ffs((int)todo) - 1 : 0;
            uint2 v = todo ? rb[(1 * kChunk + k) * kPitch] : make_uint2(0u, 0u);
            while (todo) {
                todo &= todo - 1;
                const int32_t kn = todo ? __ffs((int)todo) - 1 : k;
                const uint2 nv = rb[(1 * kChunk + kn) * kPitch];
                const uint32_t r1 = v.x, r3 = v.y;
                const int32_t d = (int32_t)(r3 & 31u);
                if (!kReclaim) {
                    const int32_t t = d / kG;
                    Q q = queue[t * kRow];
                    uint32_t n = nres[t * kRow];
                    uint32_t u_d = used[t * kRow];
                    bool missed;
                    uint2 w = settle_lru<Q>(q, n, u_d, (uint32_t)cap[d], r1, r3, weight, load, D, dp.err, missed);
                    if (kPhi && missed) {  // a reload of a model this device held before: bit 31 of the load word
                        const uint32_t m = (r3 >> 5) & 15u, e = everl[t * kRow];
                        w.x |= ((e >> m) & 1u) << 31;
                        everl[t * kRow] = (uint16_t)(e | (1u << m));
                    }
                    queue[t * kRow] = q;
                    nres[t * kRow] = (uint8_t)n;
                    used[t * kRow] = u_d;
                    rb[(1 * kChunk + k) * kPitch] = w;
                } else {
                    // Reclamation by next use: victims one at a time, a copy
                    // also resident elsewhere first, then the largest (next
                    // use - position) / reload cost (no next use or a free
                    // reload: infinite), then the least recently used.
                    const uint32_t m = (r3 >> 5) & 15u;
                    Q q = queue[d * kRow];
                    uint32_t n = nres[d * kRow];
                    uint32_t u_d = used[d * kRow];  // used + need <= cap + peak < 2^32
                    const uint32_t wm = (uint32_t)weight[m];
                    const uint32_t capd = (uint32_t)cap[d];
                    const bool was_empty = n == 0;
                    const int32_t kq = Lru<Q>::find(q, n, m);
                    const bool hit = kq < (int32_t)n;
                    q = hit ? Lru<Q>::remove(q, hit ? kq : 0) : q;  // (an index below the queue length)
                    n -= hit ? 1u : 0u;
                    const uint32_t need = hit ? r1 : wm + r1;
                    const int32_t here = c * kChunk + k;
                    while (u_d + need > capd && n > 0) {
                        // The class (redundant << 1 | infinite) ranks first; within
                        // a finite class the larger distance per unit of cost
                        // (32-bit factors, exact 64-bit products); ties keep the
                        // earlier queue entry.
                        int32_t best = 0;
                        uint32_t bcls = 0;
                        int32_t bdist = 0, bcost = 0;
                        // (Unrolled over the queue's capacity, so the entries'
                        // loads are not chained through the loop counter.)
#pragma unroll
                        for (int32_t e = 0; e < Lru<Q>::kSlots; ++e) {
                            if (e >= (int32_t)n) break;
                            const uint32_t kk = (uint32_t)(q >> (4 * e)) & 15u;
                            const uint32_t red = rcnt[kk * kP] > 1;
                            const uint32_t nu = nuse[(d * M + kk) * kP];
                            const int32_t cost = load[kk * D + d];
                            const uint32_t inf = nu == 0xFFFFu || cost == 0;
                            const uint32_t cls = (red << 1) | inf;
                            const int32_t dist = (int32_t)nu - here;
                            if (e == 0 || cls > bcls ||
                                (cls == bcls && !inf && (int64_t)dist * bcost > (int64_t)bdist * cost)) {
                                best = e; bcls = cls; bdist = dist; bcost = cost;
                            }
                        }
                        const uint32_t victim = (uint32_t)(q >> (4 * best)) & 15u;
                        u_d -= (uint32_t)weight[victim];
                        rcnt[victim * kP] -= 1;
                        q = Lru<Q>::remove(q, best);
                        n -= 1;
                    }
                    if (u_d + need > capd) atomicExch(dp.err, 2);  // unreachable for a valid plan
                    if (!hit) rcnt[m * kP] += 1;
                    nuse[(d * M + m) * kP] = (uint16_t)rb[(3 * kChunk + k) * kPitch].x;
                    q |= (Q)m << (4 * n);  // the unit's model is now the most recently used
                    n += 1;
                    u_d += hit ? 0u : wm;
                    uint32_t emptied = 0;
                    if ((r3 >> 10) & 1u) {  // retain bit 0: reclaim at the end of the unit
                        q &= ~((Q)0xF << (4 * (n - 1)));
                        n -= 1;
                        u_d -= wm;
                        emptied = n == 0;
                        rcnt[m * kP] -= 1;
                    }
                    queue[d * kRow] = q;
                    nres[d * kRow] = (uint8_t)n;
                    used[d * kRow] = u_d;
                    uint32_t reload = 0;
                    if (kPhi && !hit) {
                        const uint32_t e = everl[d * kRow];
                        reload = ((e >> m) & 1u) << 31;
                        everl[d * kRow] = (uint16_t)(e | (1u << m));
                    }
                    rb[(1 * kChunk + k) * kPitch] =
                        make_uint2(hit ? 0u : ((uint32_t)load[m * D + d] | reload),
                                   (r3 & ~(kPrefetch | kWasEmpty)) | (hit ? 0u : (r3 & kPrefetch)) |
                                       (was_empty ? kWasEmpty : 0u) | (emptied ? kEmptied : 0u));
                }
                k = kn;
                v = nv;
            }
            named_arrive(kFullR + b, kResThreads + 32);
        }
        if (live) {  // devices still occupied at the end
            uint32_t o = 0;
            for (int32_t t = 0; t * kG + g < D; ++t) o += nres[t * kRow] != 0;
            if (o) atomicAdd(open + qp, o);
        }
        named_arrive(kOpen, kResThreads + 32);
    } else {
    // ---------------- timing: lane = plan (Eq. 2, 5, 7, 10) ----------------
    const bool mine = lane < kP;  // lanes at or beyond kP own no plan and touch no per-plan state
    const int64_t p = (mine && lane < ng) ? (in_list ? (int64_t)in_list[j0 + lane] : j0 + lane) : 0;
    const bool live = mine && lane < ng && out.status[p] == 0;
    SlotArr<TT, ST, kP> slots;
    if constexpr (SlotBytes<ST>::kHi) {
        slots.lo = (uint32_t *)(sm + L.slots) + lane;
        slots.hi = sm + L.slots_hi + lane;
    } else {
        slots.v = (TT *)(sm + L.slots) + lane;
    }
    TT *tfree = (TT *)(sm + L.tfree) + lane;
    if (mine) {
        for (int32_t k = 0; k < dp.nslots + 2; ++k) slots.set(k, 0);
        for (int32_t d = 0; d < D; ++d) tfree[d * kP] = 0;
    }
    __syncthreads();
    const uint32_t trash = (uint32_t)dp.nslots;
    // u32 times: a plan is handed on when a sum carries out, or when a finish
    // reaches 2^32 - 1 (which a saturated w0 forces).  u64 times cannot wrap;
    // only a saturated w0 is handed on.
    TT end = 0;
    uint32_t ovf = 0;
    int64_t gsum = 0;
    uint32_t ph_timely = 0;  // Eq. 12 window terms (kPhi)
    uint64_t ph_life = 0;
    // Relative times (kRel): the base, the base saturated to 32 bits (for the
    // arrivals), emptied minus newly occupied devices so far (gsum counts
    // from the base), and the rebases so far.
    uint64_t base = 0;
    uint32_t bc = 0;
    int32_t net = 0, nreb = 0;
    const int64_t rcol = (int64_t)blockIdx.x * kP + lane, rstride = (int64_t)gridDim.x * kP;
    for (int32_t c = 0; c < chunks; ++c) {
        const int b = c % kBuffers;
        named_sync(kFullR + b, kResThreads + 32);
        if constexpr (kRel) {
            // Raise the base of every plan whose end nears 2^32.  The whole
            // warp walks the CTA's slot words ([slot][plan], 32 at a time,
            // word x of plan x % kP), each lowered by its plan's rise.
            if (__any_sync(0xFFFFFFFFu, live && !ovf && end > kRebaseAt)) {
                uint32_t m = 0xFFFFFFFFu;
                if (live && !ovf)
                    for (int32_t d = 0; d < D; ++d) m = min(m, tfree[d * kP]);
                const uint32_t dl = live && !ovf && m > kRebaseMin ? m - 1 : 0u;
                uint32_t *sw = (uint32_t *)(sm + L.slots);
                __syncwarp();  // every lane's slot writes are seen by the others
                const int32_t nw = W * kP, nall = (dp.nslots + 2) * kP;
                for (int32_t x0 = 0; x0 < nw; x0 += 32) {  // session slots: keep what falls below the base
                    const int32_t x = x0 + lane, q = x % kP;
                    const uint32_t dq = __shfl_sync(0xFFFFFFFFu, dl, q);
                    const uint64_t bq = __shfl_sync(0xFFFFFFFFu, base, q);
                    const int32_t rq = __shfl_sync(0xFFFFFFFFu, nreb, q);
                    if (x < nw && dq) {
                        const uint32_t v = sw[x];
                        uint64_t *r = dp.rel_ret + (int64_t)(x / kP) * rstride + (int64_t)blockIdx.x * kP + q;
                        const uint64_t keep = v && v <= dq ? bq + v : 0ull;
                        *r = rq ? max(*r, keep) : keep;
                        sw[x] = v > dq ? v - dq : 0u;
                    }
                }
                for (int32_t x0 = nw; x0 < nall; x0 += 32) {
                    const int32_t x = x0 + lane;
                    const uint32_t dq = __shfl_sync(0xFFFFFFFFu, dl, x % kP);
                    if (x < nall && dq) {
                        const uint32_t v = sw[x];
                        sw[x] = v > dq ? v - dq : 0u;
                    }
                }
                if (dl) {
                    for (int32_t d = 0; d < D; ++d) tfree[d * kP] -= dl;
                    end -= dl;
                    gsum -= (int64_t)net * dl;
                    base += dl;
                    bc = base < 0xFFFFFFFFull ? (uint32_t)base : 0xFFFFFFFFu;
                    ++nreb;
                }
                __syncwarp();
            }
        }
        const uint2 *rb = ring + b * kRW * kChunk * kPitch + lane;
        const int32_t kmax = min(kChunk, N - c * kChunk);
        if (live) {
            // The ring words of the next position are read while this one plays.
            uint2 w[3];
#pragma unroll
            for (int x = 0; x < 3; ++x) w[x] = rb[(x * kChunk) * kPitch];
            for (int32_t k = 0; k < kmax; ++k) {
                const int32_t kn = k + 1 < kmax ? k + 1 : k;
                uint2 nw[3];
#pragma unroll
                for (int x = 0; x < 3; ++x) nw[x] = rb[(x * kChunk + kn) * kPitch];
                const uint32_t r3 = w[1].y;
                if (!(r3 & kSkip)) {
                    const uint32_t run = w[0].x, arr = kRel ? max(w[0].y, bc) - bc : w[0].y, r4 = w[2].x,
                                   r5 = w[2].y;
                    const uint32_t ld = kPhi ? w[1].x & 0x7FFFFFFFu : w[1].x;  // bit 31: a reload (kPhi)
                    TT *tf_d = tfree + (r3 & 31u) * kP;
                    // Release (Eq. 2, Eq. 7); an accumulator slot is reset by its reader.
                    const uint32_t rs = r5 >> 16;
                    const TT rel = max((TT)arr, slots.get(rs & 0x7FFFu));
                    slots.set((rs & 0x8000u) ? (rs & 0x7FFFu) : trash, 0);
                    // A miss loads on this device first (ld > 0 only on a miss); a
                    // prefetched load waits only for the arrival (Eq. 5).  On a hit
                    // the residency stage cleared the prefetch bit and ld is 0.
                    const TT tf = *tf_d;
                    const TT ls = max(tf, (r3 & kPrefetch) ? (TT)arr : rel);
                    const TT le = ls + ld;
                    const TT start = max(le, rel);
                    if (kPhi) {
                        // A prefetched load (the bit survives residency only on a
                        // miss) that starts before the release and ends by it is
                        // timely; every unit adds the delay its load puts on its
                        // start, and a reload its load time.
                        ph_timely += (r3 & kPrefetch) && ls < rel && le <= rel;
                        ph_life += (uint64_t)(start - max(tf, rel)) + (w[1].x >> 31 ? (uint64_t)ld : 0ull);
                    }
                    const TT cfin = start + run;
                    if (kNarrow) ovf |= (le < ls) | (cfin < start);
                    else ovf |= run == kRunCap;
                    end = max(end, cfin);
                    if (r3 & kWasEmpty) {  // an empty device becomes occupied
                        gsum -= (int64_t)ls;
                        if (kRel) --net;
                    }
                    if (r3 & kEmptied) {  // the device empties after the unit
                        gsum += (int64_t)cfin;
                        if (kRel) ++net;
                    }

                    publish<TT>(slots, r3 >> 16, cfin);  // the sink when the unit writes nothing
                    publish<TT>(slots, r4 & 0xFFFFu, cfin);
                    const uint32_t nwl = (r3 >> 11) & 7u;
                    if (nwl > 2) {
                        publish<TT>(slots, r4 >> 16, cfin);
                        if (nwl == 4) {
                            publish<TT>(slots, r5 & 0xFFFFu, cfin);
                        } else if (nwl > 4) {  // five or more codes: the list from global memory
                            const int4 wr = __ldg(dp.noderec + 2 * (int32_t)(r5 & 0xFFFFu) + 1);
                            for (int32_t e = 3; e < wr.y; ++e) publish<TT>(slots, __ldg(dp.wl + wr.x + e), cfin);
                        }
                    }
                    *tf_d = cfin;
                }
#pragma unroll
                for (int x = 0; x < 3; ++x) w[x] = nw[x];
            }
        }
        // Once every plan of the CTA has left 32 bits, the producers stop
        // loading (they see the flag a chunk or two later).
        if (kNarrow && __all_sync(0xFFFFFFFFu, !live || ovf) && lane == 0) *gave_up = 1;
        named_arrive(kEmpty + b, kProdThreads + 32);  // buffer b may be refilled
    }
    if (kNarrow) ovf |= end == (TT)kRunCap;
    named_sync(kOpen, kResThreads + 32);  // the residency stage's final device counts
    const uint32_t bad = live ? open[lane] >> kOpenBad : 0u;  // placement bits found by the producers
    if (bad) {  // an invalid plan: its status bits and INT64_MAX metrics
        out.status[p] = bad;
        out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
        if (kPhi) dp.phi_timely[p] = dp.phi_life[p] = WF_INF64;
    } else if (live && ovf) {  // handed to the next path
        const int32_t kk = atomicAdd(ovf_count, 1);
        ovf_list[kk] = (int32_t)p;
    } else if (live && kRel) {
        // Back to absolute times: the session latencies as 64-bit values in
        // slot pairs (written from the last session down, so that no pair
        // overwrites a session slot not yet read).
        const int64_t nopen = open[lane];
        const uint64_t eabs = base + end;
        const PairArr<kP> lat{(uint32_t *)(sm + L.slots) + lane};
        for (int32_t w = W - 1; w >= 0; --w) {
            const uint32_t v = slots.get(w);
            uint64_t cw = v ? base + v : 0ull;
            if (nreb) cw = max(cw, dp.rel_ret[(int64_t)w * rstride + rcol]);
            lat.set(w, cw - arrival[w]);
        }
        out.makespan_us[p] = (int64_t)eabs - dp.first_arrival;
        out.gpu_us[p] = gsum + (int64_t)net * (int64_t)base + nopen * (int64_t)eabs;
        if (W <= kLaneSelect) out.p95_us[p] = (int64_t)select_slots<uint64_t>(lat, W, rank);
    } else if (live) {
        const int64_t nopen = open[lane];
        for (int32_t w = 0; w < W; ++w) slots.set(w, slots.get(w) - arrival[w]);  // session completion latency
        out.makespan_us[p] = (int64_t)end - dp.first_arrival;
        out.gpu_us[p] = gsum + nopen * (int64_t)end;
        if (W <= kLaneSelect) out.p95_us[p] = (int64_t)select_slots<TT>(slots, W, rank);
        if (kPhi) {
            dp.phi_timely[p] = ph_timely;
            dp.phi_life[p] = (int64_t)ph_life;
        }
    }
    // A plan whose p95 is still to be selected (more than kLaneSelect sessions).
    if (mine) open[lane] = live && !bad && !ovf && W > kLaneSelect;
    }
    __syncthreads();  // every stage is done with the group
    // The p95 of every plan played to the end with more than kLaneSelect
    // sessions (Section 4.2, nearest rank): the whole CTA, a warp per plan,
    // over the session latencies the timing stage left in the plan's slots.
    for (int q = warp; q < kP && W > kLaneSelect; q += S::kWarps) {
        if (!open[q]) continue;
        uint64_t v;
        if constexpr (kRel) {
            v = warp_select(PairArr<kP>{(uint32_t *)(sm + L.slots) + q}, W, rank);
        } else {
            SlotArr<TT, ST, kP> sq;
            if constexpr (SlotBytes<ST>::kHi) {
                sq.lo = (uint32_t *)(sm + L.slots) + q;
                sq.hi = sm + L.slots_hi + q;
            } else {
                sq.v = (TT *)(sm + L.slots) + q;
            }
            v = warp_select(sq, W, rank);
        }
        if (lane == 0) out.p95_us[in_list ? (int64_t)in_list[j0 + q] : j0 + q] = (int64_t)v;
    }
    __syncthreads();  // the group's shared state is free for the next group
  }
}

// ---------------------------------------------------------------------------
// Replica batch limit B_q (Eq. 11 over the running units, Section 3.5; the
// reading of the oracle's simulate_batched): the same producer warps build
// the unit records, and one play warp (lane = plan) settles each unit's
// admission and timing together -- under the limit an admission waits for
// running units to end, so residency cannot be settled ahead of the times.
// Per plan and device: the current replica's model, up to B_q slots (end
// time, KV), the last admission, residency stamps (dispatch position + 1 of
// the last use, 0 = not resident), resident weights and count, and the
// occupancy interval; 64-bit times, finish slots as in the sweep.
// ---------------------------------------------------------------------------
constexpr int kBqPlans = 8;                        // plans per CTA (play lanes)
constexpr int kBqProducers = kBqPlans / kPlansPerIter;  // one plan pair per producer warp
constexpr int kBqWarps = 1 + kBqProducers;
constexpr int kBqBuffers = 4;
constexpr int kBqPitch = kBqPlans | 1;
constexpr int kBqFull = 1, kBqEmpty = kBqFull + kBqBuffers;  // named barriers
static_assert(kBqEmpty + kBqBuffers <= 16, "named barriers");

struct BqLayout {
    uint32_t weight, cap, load, arr, ring, slots, stamp, se, sk, used, nres, cur, adm, occ, gpu, open, total;
};

__host__ __device__ inline BqLayout bq_layout(int32_t D, int32_t M, int32_t W, int32_t B, int32_t NS)
{
    constexpr uint32_t P = kBqPlans;
    BqLayout l;
    uint32_t o = 0;
    l.weight = o; o += round16(4u * M);
    l.cap = o; o += round16(4u * D);
    l.load = o; o += round16(4u * M * D);
    l.arr = o; o += round16(4u * W);
    l.ring = o; o += 8u * kBqBuffers * 3 * kChunk * kBqPitch;
    l.slots = o; o += 8u * (uint32_t)NS * P;
    l.stamp = o; o += 4u * D * M * P;
    l.se = o; o += 8u * D * B * P;
    l.sk = o; o += round16(4u * D * B * P);
    l.used = o; o += 4u * D * P;
    l.nres = o; o += 4u * D * P;
    l.cur = o; o += round16(4u * D * P);
    l.adm = o; o += 8u * D * P;
    l.occ = o; o += 8u * D * P;
    l.gpu = o; o += 8u * D * P;
    l.open = o; o += 16u * ((P + 3) / 4);
    l.total = o;
    return l;
}

__global__ void __launch_bounds__(32 * kBqWarps)
bq_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, int32_t *ovf_list, int32_t *ovf_count)
{
    constexpr int kP = kBqPlans, kPitch = kBqPitch;
    constexpr int kProdThreads = 32 * kBqProducers;
    extern __shared__ __align__(128) uint8_t sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W, B = dp.batch;
    const BqLayout L = bq_layout(D, M, W, B, dp.nslots + 2);
    const int64_t j0 = (int64_t)blockIdx.x * kP;
    const int ng = (int)(pl.P - j0 < kP ? pl.P - j0 : kP);
    uint2 *ring = (uint2 *)(sm + L.ring);
    const int32_t chunks = (N + kChunk - 1) / kChunk;
    int32_t *weight = (int32_t *)(sm + L.weight);
    int32_t *cap = (int32_t *)(sm + L.cap);
    int32_t *load = (int32_t *)(sm + L.load);
    uint32_t *arrival = (uint32_t *)(sm + L.arr);
    uint32_t *open = (uint32_t *)(sm + L.open);  // placement status bits from the producers (bit kOpenBad on)
    for (int32_t k = threadIdx.x; k < M; k += blockDim.x) weight[k] = __ldg(dp.weight + k);
    for (int32_t k = threadIdx.x; k < D; k += blockDim.x) cap[k] = __ldg(dp.cap + k);
    for (int32_t k = threadIdx.x; k < M * D; k += blockDim.x) load[k] = __ldg(dp.load + k);
    for (int32_t k = threadIdx.x; k < W; k += blockDim.x) arrival[k] = (uint32_t)__ldg(dp.arrival + k);
    if (threadIdx.x < kP) open[threadIdx.x] = 0;

    if (warp >= 1) {
        // ---------------- producers: lane = dispatch position (as in pc_kernel) ----------------
        __syncthreads();
        const int pw = warp - 1;
        const int pos = lane % kChunk, sub = lane / kChunk;
        const int q = pw * kPlansPerIter + sub;  // one plan per half-warp
        RowPtrs rp[1];
        int qq[1] = {q};
        bool ok = q < ng;
        rp[0].place = nullptr;
        rp[0].order = nullptr;
        rp[0].boff = 0;
        if (ok) {
            const int64_t pq = j0 + q;
            ok = __ldg(out.status + pq) == 0;
            rp[0].place = pl.place + pq * pl.place_stride;
            rp[0].order = (const uint16_t *)((const uint8_t *)pl.order + pq * pl.order_stride);
            rp[0].boff = pq * pl.bits_stride;
        }
        const uint32_t place_bytes = (uint32_t)((N + 15) & ~15), bits_bytes = (uint32_t)((((N + 31) >> 5) * 4 + 15) & ~15);
        if (pos == 0 && ok) {
            l2_prefetch(rp[0].place, place_bytes);
            l2_prefetch(bits_row(pl.fuse, rp[0].boff), bits_bytes);
            l2_prefetch(bits_row(pl.prefetch, rp[0].boff), bits_bytes);
        }
        int32_t h0[1] = {ok && pos < N ? (int32_t)__ldg(rp[0].order + pos) : 0};
        for (int32_t c = 0; c < chunks; ++c) {
            const int b = c % kBqBuffers;
            if (c >= kBqBuffers) named_sync(kBqEmpty + b, kProdThreads + 32);  // the play warp released buffer b
            uint2 *rb = ring + b * 3 * kChunk * kPitch;
            const int32_t i = c * kChunk + pos;
            const int32_t h1 = ok && i + kChunk < N ? (int32_t)__ldg(rp[0].order + i + kChunk) : 0;
            bool act[1] = {ok && i < N};
            uint32_t dev[1];
            produce_batch<1, kPitch>(dp, pl, rp, act, h0, rb, pos, qq, dev, open);
            h0[0] = h1;
            named_arrive(kBqFull + b, kProdThreads + 32);  // buffer b is full
        }
        for (int32_t c = chunks; c < chunks + kBqBuffers; ++c)
            if (c >= kBqBuffers) named_sync(kBqEmpty + c % kBqBuffers, kProdThreads + 32);
        return;
    }

    // ---------------- play: lane = plan (admission and timing together) ----------------
    const int q = lane;
    const bool mine = q < kP;
    const int64_t p = j0 + q;
    const bool live = mine && q < ng && out.status[p] == 0;
    SlotArr<uint64_t, uint64_t, kP> slots;
    slots.v = (uint64_t *)(sm + L.slots) + q;
    uint32_t *stamp = (uint32_t *)(sm + L.stamp) + q;  // [d][m]
    uint64_t *se = (uint64_t *)(sm + L.se) + q;        // [d][slot]
    int32_t *sk = (int32_t *)(sm + L.sk) + q;          // [d][slot]
    int32_t *used = (int32_t *)(sm + L.used) + q;
    int32_t *nres = (int32_t *)(sm + L.nres) + q;
    int32_t *cur = (int32_t *)(sm + L.cur) + q;
    uint64_t *ladm = (uint64_t *)(sm + L.adm) + q;
    uint64_t *occ = (uint64_t *)(sm + L.occ) + q;
    uint64_t *gpu = (uint64_t *)(sm + L.gpu) + q;
    constexpr uint64_t kIdle = ~0ull;  // no occupancy interval open
    if (mine) {
        for (int32_t k = 0; k < dp.nslots + 2; ++k) slots.set(k, 0);
        for (int32_t k = 0; k < D * M; ++k) stamp[k * kP] = 0;
        for (int32_t k = 0; k < D * B; ++k) { se[k * kP] = 0; sk[k * kP] = 0; }
        for (int32_t d = 0; d < D; ++d) {
            used[d * kP] = 0; nres[d * kP] = 0; cur[d * kP] = -1;
            ladm[d * kP] = 0; occ[d * kP] = kIdle; gpu[d * kP] = 0;
        }
    }
    __syncthreads();
    const uint32_t trash = (uint32_t)dp.nslots;
    uint64_t end = 0;
    uint32_t ovf = 0;
    // The least recently used idle model of device d other than m (-1: none).
    auto victim_of = [&](int32_t d, uint32_t m) -> int32_t {
        int32_t v = -1;
        uint32_t vs = 0xFFFFFFFFu;
        for (int32_t k = 0; k < M; ++k) {
            const uint32_t s = stamp[(d * M + k) * kP];
            if ((uint32_t)k != m && s != 0 && s < vs) { vs = s; v = k; }
        }
        return v;
    };
    for (int32_t c = 0; c < chunks; ++c) {
        const int b = c % kBqBuffers;
        named_sync(kBqFull + b, kProdThreads + 32);
        const uint2 *rb = ring + b * 3 * kChunk * kPitch + q;
        const int32_t kmax = min(kChunk, N - c * kChunk);
        for (int32_t k = 0; live && k < kmax; ++k) {
            const uint2 w0 = rb[(0 * kChunk + k) * kPitch], w1 = rb[(1 * kChunk + k) * kPitch],
                        w2 = rb[(2 * kChunk + k) * kPitch];
            const uint32_t r3 = w1.y;
            if (r3 & kSkip) continue;
            const int32_t d = (int32_t)(r3 & 31u);
            const uint32_t m = (r3 >> 5) & 15u;
            const uint64_t arr = w0.y, run = w0.x;  // run includes the grant
            const int64_t kv = (int32_t)w1.x;
            const uint32_t r4 = w2.x, r5 = w2.y;
            ovf |= w0.x == kRunCap;  // a saturated chain run: the int64 path
            // Release (Eq. 2, Eq. 7); an accumulator slot is reset by its reader.
            const uint32_t rs = r5 >> 16;
            const uint64_t rel = max(arr, slots.get(rs & 0x7FFFu));
            slots.set((rs & 0x8000u) ? (rs & 0x7FFFu) : trash, 0);
            const int64_t capd = cap[d], wm = weight[m];
            uint64_t *sed = se + d * B * kP;
            int32_t *skd = sk + d * B * kP;
            int64_t u_d = used[d * kP];
            uint64_t adm, start;
            int32_t slot = 0;
            if ((int32_t)m == cur[d * kP]) {
                // Join the current replica: the slot that frees first, no
                // earlier than the last admission (dispatch order), and Eq.
                // 11 with the running units' KV; idle models go first, then
                // the admission waits for the next running unit to end.
                for (int32_t j = 1; j < B; ++j)
                    if (sed[j * kP] < sed[slot * kP]) slot = j;
                adm = max(max(rel, sed[slot * kP]), ladm[d * kP]);
                for (;;) {
                    int64_t running = 0;
                    for (int32_t j = 0; j < B; ++j) running += sed[j * kP] > adm ? skd[j * kP] : 0;
                    while (u_d + running + kv > capd) {
                        const int32_t v = victim_of(d, m);
                        if (v < 0) break;
                        u_d -= weight[v];
                        nres[d * kP] -= 1;
                        stamp[(d * M + v) * kP] = 0;
                    }
                    if (u_d + running + kv <= capd) break;
                    uint64_t next = ~0ull;  // the next running unit to end
                    for (int32_t j = 0; j < B; ++j)
                        if (sed[j * kP] > adm && sed[j * kP] < next) next = sed[j * kP];
                    if (next == ~0ull) { atomicExch(dp.err, 2); break; }  // unreachable for a valid plan
                    adm = next;
                }
                start = adm;
            } else {
                // Another model: the device drains, then the unit hits or loads.
                uint64_t drain = 0;
                for (int32_t j = 0; j < B; ++j) drain = max(drain, sed[j * kP]);
                const bool hit = stamp[(d * M + m) * kP] != 0;
                const int64_t need = hit ? kv : wm + kv;
                while (u_d + need > capd) {
                    const int32_t v = victim_of(d, m);
                    if (v < 0) { atomicExch(dp.err, 2); break; }  // unreachable for a valid plan
                    u_d -= weight[v];
                    nres[d * kP] -= 1;
                    stamp[(d * M + v) * kP] = 0;
                }
                uint64_t ready;
                if (hit) {
                    adm = start = max(drain, rel);
                    ready = drain;
                } else {
                    const uint64_t ls = max(drain, (r3 & kPrefetch) ? arr : rel);
                    if (occ[d * kP] == kIdle) occ[d * kP] = ls;
                    u_d += wm;
                    nres[d * kP] += 1;
                    const uint64_t le = ls + (uint64_t)load[m * D + d];
                    adm = ls;
                    start = max(le, rel);
                    ready = le;
                }
                for (int32_t j = 0; j < B; ++j) { sed[j * kP] = ready; skd[j * kP] = 0; }
                cur[d * kP] = (int32_t)m;
            }
            const uint64_t cfin = start + run;
            publish<uint64_t>(slots, r3 >> 16, cfin);  // the sink when the unit writes nothing
            publish<uint64_t>(slots, r4 & 0xFFFFu, cfin);
            const uint32_t nwl = (r3 >> 11) & 7u;
            if (nwl > 2) {
                publish<uint64_t>(slots, r4 >> 16, cfin);
                if (nwl == 4) {
                    publish<uint64_t>(slots, r5 & 0xFFFFu, cfin);
                } else if (nwl > 4) {  // five or more codes: the list from global memory
                    const int4 wr = __ldg(dp.noderec + 2 * (int32_t)(r5 & 0xFFFFu) + 1);
                    for (int32_t e = 3; e < wr.y; ++e) publish<uint64_t>(slots, __ldg(dp.wl + wr.x + e), cfin);
                }
            }
            sed[slot * kP] = cfin;
            skd[slot * kP] = (int32_t)kv;
            ladm[d * kP] = adm;
            stamp[(d * M + m) * kP] = (uint32_t)(c * kChunk + k) + 1u;
            end = max(end, cfin);
            if ((r3 >> 10) & 1u) {  // retain bit 0 (B_q = 1 only): the model leaves after the unit
                u_d -= wm;
                nres[d * kP] -= 1;
                stamp[(d * M + m) * kP] = 0;
                cur[d * kP] = -1;
                if (nres[d * kP] == 0) {
                    gpu[d * kP] += cfin - occ[d * kP];
                    occ[d * kP] = kIdle;
                }
            }
            used[d * kP] = (int32_t)u_d;
        }
        named_arrive(kBqEmpty + b, kProdThreads + 32);  // buffer b may be refilled
    }
    if (!live) return;
    const uint32_t bad = open[q] >> kOpenBad;  // placement bits found by the producers
    if (bad) {
        out.status[p] = bad;
        out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
    } else if (ovf) {
        ovf_list[atomicAdd(ovf_count, 1)] = (int32_t)p;
    } else {
        int64_t g = 0;
        for (int32_t d = 0; d < D; ++d)
            g += (int64_t)gpu[d * kP] + (occ[d * kP] != kIdle ? (int64_t)(end - occ[d * kP]) : 0);
        for (int32_t w = 0; w < W; ++w) slots.set(w, slots.get(w) - arrival[w]);  // session completion latency
        const int32_t rank = (int32_t)((95 * (int64_t)W + 99) / 100 - 1);
        out.makespan_us[p] = (int64_t)end - dp.first_arrival;
        out.gpu_us[p] = g;
        out.p95_us[p] = (int64_t)select_slots<uint64_t>(slots, W, rank);
    }
}

// ---------------------------------------------------------------------------
// Stochastic latencies (row a11): one plan per CTA.  Model residency does not
// depend on times, so one residency lane settles it for every sample; the
// timing warps play kSamples samples at once (lane = sample), each drawing
// its run-time multipliers from (plan, sample, node) through SplitMix64 and
// the integer Box-Muller tables; then the CTA reduces the floor means and the
// pooled nearest-rank p95 over samples x sessions.
// ---------------------------------------------------------------------------
constexpr int kSamples = 64;                  // timing lanes (two warps)
constexpr int kSBuffers = 3;                  // record ring buffers
constexpr int kSChunk = 32;                   // positions per chunk (one producer warp)
constexpr int kSRec = kRecWords + 1;          // + head node
constexpr int kSWarps = kSamples / 32 + 2;    // timing warps, residency warp, producer warp
constexpr int kSTiming = kSamples;            // threads of the timing stage
// Named barriers of this kernel (ids reuse those of the deterministic one).
constexpr int kSFullP = 1, kSFullR = kSFullP + kSBuffers, kSEmpty = kSFullR + kSBuffers, kSOpen = kSEmpty + kSBuffers,
              kSRed = kSOpen + 1;

struct StochLayout {
    uint32_t weight, cap, load, arr, ring, slots, tfree, used, queue, nres, hist, red, total;
};

__host__ __device__ inline StochLayout stoch_layout(int32_t D, int32_t M, int32_t W, int32_t NS)
{
    StochLayout l;
    uint32_t o = 0;
    l.weight = o; o += round16(4u * M);
    l.cap = o; o += round16(4u * D);
    l.load = o; o += round16(4u * M * D);
    l.arr = o; o += round16(4u * W);
    l.ring = o; o += 4u * kSBuffers * kSRec * kSChunk;
    l.slots = o; o += 4u * (uint32_t)NS * kSamples;
    l.tfree = o; o += 4u * D * kSamples;
    l.used = o; o += round16(4u * D);
    l.queue = o; o += 8u * D;
    l.nres = o; o += round16((uint32_t)D);
    l.hist = o; o += 4u * 256 + 16;
    l.red = o; o += 8u * 2 * kSamples + 16;
    l.total = o;
    return l;
}

__device__ __forceinline__ uint64_t splitmix64(uint64_t x)
{
    x += 0x9E3779B97F4A7C15ull;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ull;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBull;
    return x ^ (x >> 31);
}

// BT: the element type of the radius and angle tables read per sample
// (int16 copies when every value fits, else the int32 tables).
template <typename Q, typename BT>
__global__ void __launch_bounds__(32 * kSWarps)
stoch_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out, int32_t *ovf_list, int32_t *ovf_count)
{
    extern __shared__ __align__(128) uint8_t sm[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int32_t N = dp.N, D = dp.D, M = dp.M, W = dp.W, S = dp.S;
    const StochLayout L = stoch_layout(D, M, W, dp.nslots + 2);
    const int64_t p = blockIdx.x;
    if (out.status[p] != 0) return;  // uniform over the CTA: the status kernel marked the plan invalid
    uint32_t *ring = (uint32_t *)(sm + L.ring);
    const int32_t chunks = (N + kSChunk - 1) / kSChunk;
    int32_t *weight = (int32_t *)(sm + L.weight);
    int32_t *cap = (int32_t *)(sm + L.cap);
    int32_t *load = (int32_t *)(sm + L.load);
    uint32_t *arrival = (uint32_t *)(sm + L.arr);
    for (int32_t k = threadIdx.x; k < M; k += blockDim.x) weight[k] = __ldg(dp.weight + k);
    for (int32_t k = threadIdx.x; k < D; k += blockDim.x) cap[k] = __ldg(dp.cap + k);
    for (int32_t k = threadIdx.x; k < M * D; k += blockDim.x) load[k] = __ldg(dp.load + k);
    for (int32_t k = threadIdx.x; k < W; k += blockDim.x) arrival[k] = (uint32_t)__ldg(dp.arrival + k);
    const int tw = kSTiming / 32;  // timing warps are 0 .. tw-1

    if (warp == tw + 1) {
        // ---------------- producer: lane = dispatch position ----------------
        __syncthreads();
        PlanPtrs r;
        r.place = pl.place + p * pl.place_stride;
        r.order = (const uint16_t *)((const uint8_t *)pl.order + p * pl.order_stride);
        r.fuse = (const uint32_t *)((const uint8_t *)pl.fuse + p * pl.bits_stride);
        r.prefetch = (const uint32_t *)((const uint8_t *)pl.prefetch + p * pl.bits_stride);
        r.retain = pl.retain ? (const uint32_t *)((const uint8_t *)pl.retain + p * pl.bits_stride) : nullptr;
        for (int32_t c = 0; c < chunks; ++c) {
            const int b = c % kSBuffers;
            if (c >= kSBuffers) named_sync(kSEmpty + b, kSTiming + 32);
            uint32_t *rb = ring + b * kSRec * kSChunk;
            const int32_t i = c * kSChunk + lane;
            uint32_t rec[kRecWords] = {0, 0, 0, kSkip, 0, 0};
            int32_t head = 0;
            if (i < N) produce(dp, r, i, rec, &head);
#pragma unroll
            for (int w = 0; w < kRecWords; ++w) rb[w * kSChunk + lane] = rec[w];
            rb[kRecWords * kSChunk + lane] = (uint32_t)head;
            named_arrive(kSFullP + b, 64);
        }
        for (int32_t c = chunks; c < chunks + kSBuffers; ++c)
            if (c >= kSBuffers) named_sync(kSEmpty + c % kSBuffers, kSTiming + 32);
        return;
    }

    if (warp == tw) {
        // ---------------- residency, once for all samples: lane = device ----------------
        // Residency is per device, so lane d owns device d's queue, weight
        // and count in registers and plays the chunk's units on d in
        // dispatch order; lanes of different devices run side by side.
        __syncthreads();
        Q q = 0;
        uint32_t n = 0, u_d = 0;
        const bool dev = lane < D;
        const uint32_t capd = dev ? (uint32_t)cap[lane] : 0u;
        for (int32_t c = 0; c < chunks; ++c) {
            const int b = c % kSBuffers;
            named_sync(kSFullP + b, 64);
            uint32_t *rb = ring + b * kSRec * kSChunk;
            const int32_t kmax = min(kSChunk, N - c * kSChunk);
            // The chunk's positions on each device: one ballot per device.
            const uint32_t r3l = lane < kmax ? rb[3 * kSChunk + lane] : kSkip;
            const int32_t dl = (r3l & kSkip) ? -1 : (int32_t)(r3l & 31u);
            uint32_t mine = 0;
            for (int32_t dd = 0; dd < D; ++dd) {
                const uint32_t bal = __ballot_sync(0xFFFFFFFFu, dl == dd);
                if (lane == dd) mine = bal;
            }
            while (mine) {
                const int32_t k = __ffs((int)mine) - 1;
                mine &= mine - 1;
                const uint32_t r3 = rb[3 * kSChunk + k];
                uint32_t &r1 = rb[1 * kSChunk + k];
                const uint32_t m = (r3 >> 5) & 15u;
                const uint32_t wm = (uint32_t)weight[m];
                const bool was_empty = n == 0;
                const int32_t kq = Lru<Q>::find(q, n, m);
                const bool hit = kq < (int32_t)n;
                q = hit ? Lru<Q>::remove(q, hit ? kq : 0) : q;  // (an index below the queue length)
                n -= hit ? 1u : 0u;
                const uint32_t need = hit ? r1 : wm + r1;
                uint32_t e = 0;
                while (u_d + need > capd && e < n) {
                    u_d -= (uint32_t)weight[(uint32_t)(q >> (4 * e)) & 15u];
                    ++e;
                }
                if (u_d + need > capd) atomicExch(dp.err, 2);  // unreachable for a valid plan
                q = e < (uint32_t)Lru<Q>::kSlots ? (q >> (4 * e)) : (Q)0;
                n -= e;
                q |= (Q)m << (4 * n);
                n += 1;
                u_d += hit ? 0u : wm;
                uint32_t emptied = 0;
                if ((r3 >> 10) & 1u) {
                    q &= ~((Q)0xF << (4 * (n - 1)));
                    n -= 1;
                    u_d -= wm;
                    emptied = n == 0;
                }
                r1 = (hit ? 1u : 0u) | (was_empty ? 2u : 0u) | (emptied << 2);
            }
            __syncwarp();
            named_arrive(kSFullR + b, kSTiming + 32);
        }
        uint32_t *hist = (uint32_t *)(sm + L.hist);
        // devices still occupied at the end (the same for every sample)
        const uint32_t open = __popc(__ballot_sync(0xFFFFFFFFu, dev && n != 0));
        if (lane == 0) hist[256] = open;
        named_arrive(kSOpen, kSTiming + 32);
        return;
    }

    // ---------------- timing: lane = sample ----------------
    const int t = threadIdx.x;  // 0 .. kSamples-1
    const bool live = t < S;
    uint32_t *slots = (uint32_t *)(sm + L.slots) + t;
    uint32_t *tfree = (uint32_t *)(sm + L.tfree) + t;
    for (int32_t k = 0; k < dp.nslots + 2; ++k) slots[k * kSamples] = 0;
    for (int32_t d = 0; d < D; ++d) tfree[d * kSamples] = 0;
    __syncthreads();
    const uint64_t key = splitmix64(splitmix64(dp.seed ^ (uint64_t)(pl.plan_base + p)) ^ (uint64_t)t);
    const uint64_t rmask = (uint64_t)(dp.bm_rn - 1), cmask = (uint64_t)(dp.bm_cn - 1);
    const int64_t zoff = (dp.bm_en - 1) >> 1;
    const BT *bmr, *bmc;
    if constexpr (sizeof(BT) == 2) { bmr = dp.bm_r16; bmc = dp.bm_c16; }
    else { bmr = dp.bm_r; bmc = dp.bm_c; }
    const uint32_t grant = (uint32_t)dp.grant;
    uint32_t end = 0, ovf = 0;
    int64_t gsum = 0;
    for (int32_t c = 0; c < chunks; ++c) {
        const int b = c % kSBuffers;
        named_sync(kSFullR + b, kSTiming + 32);
        const uint32_t *rb = ring + b * kSRec * kSChunk;
        const int32_t kmax = min(kSChunk, N - c * kSChunk);
        for (int32_t k = 0; k < kmax && live; ++k) {
            const uint32_t r3 = rb[3 * kSChunk + k];
            if (r3 & kSkip) continue;
            const uint32_t fl = rb[1 * kSChunk + k];
            const uint32_t arr = rb[2 * kSChunk + k];
            const uint32_t r4 = rb[4 * kSChunk + k];
            const uint32_t r5 = rb[5 * kSChunk + k];
            const int32_t d = (int32_t)(r3 & 31u);
            const uint32_t m = (r3 >> 5) & 15u;
            const bool hit = fl & 1u;
            // Sampled run time of the unit: every member's multiplier (Eq. 4 sum).
            const int32_t tail = (int32_t)(r5 & 0xFFFFu);
            uint64_t run = 0;
            for (int32_t j = (int32_t)rb[kRecWords * kSChunk + k];; j = (int32_t)(__ldg(dp.links + j) >> 16)) {
                const uint64_t hh = splitmix64(key ^ (uint64_t)j);
                const int64_t prod = (int64_t)__ldg(bmr + (hh & rmask)) * (int64_t)__ldg(bmc + ((hh >> 32) & cmask));
                const int64_t mult = __ldg(dp.bm_e + ((prod >> 18) + zoff));
                run += ((uint64_t)(uint32_t)__ldg(&dp.lk[j * D + d].x) * (uint64_t)mult + 32768u) >> 16;
                if (j == tail) break;
            }
            ovf |= run >> 32 ? 1u : 0u;
            uint32_t rel = arr;
            const uint32_t rs = r5 >> 16;
            if (rs != 0xFFFFu) {
                uint32_t &sv = slots[(rs & 0x7FFFu) * kSamples];
                rel = max(rel, sv);
                if (rs & 0x8000u) sv = 0;
            }
            const uint32_t tf = tfree[d * kSamples];
            const uint32_t ls = max(tf, ((r3 >> 9) & 1u) ? arr : rel);
            const uint32_t le = ls + (uint32_t)load[m * D + d];
            const uint32_t start = hit ? max(tf, rel) : max(le, rel);
            ovf |= (!hit && le < ls) ? 1u : 0u;
            gsum -= (!hit && (fl & 2u)) ? (int64_t)ls : 0;
            const uint32_t sg = start + grant;
            const uint32_t cfin = sg + (uint32_t)run;
            ovf |= (sg < start) | (cfin < sg);
            end = max(end, cfin);
            gsum += (fl & 4u) ? (int64_t)cfin : 0;
            const uint32_t nwl = (r3 >> 11) & 7u;
            uint32_t *sl = slots;
            if (nwl > 0) { uint32_t &sv = sl[((r3 >> 16) & 0x7FFFu) * kSamples]; sv = (r3 >> 31) ? max(sv, cfin) : cfin; }
            if (nwl > 1) { uint32_t &sv = sl[(r4 & 0x7FFFu) * kSamples]; sv = ((r4 >> 15) & 1u) ? max(sv, cfin) : cfin; }
            if (nwl > 2) {
                { uint32_t &sv = sl[((r4 >> 16) & 0x7FFFu) * kSamples]; sv = (r4 >> 31) ? max(sv, cfin) : cfin; }
                const int4 wr = __ldg(dp.noderec + 2 * tail + 1);
                for (int32_t e = 3; e < wr.y; ++e) {
                    const uint32_t code = __ldg(dp.wl + wr.x + e);
                    uint32_t &sv = sl[(code & 0x7FFFu) * kSamples];
                    sv = (code & 0x8000u) ? max(sv, cfin) : cfin;
                }
            }
            tfree[d * kSamples] = cfin;
        }
        named_arrive(kSEmpty + b, kSTiming + 32);
    }
    named_sync(kSOpen, kSTiming + 32);
    uint32_t *hist = (uint32_t *)(sm + L.hist);
    const int64_t open = hist[256];
    // Per-sample results, then the floor means and the pooled p95 over S x W.
    int64_t *red = (int64_t *)(sm + L.red);
    const int64_t mk = live ? (int64_t)end - dp.first_arrival : 0;
    const int64_t g = live ? gsum + open * (int64_t)end : 0;
    red[t] = mk;
    red[kSamples + t] = g;
    if (live) for (int32_t w = 0; w < W; ++w) slots[w * kSamples] -= arrival[w];
    uint32_t *flag = hist + 257;
    if (t == 0) *flag = 0;
    named_sync(kSRed, kSTiming);
    if (live && ovf) atomicOr(flag, 1u);
    named_sync(kSRed, kSTiming);
    if (*flag) {  // some sample's times do not fit u32: exact int64 path for the plan
        if (t == 0) ovf_list[atomicAdd(ovf_count, 1)] = (int32_t)p;
        return;
    }
    // Nearest-rank p95 of the pooled completions: radix select, 8 bits a pass.
    const int64_t n = (int64_t)S * W;
    uint32_t *meta = hist + 258;  // [0] prefix, [1] rank
    if (t == 0) { meta[0] = 0; meta[1] = (uint32_t)((95 * n + 99) / 100 - 1); }
    for (int shift = 24; shift >= 0; shift -= 8) {
        for (int k = t; k < 256; k += kSTiming) hist[k] = 0;
        named_sync(kSRed, kSTiming);
        const uint32_t hi = shift == 24 ? 0u : (~0u << (shift + 8));
        const uint32_t pre = meta[0];
        if (live)
            for (int32_t w = 0; w < W; ++w) {
                const uint32_t v = slots[w * kSamples];
                if ((v & hi) == pre) atomicAdd(&hist[(v >> shift) & 255u], 1u);
            }
        named_sync(kSRed, kSTiming);
        if (t == 0) {
            uint32_t r = meta[1];
            int bin = 0;
            while (hist[bin] <= r) { r -= hist[bin]; ++bin; }
            meta[1] = r;
            meta[0] |= (uint32_t)bin << shift;
        }
        named_sync(kSRed, kSTiming);
    }
    if (t == 0) {
        int64_t smk = 0, sg = 0;
        for (int k = 0; k < S; ++k) { smk += red[k]; sg += red[kSamples + k]; }
        out.makespan_us[p] = smk / S;
        out.gpu_us[p] = sg / S;
        out.p95_us[p] = (int64_t)meta[0];
    }
}

// Next use, for reclamation by next use: for every dispatch position i that
// starts a unit, the next position that starts a unit on the same device with
// the same model (0xFFFF: none).  A warp per plan walks its positions from the
// end, 32 at a time; lanes with equal (device, model) keys find each other
// with __match_any_sync, and a shared table carries the first occurrence of
// each key to the chunk before.
constexpr int kNuWarps = 4;

__global__ void __launch_bounds__(32 * kNuWarps)
nextuse_kernel(wf_dev_problem dp, wf_plans pl, const uint32_t *status, uint16_t *table)
{
    extern __shared__ __align__(16) uint8_t nsm[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int32_t N = dp.N, D = dp.D, M = dp.M;
    uint16_t *last = (uint16_t *)nsm + warp * D * M;
    for (int64_t p = (int64_t)blockIdx.x * kNuWarps + warp; p < pl.P; p += (int64_t)gridDim.x * kNuWarps) {
        if (__ldg(status + p) != 0) continue;  // uniform over the warp
        const uint8_t *place = pl.place + p * pl.place_stride;
        const uint16_t *order = (const uint16_t *)((const uint8_t *)pl.order + p * pl.order_stride);
        const uint32_t *fuse = (const uint32_t *)((const uint8_t *)pl.fuse + p * pl.bits_stride);
        uint16_t *out = table + p * (int64_t)N;
        for (int32_t k = lane; k < D * M; k += 32) last[k] = 0xFFFFu;
        __syncwarp();
        for (int32_t base = ((N - 1) / 32) * 32; base >= 0; base -= 32) {
            const int32_t j = base + lane;
            uint32_t key = 0xFFFFFFFFu;  // not the start of a unit
            if (j < N) {
                const int32_t x = __ldg(order + j);
                const int32_t d = __ldg(place + x);
                const uint4 hr = __ldg(dp.hrec + x);
                const uint32_t fp = hr.x & 0xFFFFu;
                const bool member = fp != 0xFFFFu && ((__ldg(fuse + (x >> 5)) >> (x & 31)) & 1u) &&
                                    __ldg(place + fp) == d;
                if (!member) key = (uint32_t)d * M + ((hr.y >> 16) & 15u);
            }
            const uint32_t same = __match_any_sync(0xFFFFFFFFu, key);
            const uint32_t above = lane == 31 ? 0u : (same & (0xFFFFFFFFu << (lane + 1)));
            if (key != 0xFFFFFFFFu) out[j] = above ? (uint16_t)(base + __ffs((int)above) - 1) : last[key];
            __syncwarp();
            if (key != 0xFFFFFFFFu && lane == __ffs((int)same) - 1) last[key] = (uint16_t)j;
            __syncwarp();
        }
    }
}

// Status bits of every plan (Eq. 8-10), one warp per plan.  Four nodes per
// lane check placement and fit (one fit mask per node); the warp scatters the
// inverse of the dispatch sequence (u16 positions) into shared memory and
// reads it back: a repeated node leaves some position with another position's
// entry, so every in-range sequence that reads back intact is a permutation.
// The edges (pred | succ << 16) are then checked 32 at a time.  Invalid plans
// get INT64_MAX metrics here; the sweep skips them.
__host__ __device__ inline uint32_t status_warp_bytes(int32_t N)
{
    return round16(2u * (uint32_t)N);
}

// kByte: every device index is below 8, so one byte per node holds its fit
// mask (fit8): a quarter of the table reads of the 32-bit masks.
template <bool kByte, int kU, bool kPlace>
__global__ void __launch_bounds__(128)
status_kernel(wf_dev_problem dp, wf_plans pl, wf_eval_out out)
{
    extern __shared__ __align__(16) uint8_t ssm[];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, warps = blockDim.x >> 5;
    const int32_t N = dp.N, D = dp.D, E = dp.E;
    uint16_t *pos = (uint16_t *)(ssm + (size_t)warp * status_warp_bytes(N));
    // Plans are visited from the last to the first: the rows read last stay
    // in L2, and they are those of the sweep's first wave of CTAs (the
    // lowest plan indices), which then re-reads them from L2 rather than DRAM.
    for (int64_t k = (int64_t)blockIdx.x * warps + warp; k < pl.P; k += (int64_t)gridDim.x * warps) {
        const int64_t p = pl.P - 1 - k;
        const uint8_t *place = pl.place + p * pl.place_stride;
        const uint16_t *order = (const uint16_t *)((const uint8_t *)pl.order + p * pl.order_stride);
        uint32_t st = 0;
        // Rows start 16-byte aligned and their strides are multiples of 16
        // bytes, so 16-byte reads at multiples of 16 bytes below N stay in
        // the row; lanes mask the entries at or beyond N.  The fit masks are
        // padded to 16 entries.
        // Every loop issues kU 16-byte reads per lane before it uses any: on
        // long rows a warp keeps a plan's reads in flight rather than one
        // round trip per 512 bytes (kU = 1 on short rows, whose loops run once).
        // The inverse permutation, 8 dispatch entries a lane at a time, then
        // read back: a repeated node leaves some entry unmatched.
        for (int32_t b8 = 8 * lane; b8 < N; b8 += kU * 256) {
            uint4 ow[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u)
                ow[u] = b8 + 256 * u < N ? __ldg((const uint4 *)(order + b8 + 256 * u)) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int32_t i8 = b8 + 256 * u;
                const uint32_t w[4] = {ow[u].x, ow[u].y, ow[u].z, ow[u].w};
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const uint32_t h = (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
                    if (i8 + j < N) {
                        if (h < (uint32_t)N) pos[h] = (uint16_t)(i8 + j);
                        else st |= WF_ST_PERMUTATION;
                    }
                }
            }
        }
        __syncwarp();
        for (int32_t b8 = 8 * lane; b8 < N; b8 += kU * 256) {
            uint4 ow[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u)
                ow[u] = b8 + 256 * u < N ? __ldg((const uint4 *)(order + b8 + 256 * u)) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int32_t i8 = b8 + 256 * u;
                const uint32_t w[4] = {ow[u].x, ow[u].y, ow[u].z, ow[u].w};
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const uint32_t h = (w[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
                    if (i8 + j < N && h < (uint32_t)N && pos[h] != (uint16_t)(i8 + j)) st |= WF_ST_PERMUTATION;
                }
            }
        }
        st = __reduce_or_sync(0xFFFFFFFFu, st);
        if (!(st & WF_ST_PERMUTATION)) {
            for (int32_t b4 = 4 * lane; b4 < E; b4 += kU * 128) {  // edges padded to 4
                uint4 uv[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u)
                    uv[u] = b4 + 128 * u < E ? __ldg((const uint4 *)(dp.edges + b4 + 128 * u)) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int32_t e4 = b4 + 128 * u;
                    const uint32_t w[4] = {uv[u].x, uv[u].y, uv[u].z, uv[u].w};
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        if (e4 + j < E && pos[w[j] & 0xFFFFu] > pos[w[j] >> 16]) st |= WF_ST_TOPOLOGY;
                }
            }
            st = __reduce_or_sync(0xFFFFFFFFu, st);
        }
        // Placement and fit (Eq. 8): here when asked (kPlace), else only for
        // a plan whose order is already invalid; the sweep's producers check
        // the placement of every other plan as they read it.
        if (kPlace || st) {
            for (int32_t b16 = 16 * lane; b16 < N; b16 += kU * 512) {
                uint4 pw[kU], fb[kU], fm[kU][4];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int32_t n16 = b16 + 512 * u;
                    const bool in = n16 < N;
                    pw[u] = in ? __ldg((const uint4 *)(place + n16)) : make_uint4(0u, 0u, 0u, 0u);
                    if (kByte) {
                        fb[u] = in ? __ldg((const uint4 *)(dp.fit8 + n16)) : make_uint4(0u, 0u, 0u, 0u);
                    } else {
#pragma unroll
                        for (int q = 0; q < 4; ++q)
                            fm[u][q] = in ? __ldg((const uint4 *)(dp.fitmask + n16 + 4 * q)) : make_uint4(0u, 0u, 0u, 0u);
                    }
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int32_t n16 = b16 + 512 * u;
                    const uint32_t pws[4] = {pw[u].x, pw[u].y, pw[u].z, pw[u].w};
                    if (kByte) {
                        const uint32_t fbs[4] = {fb[u].x, fb[u].y, fb[u].z, fb[u].w};
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                const uint32_t d = (pws[q] >> (8 * j)) & 255u, f = (fbs[q] >> (8 * j)) & 255u;
                                if (n16 + 4 * q + j < N)
                                    st |= d >= (uint32_t)D ? WF_ST_DEVICE
                                                           : (((f >> (d & 7u)) & 1u) ? 0u : WF_ST_CAPACITY);
                            }
                        }
                    } else {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const uint32_t f[4] = {fm[u][q].x, fm[u][q].y, fm[u][q].z, fm[u][q].w};
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                const uint32_t d = (pws[q] >> (8 * j)) & 255u;
                                if (n16 + 4 * q + j < N)
                                    st |= d >= (uint32_t)D ? WF_ST_DEVICE : (((f[j] >> d) & 1u) ? 0u : WF_ST_CAPACITY);
                            }
                        }
                    }
                }
            }
        }
        st = __reduce_or_sync(0xFFFFFFFFu, st);
        if (lane == 0) {
            out.status[p] = st;
            if (st) out.makespan_us[p] = out.p95_us[p] = out.gpu_us[p] = WF_INF64;
            if (st && dp.phi_life) dp.phi_timely[p] = dp.phi_life[p] = WF_INF64;
        }
        __syncwarp();  // pos[] is reused by the warp's next plan
    }
}

template <bool kByte, int kU, bool kPlace>
int launch_status_as(const wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    const size_t wbytes = status_warp_bytes(dp.N);
    const int swarps = (int)std::max<size_t>(1, std::min<size_t>(4, (227 * 1024) / wbytes));
    const size_t ssmem = wbytes * swarps;
    int rc = wf_cuda_check(cudaFuncSetAttribute(status_kernel<kByte, kU, kPlace>,
                                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ssmem),
                           "status smem attribute");
    if (rc) return rc;
    const int64_t sblocks = std::min<int64_t>((pl->P + swarps - 1) / swarps, (int64_t)ctx->sms * 16);
    status_kernel<kByte, kU, kPlace><<<(unsigned)sblocks, 32 * swarps, ssmem, st>>>(dp, *pl, *out);
    return WF_OK;
}

template <bool kPlace>
int launch_status_p(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, cudaStream_t st)
{
    const bool byte = ctx->dp.D <= 8, wide = ctx->dp.N >= 1024;
    if (wide)
        return byte ? launch_status_as<true, 4, kPlace>(ctx, pl, out, st)
                    : launch_status_as<false, 4, kPlace>(ctx, pl, out, st);
    return byte ? launch_status_as<true, 1, kPlace>(ctx, pl, out, st)
                : launch_status_as<false, 1, kPlace>(ctx, pl, out, st);
}

// The status pass; with place false the placement and fit checks of a plan
// whose order is valid are left to the deterministic sweep's producers.
int launch_status(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, cudaStream_t st, bool place)
{
    return place ? launch_status_p<true>(ctx, pl, out, st) : launch_status_p<false>(ctx, pl, out, st);
}

}  // namespace

// Shared memory of the producer / consumer kernel for this problem, or 0 when
// the sweep cannot run it (slots unavailable, times beyond u32, more than 16
// models, or more shared memory than a CTA may hold); the caller then uses
// the int64 path.
size_t wf_stoch_smem(const wf_dev_problem &dp)
{
    if (dp.nslots <= 0 || dp.nslots > 32765 || dp.max_arrival >= (int64_t)1 << 32 || dp.M > 16 || dp.N > 65534 ||
        dp.S < 1 || dp.S > kSamples)
        return 0;
    const size_t s = stoch_layout(dp.D, dp.M, dp.W, dp.nslots + 2).total;
    return s <= 227 * 1024 ? s : 0;
}

namespace {

template <typename Q, typename BT>
int stoch_launch(const wf_dev_problem &dp, unsigned blocks, size_t smem, const wf_plans *pl, const wf_eval_out *out,
                 int32_t *ovf_list, int32_t *ovf_count, cudaStream_t st)
{
    int rc = wf_cuda_check(cudaFuncSetAttribute(stoch_kernel<Q, BT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                (int)smem), "stochastic smem attribute");
    if (rc) return rc;
    stoch_kernel<Q, BT><<<blocks, 32 * kSWarps, smem, st>>>(dp, *pl, *out, ovf_list, ovf_count);
    return WF_OK;
}

}  // namespace

// Shared memory of the replica-batch sweep for this problem, or 0 when it
// cannot run it (the same slot and size limits as the sweep, plus room for
// every device's B_q slots); the caller then uses the int64 path.
size_t wf_batch_smem(const wf_dev_problem &dp)
{
    if (dp.batch < 1 || dp.S != 0 || dp.nslots <= 0 || dp.nslots > 32765 || dp.max_arrival >= (int64_t)1 << 32 ||
        dp.M > 16 || dp.N > 65534 || dp.phi_life || dp.reclaim)
        return 0;
    const size_t s = bq_layout(dp.D, dp.M, dp.W, dp.batch, dp.nslots + 2).total;
    return s <= 227 * 1024 ? s : 0;
}

// Status pass (placement left to the producers), then the replica-batch
// sweep; plans with a saturated chain run are listed for the int64 path.
int wf_launch_batch(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, size_t smem, int32_t *ovf_list,
                    int32_t *ovf_count, cudaStream_t st)
{
    int rc = launch_status(ctx, pl, out, st, false);
    if (!rc) rc = wf_cuda_check(cudaFuncSetAttribute(bq_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                                "batch sweep smem attribute");
    if (rc) return rc;
    const unsigned blocks = (unsigned)((pl->P + kBqPlans - 1) / kBqPlans);
    bq_kernel<<<blocks, 32 * kBqWarps, smem, st>>>(ctx->dp, *pl, *out, ovf_list, ovf_count);
    return wf_cuda_check(cudaGetLastError(), "batch sweep launch");
}

int wf_launch_stoch(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, size_t smem,
                    int32_t *ovf_list, int32_t *ovf_count, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    int rc = launch_status(ctx, pl, out, st, true);
    if (rc) return rc;
    const unsigned blocks = (unsigned)pl->P;
    const bool t16 = dp.bm_r16 != nullptr;
    if (dp.M <= 8)
        rc = t16 ? stoch_launch<uint32_t, int16_t>(dp, blocks, smem, pl, out, ovf_list, ovf_count, st)
                 : stoch_launch<uint32_t, int32_t>(dp, blocks, smem, pl, out, ovf_list, ovf_count, st);
    else
        rc = t16 ? stoch_launch<uint64_t, int16_t>(dp, blocks, smem, pl, out, ovf_list, ovf_count, st)
                 : stoch_launch<uint64_t, int32_t>(dp, blocks, smem, pl, out, ovf_list, ovf_count, st);
    if (rc) return rc;
    return wf_cuda_check(cudaGetLastError(), "stochastic launch");
}

namespace {

bool sweep_usable(const wf_dev_problem &dp)
{
    return dp.nslots > 0 && dp.nslots <= 32765 && dp.max_arrival < ((int64_t)1 << 32) && dp.M <= 16 &&
           dp.N <= 65534;
}

// The 64-bit sweep keeps its slots in 40 bits when no time of the window can
// reach 2^40 us (the context's horizon bounds every finish) and reclamation
// is least recently used.
bool split40(const wf_dev_problem &dp) { return dp.horizon < ((int64_t)1 << 40) && dp.reclaim == 0; }

// The relative-time sweep: least recently used, no window terms, and room
// for the sessions' 64-bit latencies in slot pairs at the end of a plan.
bool rel32(const wf_dev_problem &dp)
{
    return sweep_usable(dp) && dp.reclaim == 0 && !dp.phi_life && 2 * (int64_t)dp.W <= (int64_t)dp.nslots + 2;
}

template <typename Q, typename TT, int kP, int kR, bool kF, typename ST = TT>
int launch_pc(const wf_dev_problem &dp, int sms, int resident, const wf_plans *pl, const wf_eval_out *out,
              size_t smem, const int32_t *in_list, const int32_t *in_count, int32_t *list, int32_t *count, cudaStream_t st)
{
    int rc = wf_cuda_check(cudaFuncSetAttribute(pc_kernel<Q, TT, kP, kR, kF, ST>,
                                                cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem),
                           "sweep smem attribute");
    if (rc) return rc;
    // Every plan: a CTA per group.  A list (of unknown length): at most as
    // many CTAs as are resident at once, each walking over groups.
    int64_t blocks = (pl->P + kP - 1) / kP;
    if (in_list) blocks = std::min<int64_t>(blocks, (int64_t)std::max(1, resident) * sms);
    pc_kernel<Q, TT, kP, kR, kF, ST><<<(unsigned)blocks, 32 * PcShape<kP>::kWarps, smem, st>>>(
        dp, *pl, *out, in_list, in_count, list, count);
    return wf_cuda_check(cudaGetLastError(), "sweep launch");
}

template <typename T> struct Ty { using type = T; };
template <int V> struct Iv { static constexpr int value = V; };

// Calls f(Ty<Q>{}, Iv<kP>{}, Ty<ST>{}) for the sweep instantiation that this
// problem and CTA shape take: Q the LRU word (up to 8 models pack in 32 bits),
// kP the plans per CTA, ST the finish-slot storage.
template <typename TT, int kR, typename F>
int pc_visit(const wf_dev_problem &dp, int kp, F &&f)
{
    if constexpr (sizeof(TT) == 4) {  // the u32 sweep has one shape
        (void)kp;
        return dp.M <= 8 ? f(Ty<uint32_t>{}, Iv<kPlans32>{}, Ty<TT>{}) : f(Ty<uint64_t>{}, Iv<kPlans32>{}, Ty<TT>{});
    } else {
        auto by_q = [&](auto p, auto s) { return dp.M <= 8 ? f(Ty<uint32_t>{}, p, s) : f(Ty<uint64_t>{}, p, s); };
        auto by_p = [&](auto s) {
            return kp == 16 ? by_q(Iv<16>{}, s) : kp == 6 ? by_q(Iv<6>{}, s) : by_q(Iv<3>{}, s);
        };
        if constexpr (kR == 0)
            if (split40(dp)) return by_p(Ty<Split40>{});
        return by_p(Ty<TT>{});
    }
}

template <typename TT, int kR, bool kF>
int launch_pc_r(const wf_ctx *ctx, int kp, int resident, const wf_plans *pl, const wf_eval_out *out, size_t smem,
                const int32_t *in_list, const int32_t *in_count, int32_t *list, int32_t *count, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    return pc_visit<TT, kR>(dp, kp, [&](auto q, auto p, auto s) {
        return launch_pc<typename decltype(q)::type, TT, decltype(p)::value, kR, kF, typename decltype(s)::type>(
            dp, ctx->sms, resident, pl, out, smem, in_list, in_count, list, count, st);
    });
}

// CTAs of the sweep instantiation resident on one SM at this shared-memory
// size: registers and shared memory both count (0 = it does not fit).
template <typename TT, int kR, bool kF>
int resident_r(const wf_dev_problem &dp, int kp, size_t smem)
{
    if (smem > 227 * 1024) return 0;
    return pc_visit<TT, kR>(dp, kp, [&](auto q, auto p, auto s) {
        const auto k = pc_kernel<typename decltype(q)::type, TT, decltype(p)::value, kR, kF, typename decltype(s)::type>;
        int n = 0;
        if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k, 32 * PcShape<decltype(p)::value>::kWarps, smem) !=
                cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        return n;
    });
}

template <typename TT>
int resident(const wf_dev_problem &dp, int kp, size_t smem)
{
    if (dp.phi_life)
        return dp.reclaim ? resident_r<TT, 1, true>(dp, kp, smem) : resident_r<TT, 0, true>(dp, kp, smem);
    return dp.reclaim ? resident_r<TT, 1, false>(dp, kp, smem) : resident_r<TT, 0, false>(dp, kp, smem);
}

// The relative-time sweep's shapes: 16 or 6 plans per CTA.
template <typename F>
int rel_visit(const wf_dev_problem &dp, int kp, F &&f)
{
    auto by_q = [&](auto p) {
        return dp.M <= 8 ? f(Ty<uint32_t>{}, p) : f(Ty<uint64_t>{}, p);
    };
    return kp == 16 ? by_q(Iv<16>{}) : by_q(Iv<6>{});
}

int resident_rel(const wf_dev_problem &dp, int kp, size_t smem)
{
    if (smem > 227 * 1024) return 0;
    return rel_visit(dp, kp, [&](auto q, auto p) {
        const auto k = pc_kernel<typename decltype(q)::type, uint32_t, decltype(p)::value, 0, false, Rel32>;
        int n = 0;
        if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess ||
            cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, k, 32 * PcShape<decltype(p)::value>::kWarps, smem) !=
                cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        return n;
    });
}

// Every plan of the batch, in at most as many CTAs as are resident at once
// and as the evaluation scratch holds session rows for (each CTA walks
// over groups); the plans that leave 32 bits go to list.
int64_t rel_blocks(const wf_ctx *ctx, const wf_sweep_cfg &cfg, int64_t P)
{
    if (!cfg.smemRel) return 0;
    const int kp = cfg.plansRel;
    const int64_t rows = (int64_t)(ctx->eval_scratch_bytes / (8 * (size_t)std::max(ctx->dp.W, 1)));
    return std::min<int64_t>(std::min<int64_t>((P + kp - 1) / kp, (int64_t)std::max(1, cfg.resRel) * ctx->sms),
                             rows / kp);
}

int launch_rel(wf_ctx *ctx, const wf_sweep_cfg &cfg, int64_t blocks, const wf_plans *pl, const wf_eval_out *out,
               int32_t *list, int32_t *count, cudaStream_t st)
{
    wf_dev_problem dp = ctx->dp;
    dp.rel_ret = (uint64_t *)ctx->eval_scratch;
    return rel_visit(dp, cfg.plansRel, [&](auto q, auto p) {
        const auto k = pc_kernel<typename decltype(q)::type, uint32_t, decltype(p)::value, 0, false, Rel32>;
        int rc = wf_cuda_check(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cfg.smemRel),
                               "sweep smem attribute");
        if (rc) return rc;
        k<<<(unsigned)blocks, 32 * PcShape<decltype(p)::value>::kWarps, cfg.smemRel, st>>>(dp, *pl, *out, nullptr,
                                                                                           nullptr, list, count);
        return wf_cuda_check(cudaGetLastError(), "sweep launch");
    });
}

template <typename TT>
int launch_pc_q(const wf_ctx *ctx, int kp, int resident, const wf_plans *pl, const wf_eval_out *out, size_t smem,
                const int32_t *in_list, const int32_t *in_count, int32_t *list, int32_t *count, cudaStream_t st)
{
    if (ctx->dp.phi_life)
        return ctx->dp.reclaim
                   ? launch_pc_r<TT, 1, true>(ctx, kp, resident, pl, out, smem, in_list, in_count, list, count, st)
                   : launch_pc_r<TT, 0, true>(ctx, kp, resident, pl, out, smem, in_list, in_count, list, count, st);
    return ctx->dp.reclaim
               ? launch_pc_r<TT, 1, false>(ctx, kp, resident, pl, out, smem, in_list, in_count, list, count, st)
               : launch_pc_r<TT, 0, false>(ctx, kp, resident, pl, out, smem, in_list, in_count, list, count, st);
}

}  // namespace

int wf_launch_nextuse(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, cudaStream_t st)
{
    const wf_dev_problem &dp = ctx->dp;
    const size_t smem = (size_t)kNuWarps * dp.D * dp.M * sizeof(uint16_t);
    const int64_t blocks = std::min<int64_t>((pl->P + kNuWarps - 1) / kNuWarps, (int64_t)ctx->sms * 16);
    nextuse_kernel<<<(unsigned)blocks, 32 * kNuWarps, smem, st>>>(dp, *pl, out->status, dp.nextuse);
    return wf_cuda_check(cudaGetLastError(), "next-use launch");
}

// Shared memory of a sweep CTA for this problem, its reclamation order and
// whether the window terms of Eq. 12 are wanted.
template <int kP, typename TT>
size_t layout_bytes(const wf_dev_problem &dp)
{
    const int32_t NS = dp.nslots + 2;
    if (sizeof(TT) == 8 && split40(dp))
        return dp.phi_life ? pc_layout<kP, TT, 0, true, Split40>(dp.D, dp.M, dp.W, NS).total
                           : pc_layout<kP, TT, 0, false, Split40>(dp.D, dp.M, dp.W, NS).total;
    if (dp.phi_life)
        return dp.reclaim ? pc_layout<kP, TT, 1, true>(dp.D, dp.M, dp.W, NS).total
                          : pc_layout<kP, TT, 0, true>(dp.D, dp.M, dp.W, NS).total;
    return dp.reclaim ? pc_layout<kP, TT, 1, false>(dp.D, dp.M, dp.W, NS).total
                      : pc_layout<kP, TT, 0, false>(dp.D, dp.M, dp.W, NS).total;
}

namespace {

// The shape choice depends on these fields of the problem only (and on the
// device, whose registers and shared memory bound the resident CTAs).
struct CfgKey {
    int dev;
    int32_t D, M, W, nslots;
    bool usable, split, reclaim, phi;
    bool operator==(const CfgKey &o) const
    {
        return dev == o.dev && D == o.D && M == o.M && W == o.W && nslots == o.nslots && usable == o.usable &&
               split == o.split && reclaim == o.reclaim && phi == o.phi;
    }
};

wf_sweep_cfg choose(const wf_dev_problem &dp)
{
    wf_sweep_cfg c = {};
    if (!sweep_usable(dp)) return c;
    const size_t s32 = layout_bytes<kPlans32, uint32_t>(dp);
    c.res32 = resident<uint32_t>(dp, kPlans32, s32);
    if (c.res32 > 0) c.smem32 = s32;
    // The u64 sweep: 16, 6 or 3 plans per CTA, whichever keeps the most plans
    // resident per SM, registers and shared memory both counted.  Ties go to
    // the larger CTA, whose producer and residency warps serve more plans.
    const int shapes[3] = {16, 6, 3};
    int best = 0;
    for (int kp : shapes) {
        const size_t sm = kp == 16 ? layout_bytes<16, uint64_t>(dp)
                          : kp == 6 ? layout_bytes<6, uint64_t>(dp)
                                    : layout_bytes<3, uint64_t>(dp);
        const int n = resident<uint64_t>(dp, kp, sm);
        if (n > 0 && kp * n > best) {
            best = kp * n;
            c.smem64 = sm;
            c.plans64 = kp;
            c.res64 = n;
        }
    }
    // The relative-time sweep (for contexts whose plans leave 32 bits): 6 or
    // 16 plans per CTA, whichever keeps more plans resident per SM; ties go
    // to the smaller CTA, whose timing warp (the chain that paces the sweep)
    // has fewer plans to play (large window: 6-plan CTAs 72.7 ms, 8-plan CTAs
    // at the same 24 plans per SM 78.0 ms).
    if (c.smem64 && rel32(dp)) {
        const int rshapes[2] = {6, 16};
        int rbest = 0;
        for (int kp : rshapes) {
            const int32_t NS = dp.nslots + 2;
            const size_t sm = kp == 16 ? pc_layout<16, uint32_t, 0, false, Rel32>(dp.D, dp.M, dp.W, NS).total
                                       : pc_layout<6, uint32_t, 0, false, Rel32>(dp.D, dp.M, dp.W, NS).total;
            const int n = resident_rel(dp, kp, sm);
            if (n > 0 && kp * n > rbest) {
                rbest = kp * n;
                c.smemRel = sm;
                c.plansRel = kp;
                c.resRel = n;
            }
        }
    }
    return c;
}

}  // namespace

wf_sweep_cfg wf_sweep_config(const wf_dev_problem &dp)
{
    static std::mutex mu;
    static std::vector<std::pair<CfgKey, wf_sweep_cfg>> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return wf_sweep_cfg{};
    }
    const CfgKey key = {dev, dp.D, dp.M, dp.W, dp.nslots, sweep_usable(dp), split40(dp), dp.reclaim != 0,
                        dp.phi_life != 0};
    std::lock_guard<std::mutex> lock(mu);
    for (const auto &e : cache)
        if (e.first == key) return e.second;
    const wf_sweep_cfg c = choose(dp);
    if (cache.size() >= 64) cache.erase(cache.begin());
    cache.emplace_back(key, c);
    return c;
}

int wf_launch_sweep(wf_ctx *ctx, const wf_plans *pl, const wf_eval_out *out, const wf_sweep_cfg &cfg,
                    bool wide_first, int32_t *counts, int32_t *list1, int32_t *list2, cudaStream_t st,
                    const int32_t **rest_list, const int32_t **rest_count)
{
    // The next-use pass reads every plan's placement before the sweep, so
    // under that policy the status pass checks placement itself.
    int rc = launch_status(ctx, pl, out, st, ctx->dp.reclaim != 0);
    if (!rc && ctx->dp.reclaim) rc = wf_launch_nextuse(ctx, pl, out, st);
    if (rc) return rc;
    const int64_t rblocks = wide_first && ctx->start_path != WF_PATH_WIDE ? rel_blocks(ctx, cfg, pl->P) : 0;
    if (rblocks > 0) {
        // Relative u32 times for every plan; the plans that leave 32 bits
        // even so go on to the u64 sweep.
        rc = launch_rel(ctx, cfg, rblocks, pl, out, list1, counts, st);
        if (!rc) rc = launch_pc_q<uint64_t>(ctx, cfg.plans64, cfg.res64, pl, out, cfg.smem64, list1, counts, list2,
                                            counts + 1, st);
    } else if (cfg.smem32 && !(wide_first && cfg.smem64)) {
        // u32 times for every plan; the plans that leave 32 bits go on to the
        // u64 sweep, and from there (or straight) to the int64 path.
        rc = launch_pc_q<uint32_t>(ctx, kPlans32, cfg.res32, pl, out, cfg.smem32, nullptr, nullptr, list1, counts, st);
        if (rc) return rc;
        if (!cfg.smem64) { *rest_list = list1; *rest_count = counts; return WF_OK; }
        rc = launch_pc_q<uint64_t>(ctx, cfg.plans64, cfg.res64, pl, out, cfg.smem64, list1, counts, list2, counts + 1, st);
    } else {
        rc = launch_pc_q<uint64_t>(ctx, cfg.plans64, cfg.res64, pl, out, cfg.smem64, nullptr, nullptr, list2, counts + 1, st);
    }
    *rest_list = list2;
    *rest_count = counts + 1;
    return rc;
}
