/*
 * Seeded synthetic plan generator (input data only).
 *
 * A plan for one window of the activation DAG fixes, per activation, a device
 * (uint8), a dispatch sequence (uint16, position -> node), and per-node bits
 * for fusion, prefetch and retain (rows of uint32 words).  This file draws
 * such plans: placements uniform over the devices a node fits on, a random
 * topological dispatch sequence (Kahn's algorithm, always popping the ready
 * node with the smallest hashed priority), and independent Bernoulli bits.
 *
 * It holds none of the evaluation arithmetic: it never computes a time, a
 * residency state or a metric.  Every random draw is a pure function of
 * (seed, stream, plan index, element index) through the SplitMix64 output
 * function (Steele, Lea and Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014), so plan p is the same whichever chunk or thread
 * produces it, on any host.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define WFG_GOLDEN 0x9E3779B97F4A7C15ULL

static uint64_t wfg_mix(uint64_t x)
{
    x += WFG_GOLDEN;
    x = (x ^ (x >> 30)) * 0xBF58476D1CE4E5B9ULL;
    x = (x ^ (x >> 27)) * 0x94D049BB133111EBULL;
    return x ^ (x >> 31);
}

enum { WFG_S_PLACE = 1, WFG_S_ORDER = 2, WFG_S_FUSE = 3, WFG_S_PREFETCH = 4, WFG_S_RETAIN = 5 };

/* key of one (seed, stream, plan) triple; element i then draws wfg_mix(key ^ i) */
static uint64_t wfg_key(uint64_t seed, uint64_t stream, uint64_t plan)
{
    return wfg_mix(wfg_mix(seed ^ (stream * 0xD1B54A32D192ED03ULL)) ^ plan);
}

/* min-heap of (key, node) */
typedef struct { uint64_t key; int32_t node; } wfg_item;

static int wfg_less(const wfg_item *a, const wfg_item *b)
{
    return a->key < b->key || (a->key == b->key && a->node < b->node);
}

static void wfg_push(wfg_item *h, int32_t *n, wfg_item it)
{
    int32_t i = (*n)++;
    while (i > 0) {
        int32_t p = (i - 1) / 2;
        if (!wfg_less(&it, &h[p])) break;
        h[i] = h[p];
        i = p;
    }
    h[i] = it;
}

static wfg_item wfg_pop(wfg_item *h, int32_t *n)
{
    wfg_item top = h[0], last = h[--(*n)];
    const int32_t cnt = *n;
    int32_t i = 0;
    for (;;) {
        int32_t c = 2 * i + 1;
        if (c >= cnt) break;
        if (c + 1 < cnt && wfg_less(&h[c + 1], &h[c])) c = c + 1;
        if (!wfg_less(&h[c], &last)) break;
        h[i] = h[c];
        i = c;
    }
    if (cnt > 0) h[i] = last;
    return top;
}

static void wfg_bits(uint64_t seed, uint64_t stream, uint64_t plan, int32_t N,
                     uint64_t thresh, uint32_t *row, int64_t words)
{
    const uint64_t key = wfg_key(seed, stream, plan);
    memset(row, 0, (size_t)words * 4);
    for (int32_t n = 0; n < N; ++n)
        if ((wfg_mix(key ^ (uint64_t)n) >> 32) < thresh)
            row[n >> 5] |= 1u << (n & 31);
}

/*
 * Fill plans [plan_lo, plan_hi) of a batch whose first plan has global index
 * plan_base.  Rows are written at (p - plan_lo) * stride.  Thresholds are
 * probabilities scaled by 2^32 (0 = never, 2^32 = always).  retain may be
 * NULL.  Returns 0, or -1 if scratch allocation fails.
 */
int wfg_make_plans(int32_t N,
                   const int32_t *succ_off, const int32_t *succ_idx,
                   const int32_t *indeg,
                   const int32_t *feas_off, const uint8_t *feas_dev,
                   uint64_t seed, int64_t plan_base, int64_t plan_lo, int64_t plan_hi,
                   uint64_t t_fuse, uint64_t t_prefetch, uint64_t t_retain,
                   uint8_t *place, int64_t place_stride,
                   uint16_t *order, int64_t order_stride,
                   uint32_t *fuse, uint32_t *prefetch, uint32_t *retain,
                   int64_t bits_stride)
{
    wfg_item *heap = (wfg_item *)malloc(sizeof(wfg_item) * (size_t)(N > 0 ? N : 1));
    int32_t *deg = (int32_t *)malloc(sizeof(int32_t) * (size_t)(N > 0 ? N : 1));
    if (!heap || !deg) { free(heap); free(deg); return -1; }
    const int64_t words = bits_stride / 4;

    for (int64_t p = plan_lo; p < plan_hi; ++p) {
        const uint64_t gp = (uint64_t)(plan_base + p);
        const int64_t r = p - plan_lo;
        uint8_t *pl = place + r * place_stride;
        uint16_t *od = (uint16_t *)((uint8_t *)order + r * order_stride);

        const uint64_t kplace = wfg_key(seed, WFG_S_PLACE, gp);
        const uint64_t korder = wfg_key(seed, WFG_S_ORDER, gp);
        memset(pl, 0, (size_t)place_stride);
        for (int32_t n = 0; n < N; ++n) {
            int32_t nf = feas_off[n + 1] - feas_off[n];
            uint64_t h = wfg_mix(kplace ^ (uint64_t)n);
            int32_t k = (int32_t)(((h >> 32) * (uint64_t)nf) >> 32);
            pl[n] = feas_dev[feas_off[n] + k];
        }

        memset(od, 0, (size_t)order_stride);
        int32_t hn = 0, out = 0;
        for (int32_t n = 0; n < N; ++n) {
            deg[n] = indeg[n];
            if (deg[n] == 0) {
                wfg_item it = { wfg_mix(korder ^ (uint64_t)n), n };
                wfg_push(heap, &hn, it);
            }
        }
        while (hn > 0) {
            wfg_item it = wfg_pop(heap, &hn);
            od[out++] = (uint16_t)it.node;
            for (int32_t e = succ_off[it.node]; e < succ_off[it.node + 1]; ++e) {
                int32_t s = succ_idx[e];
                if (--deg[s] == 0) {
                    wfg_item nx = { wfg_mix(korder ^ (uint64_t)s), s };
                    wfg_push(heap, &hn, nx);
                }
            }
        }

        wfg_bits(seed, WFG_S_FUSE, gp, N, t_fuse,
                 (uint32_t *)((uint8_t *)fuse + r * bits_stride), words);
        wfg_bits(seed, WFG_S_PREFETCH, gp, N, t_prefetch,
                 (uint32_t *)((uint8_t *)prefetch + r * bits_stride), words);
        if (retain)
            wfg_bits(seed, WFG_S_RETAIN, gp, N, t_retain,
                     (uint32_t *)((uint8_t *)retain + r * bits_stride), words);
    }
    free(heap);
    free(deg);
    return 0;
}
