/*
 * tracegen.c -- seeded synthetic allocation traces for the memory-planning path.
 *
 * A trace is the list of intermediate tensors of one forward pass, each given
 * by (alloc_step, free_step, size_bytes) with the lifetime half-open
 * [alloc_step, free_step).  The paper captures such traces with an
 * instrumented allocator (Sec. 3.1, Table 3.1); none are available here, so
 * this module draws DNN-shaped stand-ins whose shapes follow Table 1.1,
 * Table 3.1 and the "mostly below 1 MB" size distributions of Sec. 2.2.
 *
 * This file holds only random-number generation and sampling: none of the
 * planning arithmetic.  Both the CPU oracle and the CUDA path consume the
 * bytes it writes, so neither side needs cross-platform float agreement of
 * its own.  To make the bytes identical on x86-64 and AArch64 hosts the only
 * floating point used is IEEE double add/multiply/compare in a fixed order
 * (build with -ffp-contract=off), and exp2 is evaluated by the series below
 * rather than by libm.
 *
 * Generators:
 *   SplitMix64 (Steele, Lea, Flood, OOPSLA 2014) expands a 64-bit seed into
 *   the 256-bit state of xoshiro256** (Blackman, Vigna, 2018).
 */
#include <stdint.h>
#include <string.h>

#define TG_EXPORT __attribute__((visibility("default")))

typedef struct {
    uint64_t s[4];
} tg_rng;

static inline uint64_t tg_rotl(uint64_t x, int k) { return (x << k) | (x >> (64 - k)); }

/* SplitMix64: add the golden-gamma increment, then two xor-shift-multiply
 * mixing rounds and a final xor-shift. */
static uint64_t tg_splitmix64(uint64_t *state)
{
    uint64_t z = (*state += 0x9e3779b97f4a7c15ULL);
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

static void tg_seed(tg_rng *r, uint64_t seed)
{
    uint64_t sm = seed;
    for (int k = 0; k < 4; ++k) r->s[k] = tg_splitmix64(&sm);
}

/* xoshiro256**: output rotl(s1 * 5, 7) * 9, then the xor/shift/rotate state
 * update of the published generator. */
static uint64_t tg_next(tg_rng *r)
{
    uint64_t *s = r->s;
    uint64_t out = tg_rotl(s[1] * 5u, 7) * 9u;
    uint64_t t = s[1] << 17;
    s[2] ^= s[0];
    s[3] ^= s[1];
    s[1] ^= s[2];
    s[0] ^= s[3];
    s[2] ^= t;
    s[3] = tg_rotl(s[3], 45);
    return out;
}

/* Uniform double in [0, 1) from the top 53 bits. */
static double tg_unit(tg_rng *r) { return (double)(tg_next(r) >> 11) * 0x1.0p-53; }

/* Uniform integer in [lo, hi] (inclusive), unbiased: draws below
 * 2^64 mod range are rejected so that x mod range is exactly uniform. */
static int64_t tg_uniform_int(tg_rng *r, int64_t lo, int64_t hi)
{
    uint64_t range = (uint64_t)(hi - lo) + 1u;
    if (range == 0) return (int64_t)tg_next(r); /* full 64-bit range */
    uint64_t reject_below = (0u - range) % range;
    for (;;) {
        uint64_t x = tg_next(r);
        if (x >= reject_below) return lo + (int64_t)(x % range);
    }
}

/* Number of failures before the first success of Bernoulli(p) trials
 * (support 0, 1, 2, ...).  Capped far beyond any probability that matters. */
static int64_t tg_geometric(tg_rng *r, double p)
{
    int64_t k = 0;
    while (!(tg_unit(r) < p)) {
        if (++k >= (int64_t)1 << 24) break;
    }
    return k;
}

/* 2^x for 0 <= x < 64: integer part by exact scaling, fractional part by the
 * Taylor series of exp(r ln 2) summed to 24 terms (|r ln 2| < 0.7, so the
 * truncation error is below 1e-25 relative).  Plain double operations only. */
static double tg_exp2(double x)
{
    int64_t n = (int64_t)x; /* x >= 0: truncation is floor */
    double r = x - (double)n;
    const double ln2 = 0.693147180559945309417232121458176568;
    double y = r * ln2;
    double term = 1.0, sum = 1.0;
    for (int k = 1; k <= 24; ++k) {
        term = term * y / (double)k;
        sum = sum + term;
    }
    double scale = 1.0;
    for (int64_t k = 0; k < n; ++k) scale = scale * 2.0;
    return sum * scale;
}

/* Log-uniform size in [2^lo_e, 2^hi_e], rounded up to a multiple of 64 bytes
 * and clamped to the interval. */
static int64_t tg_log_uniform_size(tg_rng *r, int lo_e, int hi_e)
{
    double u = tg_unit(r);
    double v = tg_exp2((double)lo_e + u * (double)(hi_e - lo_e));
    int64_t c = (int64_t)v;
    if ((double)c < v) c += 1; /* ceil */
    c = ((c + 63) / 64) * 64;
    int64_t lo = (int64_t)1 << lo_e, hi = (int64_t)1 << hi_e;
    if (c < lo) c = lo;
    if (c > hi) c = hi;
    return c;
}

static int32_t tg_cap(int64_t a, int64_t life, int32_t T)
{
    int64_t f = a + life;
    return (int32_t)(f < T ? f : T);
}

/* Marks exactly k of the n tensors via a partial Fisher-Yates shuffle of the
 * index list: position j is swapped with a uniform position in [j, n). */
static void tg_pick_subset(tg_rng *r, int32_t n, int32_t k, int32_t *idx_scratch, uint8_t *mark)
{
    for (int32_t i = 0; i < n; ++i) {
        idx_scratch[i] = i;
        mark[i] = 0;
    }
    for (int32_t j = 0; j < k && j < n; ++j) {
        int32_t p = (int32_t)tg_uniform_int(r, j, n - 1);
        int32_t t = idx_scratch[j];
        idx_scratch[j] = idx_scratch[p];
        idx_scratch[p] = t;
        mark[idx_scratch[j]] = 1;
    }
}

/* ------------------------------------------------------------------ exports */

TG_EXPORT uint64_t tg_debug_next(uint64_t seed, int32_t skip)
{
    tg_rng r;
    tg_seed(&r, seed);
    for (int32_t i = 0; i < skip; ++i) tg_next(&r);
    return tg_next(&r);
}

TG_EXPORT double tg_debug_exp2(double x) { return tg_exp2(x); }

TG_EXPORT int64_t tg_debug_uniform_int(uint64_t seed, int64_t lo, int64_t hi, int32_t skip)
{
    tg_rng r;
    tg_seed(&r, seed);
    for (int32_t i = 0; i < skip; ++i) tg_uniform_int(&r, lo, hi);
    return tg_uniform_int(&r, lo, hi);
}

/* Random trace (one trace of the single-trace and batched random workloads):
 * per tensor, in id order: alloc ~ U[0, T-1], life = 1 + Geometric(p),
 * free = min(alloc + life, T), size log-uniform in [2^lo_e, 2^hi_e] rounded
 * up to 64 B. */
TG_EXPORT void tg_random_trace(uint64_t seed, int32_t n, int32_t T, double p, int32_t lo_e,
                               int32_t hi_e, int32_t *alloc_step, int32_t *free_step,
                               int64_t *size_bytes)
{
    tg_rng r;
    tg_seed(&r, seed);
    for (int32_t i = 0; i < n; ++i) {
        int64_t a = tg_uniform_int(&r, 0, T - 1);
        int64_t life = 1 + tg_geometric(&r, p);
        alloc_step[i] = (int32_t)a;
        free_step[i] = tg_cap(a, life, T);
        size_bytes[i] = tg_log_uniform_size(&r, lo_e, hi_e);
    }
}

/* Many random traces with consecutive seeds, written back to back
 * (trace k has seed seed0 + k and occupies [k*n, (k+1)*n)). */
TG_EXPORT void tg_random_batch(uint64_t seed0, int32_t n_traces, int32_t n, int32_t T, double p,
                               int32_t lo_e, int32_t hi_e, int32_t *alloc_step,
                               int32_t *free_step, int64_t *size_bytes)
{
    for (int32_t k = 0; k < n_traces; ++k) {
        int64_t base = (int64_t)k * n;
        tg_random_trace(seed0 + (uint64_t)k, n, T, p, lo_e, hi_e, alloc_step + base,
                        free_step + base, size_bytes + base);
    }
}

/* ResNet-50-shaped chain: 160 ops, op k runs at step k, T = 160.  Each of the
 * five 32-op stages takes its (C, H) uniformly from the five ResNet-50 stage
 * shapes (drawn first, stage 0..4).  Op k allocates two fp32 NCHW activations
 * (batch 1, 4*C*H*H bytes) living U{1..3} steps each and, when k % 3 == 0, a
 * residual living U{3,4} steps.  Writes up to 374 tensors; returns the count. */
TG_EXPORT int32_t tg_resnet_chain_trace(uint64_t seed, int32_t *alloc_step, int32_t *free_step,
                                        int64_t *size_bytes)
{
    static const int64_t shapes[5][2] = {{64, 112}, {256, 56}, {512, 28}, {1024, 14}, {2048, 7}};
    const int32_t n_ops = 160, per_stage = 32, T = 160;
    tg_rng r;
    tg_seed(&r, seed);
    int32_t stage_shape[5];
    for (int st = 0; st < 5; ++st) stage_shape[st] = (int32_t)tg_uniform_int(&r, 0, 4);
    int32_t n = 0;
    for (int32_t k = 0; k < n_ops; ++k) {
        const int64_t *cs = shapes[stage_shape[k / per_stage]];
        int64_t bytes = 4 * cs[0] * cs[1] * cs[1];
        for (int rep = 0; rep < 2; ++rep) {
            int64_t life = tg_uniform_int(&r, 1, 3);
            alloc_step[n] = k;
            free_step[n] = tg_cap(k, life, T);
            size_bytes[n] = bytes;
            ++n;
        }
        if (k % 3 == 0) {
            int64_t life = tg_uniform_int(&r, 3, 4);
            alloc_step[n] = k;
            free_step[n] = tg_cap(k, life, T);
            size_bytes[n] = bytes;
            ++n;
        }
    }
    return n;
}

/* Large single trace with a long-lived minority: exactly n_long tensors
 * (a Fisher-Yates subset, chosen first) live U[long_lo, long_hi] steps, the
 * rest 1 + Geometric(p); alloc ~ U[0, T-1]; sizes log-uniform in
 * [2^lo_e, 2^hi_e], 64 B-rounded.  Draw order per tensor: alloc, life, size.
 * idx_scratch needs n int32 and mark_scratch n bytes. */
TG_EXPORT void tg_long_tail_trace(uint64_t seed, int32_t n, int32_t T, int32_t n_long,
                                  int32_t long_lo, int32_t long_hi, double p, int32_t lo_e,
                                  int32_t hi_e, int32_t *alloc_step, int32_t *free_step,
                                  int64_t *size_bytes, int32_t *idx_scratch, uint8_t *mark_scratch)
{
    tg_rng r;
    tg_seed(&r, seed);
    tg_pick_subset(&r, n, n_long, idx_scratch, mark_scratch);
    for (int32_t i = 0; i < n; ++i) {
        int64_t a = tg_uniform_int(&r, 0, T - 1);
        int64_t life = mark_scratch[i] ? tg_uniform_int(&r, long_lo, long_hi) : 1 + tg_geometric(&r, p);
        alloc_step[i] = (int32_t)a;
        free_step[i] = tg_cap(a, life, T);
        size_bytes[i] = tg_log_uniform_size(&r, lo_e, hi_e);
    }
}

/* Seq2seq serving trace: batch B ~ U{1..8} and sequence length S ~ U[1, 512]
 * for the whole trace (drawn first), then exactly n_full tensors spanning
 * [0, T) (a Fisher-Yates subset).  Per tensor, in id order: with probability
 * 0.75 an activation of 4*B*S*H bytes, else per-token state of 4*B*H bytes;
 * H = 1024 with probability 0.7, else 4096; then, unless full-span,
 * alloc ~ U[0, T-1] and life = 1 + Geometric(p). */
TG_EXPORT void tg_seq2seq_trace(uint64_t seed, int32_t n, int32_t T, int32_t n_full, double p,
                                int32_t *alloc_step, int32_t *free_step, int64_t *size_bytes,
                                int32_t *idx_scratch, uint8_t *mark_scratch)
{
    tg_rng r;
    tg_seed(&r, seed);
    int64_t B = tg_uniform_int(&r, 1, 8);
    int64_t S = tg_uniform_int(&r, 1, 512);
    tg_pick_subset(&r, n, n_full, idx_scratch, mark_scratch);
    for (int32_t i = 0; i < n; ++i) {
        int activation = tg_unit(&r) < 0.75;
        int64_t H = tg_unit(&r) < 0.7 ? 1024 : 4096;
        size_bytes[i] = activation ? 4 * B * S * H : 4 * B * H;
        if (mark_scratch[i]) {
            alloc_step[i] = 0;
            free_step[i] = T;
        } else {
            int64_t a = tg_uniform_int(&r, 0, T - 1);
            int64_t life = 1 + tg_geometric(&r, p);
            alloc_step[i] = (int32_t)a;
            free_step[i] = tg_cap(a, life, T);
        }
    }
}
