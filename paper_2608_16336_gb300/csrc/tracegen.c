/*
 * tracegen.c -- seeded synthetic request traces for the multi-tier scheduler
 * simulation.  This module produces INPUTS only: arrival times, prompt and
 * output lengths and priority tiers.  It holds none of the scheduling
 * arithmetic (headroom, freeness, dispatch, migration, batching); both the CPU
 * oracle and the CUDA simulator read the arrays it writes.
 *
 * Workload shapes follow the paper's evaluation setup (Sec. 4.2 priority
 * sampling, Sec. 4.3 request lengths, Sec. 4.4 Poisson arrivals): priorities
 * are drawn from a per-replica categorical distribution over K tiers (tier 0 =
 * highest priority, Sec. 4.2), lengths from clipped, rounded lognormals, and
 * arrivals from a Poisson process or a Gamma renewal process with a given
 * coefficient of variation (bursty traffic).
 *
 * Random numbers: xoshiro256** (Blackman & Vigna, 2018) seeded through
 * SplitMix64 (Steele, Lea & Flood, 2014), one independent stream per replica.
 * Normal deviates: Box-Muller.  Gamma deviates: Marsaglia & Tsang (2000), with
 * the U^(1/a) boost for shape a < 1.
 *
 * Plain C99 + pthreads, no architecture-specific code, so it builds the same
 * on x86-64 and aarch64.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define TG_MAX_TIERS 16

#define TG_OK 0
#define TG_ERR_ARG (-1)
#define TG_ERR_OVERFLOW (-2)

#define TG_ARRIVAL_POISSON 0
#define TG_ARRIVAL_GAMMA 1

/* Per-replica trace parameters.  Must match tg_params_t in workloads.py. */
typedef struct {
    uint64_t seed;
    int64_t num_requests;
    int32_t num_tiers;
    int32_t arrival_kind;      /* TG_ARRIVAL_POISSON or TG_ARRIVAL_GAMMA */
    double rate_per_s;         /* mean arrival rate (requests / second) */
    double gamma_cv;           /* coefficient of variation of gaps (Gamma only) */
    double prompt_mu, prompt_sigma;
    int32_t prompt_min, prompt_max;
    double output_mu, output_sigma;
    int32_t output_min, output_max;
    double tier_probs[TG_MAX_TIERS]; /* categorical over tiers 0..K-1 */
} tg_params_t;

/* ---------------------------------------------------------------- PRNG --- */
static uint64_t splitmix64_next(uint64_t *s) {
    uint64_t z = (*s += 0x9E3779B97F4A7C15ULL);
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

typedef struct { uint64_t s[4]; int have_spare; double spare; } rng_t;

static uint64_t rotl64(uint64_t x, int k) { return (x << k) | (x >> (64 - k)); }

static uint64_t xoshiro_next(rng_t *r) {
    uint64_t *s = r->s;
    const uint64_t result = rotl64(s[1] * 5, 7) * 9;
    const uint64_t t = s[1] << 17;
    s[2] ^= s[0];
    s[3] ^= s[1];
    s[1] ^= s[2];
    s[0] ^= s[3];
    s[2] ^= t;
    s[3] = rotl64(s[3], 45);
    return result;
}

static void rng_seed(rng_t *r, uint64_t seed) {
    uint64_t sm = seed;
    for (int i = 0; i < 4; ++i) r->s[i] = splitmix64_next(&sm);
    r->have_spare = 0;
    r->spare = 0.0;
}

/* Uniform in the open interval (0, 1). */
static double rng_uniform(rng_t *r) {
    return ((double)(xoshiro_next(r) >> 11) + 0.5) * (1.0 / 9007199254740992.0);
}

static double rng_normal(rng_t *r) {
    if (r->have_spare) { r->have_spare = 0; return r->spare; }
    double u1 = rng_uniform(r), u2 = rng_uniform(r);
    double rad = sqrt(-2.0 * log(u1));
    double ang = 6.283185307179586476925286766559 * u2;
    r->spare = rad * sin(ang);
    r->have_spare = 1;
    return rad * cos(ang);
}

static double rng_gamma(rng_t *r, double shape) {
    if (shape < 1.0) {
        double g = rng_gamma(r, shape + 1.0);
        return g * pow(rng_uniform(r), 1.0 / shape);
    }
    double d = shape - 1.0 / 3.0, c = 1.0 / sqrt(9.0 * d);
    for (;;) {
        double x, v;
        do { x = rng_normal(r); v = 1.0 + c * x; } while (v <= 0.0);
        v = v * v * v;
        double u = rng_uniform(r);
        if (u < 1.0 - 0.0331 * x * x * x * x) return d * v;
        if (log(u) < 0.5 * x * x + d * (1.0 - v + log(v))) return d * v;
    }
}

static int32_t clipped_lognormal(rng_t *r, double mu, double sigma, int32_t lo, int32_t hi) {
    double v = exp(mu + sigma * rng_normal(r));
    double rv = floor(v + 0.5);
    if (rv < (double)lo) return lo;
    if (rv > (double)hi) return hi;
    return (int32_t)rv;
}

/* ------------------------------------------------------------ one trace --- */
static int validate(const tg_params_t *p) {
    if (p->num_requests < 0 || p->num_tiers < 1 || p->num_tiers > TG_MAX_TIERS) return TG_ERR_ARG;
    if (!(p->rate_per_s > 0.0)) return TG_ERR_ARG;
    if (p->arrival_kind != TG_ARRIVAL_POISSON && p->arrival_kind != TG_ARRIVAL_GAMMA) return TG_ERR_ARG;
    if (p->arrival_kind == TG_ARRIVAL_GAMMA && !(p->gamma_cv > 0.0)) return TG_ERR_ARG;
    if (p->prompt_min < 1 || p->prompt_max < p->prompt_min || p->prompt_max > 65535) return TG_ERR_ARG;
    if (p->output_min < 1 || p->output_max < p->output_min || p->output_max > 65535) return TG_ERR_ARG;
    double tot = 0.0;
    for (int k = 0; k < p->num_tiers; ++k) {
        if (!(p->tier_probs[k] >= 0.0)) return TG_ERR_ARG;
        tot += p->tier_probs[k];
    }
    if (!(tot > 0.0)) return TG_ERR_ARG;
    return TG_OK;
}

/* Writes num_requests records sorted by arrival (ties keep index order). */
int tg_generate(const tg_params_t *p, uint32_t *arrival_us, uint16_t *prompt_len,
                uint16_t *output_len, uint8_t *tier) {
    int rc = validate(p);
    if (rc) return rc;
    rng_t r;
    rng_seed(&r, p->seed);
    double cdf[TG_MAX_TIERS], tot = 0.0;
    for (int k = 0; k < p->num_tiers; ++k) { tot += p->tier_probs[k]; cdf[k] = tot; }
    const double mean_gap_s = 1.0 / p->rate_per_s;
    const double shape = (p->arrival_kind == TG_ARRIVAL_GAMMA) ? 1.0 / (p->gamma_cv * p->gamma_cv) : 1.0;
    double now_s = 0.0;
    for (int64_t i = 0; i < p->num_requests; ++i) {
        double gap;
        if (p->arrival_kind == TG_ARRIVAL_POISSON) gap = -log(rng_uniform(&r)) * mean_gap_s;
        else gap = rng_gamma(&r, shape) * (mean_gap_s / shape);
        now_s += gap;
        double us = floor(now_s * 1e6 + 0.5);
        if (us > 4294967294.0) return TG_ERR_OVERFLOW;
        arrival_us[i] = (uint32_t)us;
        double u = rng_uniform(&r) * tot;
        int k = 0;
        while (k < p->num_tiers - 1 && u >= cdf[k]) ++k;
        tier[i] = (uint8_t)k;
        prompt_len[i] = (uint16_t)clipped_lognormal(&r, p->prompt_mu, p->prompt_sigma, p->prompt_min, p->prompt_max);
        output_len[i] = (uint16_t)clipped_lognormal(&r, p->output_mu, p->output_sigma, p->output_min, p->output_max);
    }
    return TG_OK;
}

/* ------------------------------------------------------- many replicas --- */
typedef struct {
    int nrep;
    const tg_params_t *params;
    const int64_t *offsets;
    uint32_t *arrival_us;
    uint16_t *prompt_len, *output_len;
    uint8_t *tier;
    int next;
    int rc;
    pthread_mutex_t mu;
} job_t;

static void *worker(void *arg) {
    job_t *j = (job_t *)arg;
    for (;;) {
        pthread_mutex_lock(&j->mu);
        int r = j->next++;
        pthread_mutex_unlock(&j->mu);
        if (r >= j->nrep) break;
        int64_t o = j->offsets[r];
        int rc = TG_OK;
        if (j->offsets[r + 1] - o != j->params[r].num_requests) rc = TG_ERR_ARG;
        else rc = tg_generate(&j->params[r], j->arrival_us + o, j->prompt_len + o, j->output_len + o, j->tier + o);
        if (rc) {
            pthread_mutex_lock(&j->mu);
            if (!j->rc) j->rc = rc;
            pthread_mutex_unlock(&j->mu);
        }
    }
    return NULL;
}

/* Generates every replica's trace into one concatenated SoA; replica r owns
 * records [offsets[r], offsets[r+1]).  Replicas are independent streams, so
 * the result does not depend on nthreads. */
int tg_generate_many(int nrep, const tg_params_t *params, const int64_t *offsets,
                     uint32_t *arrival_us, uint16_t *prompt_len, uint16_t *output_len,
                     uint8_t *tier, int nthreads) {
    if (nrep < 0 || !params || !offsets) return TG_ERR_ARG;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    job_t j;
    memset(&j, 0, sizeof j);
    j.nrep = nrep; j.params = params; j.offsets = offsets;
    j.arrival_us = arrival_us; j.prompt_len = prompt_len; j.output_len = output_len; j.tier = tier;
    pthread_mutex_init(&j.mu, NULL);
    pthread_t th[256];
    int started = 0;
    for (int i = 0; i < nthreads - 1; ++i)
        if (pthread_create(&th[started], NULL, worker, &j) == 0) ++started;
    worker(&j);
    for (int i = 0; i < started; ++i) pthread_join(th[i], NULL);
    pthread_mutex_destroy(&j.mu);
    return j.rc;
}

/* Monte-Carlo mean of a clipped, rounded lognormal (used to turn a target
 * load into an arrival rate).  Deterministic for a given seed. */
double tg_mean_clipped_lognormal(double mu, double sigma, int32_t lo, int32_t hi,
                                 int64_t nsamples, uint64_t seed) {
    rng_t r;
    rng_seed(&r, seed);
    double acc = 0.0;
    for (int64_t i = 0; i < nsamples; ++i) acc += (double)clipped_lognormal(&r, mu, sigma, lo, hi);
    return nsamples > 0 ? acc / (double)nsamples : 0.0;
}

/* SplitMix64 finaliser exposed for deriving per-replica seeds. */
uint64_t tg_mix_seed(uint64_t a, uint64_t b) {
    uint64_t s = a * 0x9E3779B97F4A7C15ULL ^ (b + 0x632BE59BD9B4E019ULL);
    return splitmix64_next(&s);
}
