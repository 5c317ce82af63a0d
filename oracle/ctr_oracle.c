/*
 * ctr_oracle.c -- CPU oracle for the marginal-cost routing simulation of
 * "Calibrate, Then Route" (arXiv 2609.16206).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load this library.  The
 * product path (the CUDA library under paper_2609_16206_gb300/) never does,
 * and this file shares no code, header, table or constant generator with it.
 *
 * Plain, slow, single-threaded, int64 (fp64 for the scorer), written for
 * checking by eye:
 *   - Philox4x32-10 counter-based generator (Salmon et al., SC'11, sec. 3).
 *   - Deterministic fp32 log / exp (argument reduction + series) and the
 *     normal quantile of Wichura, Applied Statistics AS241 (PPND16, 1988),
 *     the precision in which the trace's integer decisions are defined.
 *   - The synthetic request trace: lognormal prompt / output lengths, a noisy
 *     output-length prediction (sec. III-C) and Poisson or two-state
 *     Markov-modulated Poisson arrivals, all in integer microseconds.
 *   - The routing simulator of sec. III-D: explicit prefill and decode pools,
 *     KV transfer delay, continuous decode batching (sec. VI), the
 *     marginal-cost router of sec. III-A (the cost(d) display and
 *     Algorithm 1) and the sec. IV-C baselines, driven by ONE global
 *     binary heap of events.  Per-instance aggregates (queue length,
 *     remaining work, resident KV) are recomputed from per-request state
 *     by scanning, never kept as running counters.
 *   - SLO goodput and nearest-rank P99 TTFT and TPOT (sec. IV-B, Table 2) by sorting.
 *   - The standalone fp64 brute-force request x instance scorer.
 *
 * Every function names the passage it follows.  Where the paper is silent
 * the reading taken is the one written in the project's design notes; each
 * such reading is flagged "[reading]" below.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>

#define ORC_OK 0
#define ORC_EINVAL (-1)
#define ORC_ENOMEM (-2)
#define ORC_EOVERFLOW (-3)
#define ORC_ETIMEOUT (-4)

#define T_LIMIT (((int64_t)1) << 40)     /* every simulated time must stay below 2^40 us */
#define ARR_LIMIT (((int64_t)1) << 39)   /* arrival times must be below 2^39 us */
#define B_CLAMP (((int64_t)1) << 40)     /* backlog clamp of the fixed-point cost */
#define P_CLAMP (((int64_t)1) << 18)     /* pressure clamp (2^16 == 100 %) */

/* ======================================================================
 * Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as
 * easy as 1, 2, 3", SC'11, sec. 3.3): 10 rounds of two 32x32->64 products,
 * the key bumped by the Weyl constants between rounds.
 * ==================================================================== */
void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2], uint32_t out[4])
{
    uint32_t c[4] = {ctr_in[0], ctr_in[1], ctr_in[2], ctr_in[3]};
    uint32_t k0 = key_in[0], k1 = key_in[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += 0x9E3779B9u;
            k1 += 0xBB67AE85u;
        }
        uint64_t prod0 = (uint64_t)0xD2511F53u * (uint64_t)c[0];
        uint64_t prod1 = (uint64_t)0xCD9E8D57u * (uint64_t)c[2];
        uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
        uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
        uint32_t n0 = hi1 ^ c[1] ^ k0;
        uint32_t n2 = hi0 ^ c[3] ^ k1;
        c[0] = n0;
        c[1] = lo1;
        c[2] = n2;
        c[3] = lo0;
    }
    out[0] = c[0]; out[1] = c[1]; out[2] = c[2]; out[3] = c[3];
}

/* ======================================================================
 * Deterministic fp32 elementary functions.  The trace's floating point only
 * decides integers (lengths, gaps), so it is defined in the kernel's
 * precision, fp32: only +, -, *, / and sqrt, each correctly rounded by IEEE
 * 754, in a fixed order (built with -ffp-contract=off so nothing is fused).
 * [reading: the paper fixes no numerics for its trace.]
 * ==================================================================== */
static float bits_to_f32(uint32_t b) { float f; memcpy(&f, &b, 4); return f; }
static uint32_t f32_to_bits(float f) { uint32_t b; memcpy(&b, &f, 4); return b; }

/* ln 2 split for Cody-Waite reduction: HI carries 16 significant bits, so
 * e * HI is exact for |e| < 2^8; LO is the rounded remainder. */
static const float ORC_LN2_HI = 0x1.62e4p-1f;
static const float ORC_LN2_LO = 0x1.7f7d1cp-20f;
static const float ORC_INV_LN2 = 0x1.715476p+0f;
static const float ORC_SQRT2 = 0x1.6a09e6p+0f;

/* log: x = m * 2^e with m in (sqrt(1/2), sqrt(2)]; with s = (m-1)/(m+1),
 * ln m = 2 s * sum_{i=0..5} s^(2i) / (2i+1) (|s| <= 0.1716: the next term is
 * below 2^-26 of the sum). */
float orc_det_logf(float x)
{
    static const float inv_odd[6] = {0x1p+0f, 0x1.555556p-2f, 0x1.99999ap-3f, 0x1.24924ap-3f, 0x1.c71c72p-4f,
                                     0x1.745d18p-4f};
    uint32_t b = f32_to_bits(x);
    int32_t e = (int32_t)((b >> 23) & 0xffu) - 127;
    float m = bits_to_f32((b & 0x007FFFFFu) | 0x3F800000u);
    if (m > ORC_SQRT2) {
        m = m * 0.5f;
        e = e + 1;
    }
    float f = m - 1.0f;
    float s = f / (m + 1.0f);
    float z = s * s;
    float poly = inv_odd[5];
    for (int i = 4; i >= 0; --i) poly = poly * z + inv_odd[i];
    float log_m = (s + s) * poly;
    float ed = (float)e;
    return ed * ORC_LN2_HI + (ed * ORC_LN2_LO + log_m);
}

/* exp: x = k ln2 + r with k = nearest integer to x / ln2 (halves away from
 * zero), |r| <= ln2 / 2; e^r by its Taylor series to degree 7 (remainder
 * below 2^-27), scaled by 2^k through the exponent field; x clamped to
 * [-87, 88] so 2^k stays a normal number. */
float orc_det_expf(float x)
{
    static const float inv_fact[8] = {0x1p+0f, 0x1p+0f, 0x1p-1f, 0x1.555556p-3f, 0x1.555556p-5f, 0x1.111112p-7f,
                                      0x1.6c16c2p-10f, 0x1.a01a02p-13f};
    if (x > 88.0f) x = 88.0f;
    if (x < -87.0f) x = -87.0f;
    float kf = x * ORC_INV_LN2;
    int32_t k = (int32_t)(kf >= 0.0f ? kf + 0.5f : kf - 0.5f);
    float kd = (float)k;
    float r = (x - kd * ORC_LN2_HI) - kd * ORC_LN2_LO;
    float poly = inv_fact[7];
    for (int i = 6; i >= 0; --i) poly = poly * r + inv_fact[i];
    return poly * bits_to_f32((uint32_t)(k + 127) << 23);
}

/* The uniform of a 32-bit word: (u + 1/2) 2^-32, rounded once to fp32.  Its
 * complement 1 - U is the same construction applied to ~u, so a tail never
 * needs a cancelling subtraction. */
float orc_unit_uniform(uint32_t u) { return (float)(int64_t)(2 * (uint64_t)u + 1) * 0x1p-33f; }

/* Normal quantile of U(u), Wichura (1988) AS241 PPND16 evaluated in fp32: a
 * degree-7 rational function of r = 0.180625 - q^2 for |q| = |U - 1/2| <= 0.425,
 * otherwise of r = sqrt(-ln min(U, 1-U)) shifted by 1.6 (r <= 5) or by 5. */
static const float AS241_A[8] = {0x1.b18d92p+1f, 0x1.0a4888p+7f, 0x1.ece5d2p+10f, 0x1.ad1d8cp+13f,
                                 0x1.66c3e8p+15f, 0x1.06c1c6p+16f, 0x1.052d26p+15f, 0x1.39a296p+11f};
static const float AS241_B[8] = {0x1p+0f, 0x1.5281b4p+5f, 0x1.5797fp+9f, 0x1.512322p+12f,
                                 0x1.4b772ep+14f, 0x1.3317cap+15f, 0x1.c0e458p+14f, 0x1.46a7ecp+12f};
static const float AS241_C[8] = {0x1.6c666p+0f, 0x1.285774p+2f, 0x1.713f72p+2f, 0x1.d2ecb2p+1f,
                                 0x1.453ccp+0f, 0x1.ef2abcp-3f, 0x1.744eb6p-6f, 0x1.9615acp-11f};
static const float AS241_D[8] = {0x1p+0f, 0x1.06cefcp+1f, 0x1.ad278ep+0f, 0x1.61293p-1f,
                                 0x1.2f5124p-3f, 0x1.f207a8p-7f, 0x1.1f18ccp-11f, 0x1.20d3f6p-30f};
static const float AS241_E[8] = {0x1.aa1b1cp+2f, 0x1.5daea6p+2f, 0x1.c8ea64p+0f, 0x1.2fad94p-2f,
                                 0x1.b2b412p-6f, 0x1.45c19p-10f, 0x1.c6ec6cp-16f, 0x1.afb74ep-23f};
static const float AS241_F[8] = {0x1p+0f, 0x1.331d34p-1f, 0x1.186eb2p-3f, 0x1.e76f94p-7f,
                                 0x1.9c8bcap-11f, 0x1.35c2c4p-16f, 0x1.31447p-23f, 0x1.269cp-49f};

static float horner7(const float c[8], float r)
{
    float acc = c[7];
    for (int i = 6; i >= 0; --i) acc = acc * r + c[i];
    return acc;
}

float orc_det_ndtrif(uint32_t u)
{
    int64_t c = 2 * (int64_t)u + 1 - 4294967296LL; /* 2^33 (U - 1/2), odd, never 0 */
    float q = (float)c * 0x1p-33f;
    float aq = q < 0.0f ? -q : q;
    if (aq <= 0x1.b33334p-2f /* 0.425 */) {
        float r = 0x1.71eb86p-3f /* 0.180625 */ - q * q;
        return (q * horner7(AS241_A, r)) / horner7(AS241_B, r);
    }
    float tail = c < 0 ? orc_unit_uniform(u) : orc_unit_uniform(~u);
    float r = sqrtf(-orc_det_logf(tail));
    float v;
    if (r <= 5.0f) {
        r = r - 0x1.99999ap+0f; /* 1.6 */
        v = horner7(AS241_C, r) / horner7(AS241_D, r);
    } else {
        r = r - 5.0f;
        v = horner7(AS241_E, r) / horner7(AS241_F, r);
    }
    return c < 0 ? -v : v;
}

/* vectorised entry points for the pin tests */
void orc_det_logf_v(const float* x, float* y, int64_t n) { for (int64_t i = 0; i < n; ++i) y[i] = orc_det_logf(x[i]); }
void orc_det_expf_v(const float* x, float* y, int64_t n) { for (int64_t i = 0; i < n; ++i) y[i] = orc_det_expf(x[i]); }
void orc_det_ndtrif_v(const uint32_t* u, float* y, int64_t n) { for (int64_t i = 0; i < n; ++i) y[i] = orc_det_ndtrif(u[i]); }
void orc_unit_uniform_v(const uint32_t* u, float* y, int64_t n) { for (int64_t i = 0; i < n; ++i) y[i] = orc_unit_uniform(u[i]); }

/* ======================================================================
 * Synthetic trace (the workloads of Table 1 as length laws; sec. III-C
 * predictor with injected multiplicative noise, sec. V-G).  [reading: the
 * paper gives length profiles only; the laws, the counter layout and the
 * integer arrival construction are the spec's.]
 * ==================================================================== */
typedef struct {
    uint64_t seed;            /* replica g draws with key seed + (g mod n_seeds) */
    int64_t n_seeds;          /* >= 1; sub-stream of replica g is g / n_seeds */
    int64_t arrival_kind;     /* 0 Poisson, 1 two-state MMPP (low state first) */
    int64_t rate_mreq[2];     /* arrival rate in milli-requests per second */
    int64_t dwell_mean_us;    /* MMPP mean state dwell */
    double prompt_mu, prompt_sigma;
    int64_t prompt_min, prompt_max;
    uint64_t mix_short_thr;   /* P(short output component) * 2^32 */
    double short_mu, short_sigma, long_mu, long_sigma;
    int64_t out_min, out_max;
    double noise_sigma;
    int64_t pred_min, pred_max;
    int64_t n_classes;
    uint64_t class_thr[3];    /* cumulative class probabilities * 2^32 */
} orc_trace_cfg;

/* clip(floor(v + 1/2), lo, hi) for v >= 0 (NaN / inf / huge -> hi) */
static int64_t round_clip(float v, int64_t lo, int64_t hi)
{
    float y = v + 0.5f;
    if (!(y < (float)hi)) return hi;
    int64_t t = (int64_t)y;
    return t < lo ? lo : t;
}

static void draw(const orc_trace_cfg* cfg, uint64_t sub, uint32_t stream, uint64_t idx, uint32_t group,
                 uint32_t out[4])
{
    uint64_t g_seed = cfg->seed; /* caller folds the replica seed in */
    uint32_t key[2] = {(uint32_t)g_seed, (uint32_t)(g_seed >> 32)};
    uint32_t ctr[4] = {(uint32_t)idx, (uint32_t)sub, stream, group};
    orc_philox4x32_10(ctr, key, out);
}

/* MMPP state dwell j (stream 1): floor(-ln U * mean) microseconds */
static int64_t dwell_us(const orc_trace_cfg* cfg, uint64_t sub, uint64_t j)
{
    uint32_t x[4];
    draw(cfg, sub, 1u, j, 0u, x);
    float g = orc_det_logf(orc_unit_uniform(x[0]));
    return (int64_t)((-g) * (float)cfg->dwell_mean_us);
}

/* One replica (global index g) of n requests, written to the five arrays. */
int orc_gen_trace(const orc_trace_cfg* cfg_in, int64_t g, int64_t n, int64_t* arrival, int32_t* prompt,
                  int32_t* out_len, int32_t* pred, uint8_t* cls)
{
    if (cfg_in->n_seeds < 1 || cfg_in->rate_mreq[0] < 1 || cfg_in->rate_mreq[1] < 1) return ORC_EINVAL;
    orc_trace_cfg cfg = *cfg_in;
    cfg.seed = cfg_in->seed + (uint64_t)(g % cfg_in->n_seeds);
    uint64_t sub = (uint64_t)(g / cfg_in->n_seeds);

    int64_t lambda = 0;                     /* cumulative unit-rate work, nano-events */
    /* MMPP: interval j covers [T_j, T_j + D_j) during which the cumulative
     * work grows from A_j at rate rate[j mod 2] (milli-req/s * us = nano-events) */
    int64_t j = 0, T = 0, A = 0, D = 0, A_next = 0;
    if (cfg.arrival_kind == 1) {
        D = dwell_us(&cfg, sub, 0);
        A_next = A + cfg.rate_mreq[0] * D;
    }
    for (int64_t k = 0; k < n; ++k) {
        uint32_t x[4], y[4];
        draw(&cfg, sub, 0u, (uint64_t)k, 0u, x);
        draw(&cfg, sub, 0u, (uint64_t)k, 1u, y);

        float zp = orc_det_ndtrif(x[0]);
        int64_t p = round_clip(orc_det_expf((float)cfg.prompt_mu + (float)cfg.prompt_sigma * zp), cfg.prompt_min,
                               cfg.prompt_max);

        int is_short = (uint64_t)x[1] < cfg.mix_short_thr;
        float mu = is_short ? (float)cfg.short_mu : (float)cfg.long_mu;
        float sg = is_short ? (float)cfg.short_sigma : (float)cfg.long_sigma;
        float zo = orc_det_ndtrif(x[2]);
        int64_t o = round_clip(orc_det_expf(mu + sg * zo), cfg.out_min, cfg.out_max);

        float zn = orc_det_ndtrif(x[3]);
        float factor = orc_det_expf((float)cfg.noise_sigma * zn);
        int64_t oh = round_clip((float)o * factor, cfg.pred_min, cfg.pred_max);

        int64_t c = 0;
        while (c < cfg.n_classes - 1 && (uint64_t)y[0] >= cfg.class_thr[c]) c++;

        float lg = orc_det_logf(orc_unit_uniform(y[1]));
        int64_t gap = (int64_t)((-lg) * 0x1.dcd65p+29f /* 1e9 */);
        lambda += gap;

        int64_t t;
        if (cfg.arrival_kind == 0) {
            t = lambda / cfg.rate_mreq[0];
        } else {
            while (lambda >= A_next) { /* the last interval j with A_j <= lambda */
                T += D;
                A = A_next;
                j += 1;
                D = dwell_us(&cfg, sub, (uint64_t)j);
                A_next = A + cfg.rate_mreq[j & 1] * D;
            }
            t = T + (lambda - A) / cfg.rate_mreq[j & 1];
        }
        arrival[k] = t;
        prompt[k] = (int32_t)p;
        out_len[k] = (int32_t)o;
        pred[k] = (int32_t)oh;
        cls[k] = (uint8_t)c;
    }
    return ORC_OK;
}

/* ======================================================================
 * Routing simulator (sec. III-D; decode continuous batching of sec. VI;
 * cost of sec. III-A; baselines of sec. IV-C).
 * ==================================================================== */
typedef struct {
    int64_t n_prefill, n_decode;
    int64_t kv_cap;                        /* KV tokens per decode instance */
    int64_t pre_base, pre_per_tok;         /* prefill service = base + per_tok * p */
    int64_t xfer_per_tok;                  /* KV transfer delay = per_tok * p */
    int64_t dec_base, dec_per_seq, dec_kv_div; /* step = base + per_seq*n + floor(KV/div) */
    int64_t n_classes;
    int64_t ttft[4], tpot[4];
    int64_t max_steps;                     /* decode steps allowed per decode instance */
    int64_t cap_pending, cap_waiting, cap_active, cap_prefill; /* 0 = unlimited */
    int64_t heur_thresh;
    int64_t pre_batch_tokens;              /* 0: serial FCFS prefill; > 0: batched prefill with this token budget */
} orc_sim_cfg;

typedef struct {
    int64_t tau_pre0, tau_pre, tau_dec, w_q;
    int64_t w_b_q8, w_s_q8, rho_q8, sigma_q8[4];
    int64_t ablate; /* bit 0: predicted length, bit 1: KV pressure, bit 2: SLO class (sec. V-F) */
    int64_t proxy_backlog; /* 1: backlog from the proxy's priced in-flight ledger (sec. IV-A, VI) */
    int64_t poll_us;       /* > 0: KV occupancy seen as polled every poll_us (sec. IV-A); 0: live */
} orc_consts;

typedef struct {
    int64_t max_pending, max_waiting, max_active, max_prefill; /* peak occupancy seen */
    int64_t max_reserved;                  /* peak reserved KV on any decode instance */
    int64_t steps;                         /* decode steps over all instances */
    int64_t events;                        /* heap events processed */
} orc_stats;

enum { POL_LEARNED = 0, POL_RR = 1, POL_JSQ = 2, POL_HEUR = 3, POL_LEARNED_P2 = 4 };
enum { EV_STEP_END = 0, EV_PREFILL_END = 1, EV_KV_READY = 2 };
enum { ST_NONE = 0, ST_PENDING = 1, ST_WAITING = 2, ST_ACTIVE = 3, ST_DONE = 4 };

typedef struct { int64_t t; int64_t kind; int64_t k; int64_t inst; } ev_t;

typedef struct { ev_t* a; int64_t n, cap; } heap_t;

static int ev_less(const ev_t* x, const ev_t* y)
{
    if (x->t != y->t) return x->t < y->t;
    if (x->kind != y->kind) return x->kind < y->kind;
    if (x->k != y->k) return x->k < y->k;
    return x->inst < y->inst;
}

static int heap_push(heap_t* h, ev_t e)
{
    if (h->n == h->cap) {
        int64_t nc = h->cap ? 2 * h->cap : 64;
        ev_t* na = (ev_t*)realloc(h->a, (size_t)nc * sizeof(ev_t));
        if (!na) return ORC_ENOMEM;
        h->a = na;
        h->cap = nc;
    }
    int64_t i = h->n++;
    h->a[i] = e;
    while (i > 0) {
        int64_t parent = (i - 1) / 2;
        if (!ev_less(&h->a[i], &h->a[parent])) break;
        ev_t tmp = h->a[i]; h->a[i] = h->a[parent]; h->a[parent] = tmp;
        i = parent;
    }
    return ORC_OK;
}

static ev_t heap_pop(heap_t* h)
{
    ev_t top = h->a[0];
    h->a[0] = h->a[--h->n];
    int64_t i = 0;
    for (;;) {
        int64_t l = 2 * i + 1, r = l + 1, m = i;
        if (l < h->n && ev_less(&h->a[l], &h->a[m])) m = l;
        if (r < h->n && ev_less(&h->a[r], &h->a[m])) m = r;
        if (m == i) break;
        ev_t tmp = h->a[i]; h->a[i] = h->a[m]; h->a[m] = tmp;
        i = m;
    }
    return top;
}

/* splitmix64 output mix (Steele, Lea, Flood, OOPSLA'14) */
static uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static uint64_t hash_term(int64_t k, uint64_t tag, uint64_t v)
{
    return mix64(mix64((tag << 56) ^ (uint64_t)k) ^ v);
}

/* Order-independent row checksum: the 64-bit sum over requests of the
 * routing, first-token and completion terms. */
uint64_t orc_row_hash(int64_t n, const uint8_t* i_pre, const uint8_t* i_dec, const int64_t* t_first,
                      const int64_t* t_done)
{
    uint64_t h = 0;
    for (int64_t k = 0; k < n; ++k) {
        h += hash_term(k, 1, ((uint64_t)i_pre[k] << 8) | (uint64_t)i_dec[k]);
        h += hash_term(k, 2, (uint64_t)t_first[k]);
        h += hash_term(k, 3, (uint64_t)t_done[k]);
    }
    return h;
}

typedef struct {
    const orc_sim_cfg* cfg;
    const orc_consts* cc;
    int64_t policy, n;
    const int64_t* arr; const int32_t* p; const int32_t* o; const int32_t* oh; const uint8_t* cls;
    /* per request */
    int64_t* stage; int64_t* gen; int64_t* dec_of;
    /* per decode instance: committed (routed here, not done) request lists */
    int64_t** committed; int64_t* n_committed;
    int64_t** fifo; int64_t* fifo_head; int64_t* fifo_tail;
    int64_t* stepping; int64_t* steps;
    /* per prefill instance: in-flight (routed, prefill not ended) request lists */
    int64_t* busy; int64_t* inflight; int64_t** pre_list;
    /* KV occupancy of each decode instance at the last poll instant */
    int64_t* polled_kv;
    /* batched prefill: per instance the FIFO of requests not yet in a batch
     * and the members of the running batch */
    int64_t** pfifo; int64_t* pfifo_head; int64_t* pfifo_tail;
    int64_t** prun; int64_t* prun_n; int64_t* prun_end; int64_t* prun_on;
    heap_t heap;
    orc_stats* st;
    int64_t* admitted;
    /* outputs */
    uint8_t* i_pre; uint8_t* i_dec; int64_t* t_first; int64_t* t_done; int64_t* pre_end; int64_t* t_ready;
} sim_t;

/* aggregates of a decode instance, recomputed from per-request state */
static int64_t dec_active(const sim_t* s, int64_t d)
{
    int64_t c = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) c += s->stage[s->committed[d][i]] == ST_ACTIVE;
    return c;
}
static int64_t dec_reserved(const sim_t* s, int64_t d)
{
    int64_t r = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) {
        int64_t j = s->committed[d][i];
        if (s->stage[j] == ST_ACTIVE) r += (int64_t)s->p[j] + (int64_t)s->o[j];
    }
    return r;
}
static int64_t dec_resident(const sim_t* s, int64_t d)
{
    int64_t r = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) {
        int64_t j = s->committed[d][i];
        if (s->stage[j] == ST_ACTIVE) r += (int64_t)s->p[j] + s->gen[j];
    }
    return r;
}
static int64_t dec_remaining(const sim_t* s, int64_t d)
{
    int64_t r = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) {
        int64_t j = s->committed[d][i];
        r += (int64_t)s->o[j] - s->gen[j];
    }
    return r;
}
static int64_t dec_pred_sum(const sim_t* s, int64_t d)
{
    int64_t r = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) r += (int64_t)s->oh[s->committed[d][i]];
    return r;
}
static int64_t dec_pending(const sim_t* s, int64_t d)
{
    int64_t c = 0;
    for (int64_t i = 0; i < s->n_committed[d]; ++i) c += s->stage[s->committed[d][i]] == ST_PENDING;
    return c;
}

static int64_t step_time(const orc_sim_cfg* cfg, int64_t n_active, int64_t resident)
{
    return cfg->dec_base + cfg->dec_per_seq * n_active + resident / cfg->dec_kv_div;
}

/* decode step end at t: every active request gains one token; those that
 * reach their true output length complete and release their KV */
static void on_step_end(sim_t* s, int64_t d, int64_t t)
{
    for (int64_t i = 0; i < s->n_committed[d]; ++i) {
        int64_t j = s->committed[d][i];
        if (s->stage[j] == ST_ACTIVE) s->gen[j] += 1;
    }
    int64_t i = 0;
    while (i < s->n_committed[d]) {
        int64_t j = s->committed[d][i];
        if (s->stage[j] == ST_ACTIVE && s->gen[j] == (int64_t)s->o[j]) {
            s->stage[j] = ST_DONE;
            s->t_done[j] = t;
            s->committed[d][i] = s->committed[d][--s->n_committed[d]];
        } else {
            ++i;
        }
    }
    s->stepping[d] = 0;
}

/* at a step boundary or while idle: admit strictly FCFS from the waiting
 * queue while the reservation p + o fits the KV capacity, then start a step
 * if anything is active.  Returns a status. */
static int admit_and_start(sim_t* s, int64_t d, int64_t t)
{
    const orc_sim_cfg* cfg = s->cfg;
    int64_t n_adm = 0;
    while (s->fifo_head[d] < s->fifo_tail[d]) {
        int64_t h = s->fifo[d][s->fifo_head[d]];
        int64_t need = (int64_t)s->p[h] + (int64_t)s->o[h];
        if (dec_reserved(s, d) + need > cfg->kv_cap) break;
        s->fifo_head[d]++;
        s->stage[h] = ST_ACTIVE;
        s->gen[h] = 0;
        s->admitted[n_adm++] = h;
        int64_t na = dec_active(s, d);
        if (na > s->st->max_active) s->st->max_active = na;
        if (cfg->cap_active > 0 && na > cfg->cap_active) return ORC_EOVERFLOW;
        int64_t rs = dec_reserved(s, d);
        if (rs > s->st->max_reserved) s->st->max_reserved = rs;
    }
    int64_t na = dec_active(s, d);
    if (na == 0) return ORC_OK;
    s->steps[d] += 1;
    s->st->steps += 1;
    if (s->steps[d] > cfg->max_steps) return ORC_ETIMEOUT;
    int64_t end = t + step_time(cfg, na, dec_resident(s, d));
    if (end >= T_LIMIT) return ORC_EOVERFLOW;
    ev_t e = {end, EV_STEP_END, -1, d};
    if (heap_push(&s->heap, e)) return ORC_ENOMEM;
    s->stepping[d] = 1;
    for (int64_t i = 0; i < n_adm; ++i) s->t_first[s->admitted[i]] = end;
    return ORC_OK;
}

static int64_t argmin_lowest(const int64_t* v, int64_t n)
{
    int64_t best = 0;
    for (int64_t i = 1; i < n; ++i)
        if (v[i] < v[best]) best = i;
    return best;
}

/* B_d = floor(R_d * step_d / max(1, n_d)), saturated at 2^40 [reading: the
 * true remaining work of sec. VI, priced at the current batch step time] */
static int64_t decode_backlog(int64_t remaining, int64_t step, int64_t n_active)
{
    unsigned __int128 prod = (unsigned __int128)(uint64_t)remaining * (uint64_t)step;
    if (prod >= ((unsigned __int128)1 << 62)) return B_CLAMP;
    int64_t b = (int64_t)prod / (n_active > 1 ? n_active : 1);
    return b < B_CLAMP ? b : B_CLAMP;
}

/* Power-of-two candidates [reading: the paper names the sampled variant only].
 * Philox4x32-10 with key (0x243F6A88, 0x85A308D3) and counter
 * (k, t lo, t hi, 0x5032) gives words u0..u3; a pool of n instances offers
 * c0 = floor(u * n / 2^32) and c1 = (c0 + 1 + floor(u' (n - 1) / 2^32)) mod n
 * (distinct when n > 1), decode from (u0, u1), prefill from (u2, u3). */
static void p2_words(int64_t k, int64_t t, uint32_t out[4])
{
    uint32_t ctr[4] = {(uint32_t)k, (uint32_t)t, (uint32_t)((uint64_t)t >> 32), 0x5032u};
    uint32_t key[2] = {0x243F6A88u, 0x85A308D3u};
    orc_philox4x32_10(ctr, key, out);
}

static void p2_pair(uint32_t u, uint32_t v, int64_t n, int64_t c[2])
{
    c[0] = (int64_t)(((uint64_t)u * (uint64_t)n) >> 32);
    c[1] = n > 1 ? (c[0] + 1 + (int64_t)(((uint64_t)v * (uint64_t)(n - 1)) >> 32)) % n : c[0];
}

static void p2_candidates_dec(int64_t k, int64_t t, int64_t nd, int64_t c[2])
{
    uint32_t w[4];
    p2_words(k, t, w);
    p2_pair(w[0], w[1], nd, c);
}

static void p2_candidates(int64_t k, int64_t t, int64_t np, int64_t c[2])
{
    uint32_t w[4];
    p2_words(k, t, w);
    p2_pair(w[2], w[3], np, c);
}

/* Batched prefill (sec. VI batches the prefill stage as well as the decode stage) [reading]:
 * an instance runs one batch at a time.  A batch takes, FCFS from the
 * instance's queue, the head request and then every next request while the
 * batch's prompt tokens stay within pre_batch_tokens; it lasts
 * pre_base + pre_per_tok * (sum of its prompts), and each member's KV transfer
 * starts when the batch ends.  A batch starts when the previous one ends (if
 * anything waits) or when a request reaches an idle instance. */
static int start_prefill_batch(sim_t* s, int64_t i, int64_t t)
{
    const orc_sim_cfg* cfg = s->cfg;
    int64_t tokens = 0;
    s->prun_n[i] = 0;
    while (s->pfifo_head[i] < s->pfifo_tail[i]) {
        int64_t j = s->pfifo[i][s->pfifo_head[i]];
        if (s->prun_n[i] > 0 && tokens + (int64_t)s->p[j] > cfg->pre_batch_tokens) break;
        tokens += s->p[j];
        s->prun[i][s->prun_n[i]++] = j;
        s->pfifo_head[i]++;
    }
    int64_t end = t + cfg->pre_base + cfg->pre_per_tok * tokens;
    if (end >= T_LIMIT) return ORC_EOVERFLOW;
    ev_t e = {end, EV_PREFILL_END, -1, i};
    if (heap_push(&s->heap, e)) return ORC_ENOMEM;
    for (int64_t m = 0; m < s->prun_n[i]; ++m) {
        int64_t j = s->prun[i][m];
        int64_t ready = end + cfg->xfer_per_tok * (int64_t)s->p[j];
        if (ready >= T_LIMIT) return ORC_EOVERFLOW;
        ev_t r = {ready, EV_KV_READY, j, s->dec_of[j]};
        if (heap_push(&s->heap, r)) return ORC_ENOMEM;
        s->pre_end[j] = end;
        s->t_ready[j] = ready;
    }
    s->prun_on[i] = 1;
    s->prun_end[i] = end;
    return ORC_OK;
}

/* True prefill backlog under batching [reading]: the time until the instance
 * would have served everything committed to it if nothing else arrived --
 * the rest of the running batch, then the queue cut into batches by the same
 * FCFS token-budget rule, each costing base + per_tok * its prompt tokens.
 * Saturates at 2^40. */
static int64_t batched_backlog_pre(const sim_t* s, int64_t i, int64_t t)
{
    const orc_sim_cfg* cfg = s->cfg;
    int64_t b = s->prun_on[i] && s->prun_end[i] > t ? s->prun_end[i] - t : 0;
    int64_t m = s->pfifo_head[i];
    while (m < s->pfifo_tail[i]) {
        int64_t tokens = 0, members = 0;
        while (m < s->pfifo_tail[i]) {
            int64_t pj = s->p[s->pfifo[i][m]];
            if (members > 0 && tokens + pj > cfg->pre_batch_tokens) break;
            tokens += pj;
            members++;
            m++;
        }
        b += cfg->pre_base + cfg->pre_per_tok * tokens;
        if (b >= B_CLAMP) return B_CLAMP;
    }
    return b;
}

/* Backlog as the deployed proxy sees it [reading: sec. IV-A's ledger of
 * in-flight requests, from which the proxy derives seconds of backlog, priced
 * with the router's own constants as sec. VI describes]: the sum over requests routed to the
 * instance and still in flight there of their priced work, each priced once
 * at admission and never decremented.  Prefill: tau_pre0 + tau_pre * p until
 * the prefill ends; decode: o_hat * tau_dec until the request completes (o_hat
 * taken as 0 when the predicted length is ablated).  Saturates at 2^40. */
static int64_t proxy_backlog_pre(const sim_t* s, int64_t i)
{
    int64_t b = 0;
    for (int64_t m = 0; m < s->inflight[i]; ++m) {
        b += s->cc->tau_pre0 + (int64_t)s->p[s->pre_list[i][m]] * s->cc->tau_pre;
        if (b >= B_CLAMP) return B_CLAMP;
    }
    return b;
}
static int64_t proxy_backlog_dec(const sim_t* s, int64_t d)
{
    if (s->cc->ablate & 1) return 0;
    int64_t b = 0;
    for (int64_t m = 0; m < s->n_committed[d]; ++m) {
        b += (int64_t)s->oh[s->committed[d][m]] * s->cc->tau_dec;
        if (b >= B_CLAMP) return B_CLAMP;
    }
    return b;
}

/* Route request k at time t (Algorithm 1) and commit it. */
static int route(sim_t* s, int64_t k, int64_t t)
{
    const orc_sim_cfg* cfg = s->cfg;
    const orc_consts* cc = s->cc;
    int64_t np = cfg->n_prefill, nd = cfg->n_decode;
    int64_t pk = s->p[k], ok = s->o[k], ohk = s->oh[k], ck = s->cls[k];
    int64_t cost_p[32], cost_d[32];
    int64_t ip = 0, id = 0;

    if (s->policy == POL_RR) {
        ip = k % np;
        id = k % nd;
    } else {
        int learned = s->policy == POL_LEARNED || s->policy == POL_LEARNED_P2;
        /* feature ablation (sec. V-F): a removed feature takes its neutral value */
        int64_t oh_f = (cc->ablate & 1) ? 0 : ohk;
        int64_t sig = (cc->ablate & 4) ? 256 : cc->sigma_q8[ck];
        for (int64_t i = 0; i < np; ++i) {
            int64_t q = s->inflight[i];
            if (learned) {
                int64_t b = s->busy[i] - t;
                if (b < 0) b = 0;
                if (b > B_CLAMP) b = B_CLAMP;
                if (cfg->pre_batch_tokens > 0) b = batched_backlog_pre(s, i, t);
                if (cc->proxy_backlog) b = proxy_backlog_pre(s, i);
                int64_t own = cc->tau_pre0 + pk * cc->tau_pre;
                int64_t load = cc->w_b_q8 * b + cc->w_s_q8 * own;
                cost_p[i] = load * sig + cc->w_q * q * 65536;
            } else {
                cost_p[i] = q; /* JSQ and the heuristic place prefill by queue length */
            }
        }
        for (int64_t d = 0; d < nd; ++d) {
            int64_t q = s->n_committed[d];
            if (learned) {
                int64_t na = dec_active(s, d);
                int64_t res = dec_resident(s, d);
                int64_t b = decode_backlog(dec_remaining(s, d), step_time(cfg, na, res), na);
                if (cc->proxy_backlog) b = proxy_backlog_dec(s, d);
                /* press+ from the occupancy the router sees: live, or the last poll */
                int64_t seen = cc->poll_us > 0 ? s->polled_kv[d] : res;
                int64_t press = ((seen + pk + oh_f) * 65536) / cfg->kv_cap;
                if (press > P_CLAMP) press = P_CLAMP;
                if (cc->ablate & 2) press = 0;
                int64_t own = oh_f * cc->tau_dec;
                int64_t priced = own + (((own * press) >> 16) * cc->rho_q8 >> 8);
                int64_t load = cc->w_b_q8 * b + cc->w_s_q8 * priced;
                cost_d[d] = load * sig + cc->w_q * q * 65536;
            } else if (s->policy == POL_HEUR && ohk >= cfg->heur_thresh) {
                cost_d[d] = dec_pred_sum(s, d);
            } else {
                cost_d[d] = q;
            }
        }
        if (s->policy == POL_LEARNED_P2) {
            /* power-of-two choices (sec. V-D, VI): only two sampled candidates per pool are priced */
            int64_t cp[2], cd[2];
            p2_candidates(k, t, np, cp);
            p2_candidates_dec(k, t, nd, cd);
            ip = cost_p[cp[1]] < cost_p[cp[0]] || (cost_p[cp[1]] == cost_p[cp[0]] && cp[1] < cp[0]) ? cp[1] : cp[0];
            id = cost_d[cd[1]] < cost_d[cd[0]] || (cost_d[cd[1]] == cost_d[cd[0]] && cd[1] < cd[0]) ? cd[1] : cd[0];
        } else {
            ip = argmin_lowest(cost_p, np);
            id = argmin_lowest(cost_d, nd);
        }
    }

    s->stage[k] = ST_PENDING;
    s->dec_of[k] = id;
    s->pre_list[ip][s->inflight[ip]++] = k;
    if (s->inflight[ip] > s->st->max_prefill) s->st->max_prefill = s->inflight[ip];
    if (cfg->cap_prefill > 0 && s->inflight[ip] > cfg->cap_prefill) return ORC_EOVERFLOW;
    if (cfg->pre_batch_tokens > 0) {
        /* batched: join the instance's queue; an idle instance starts a batch at once */
        s->pfifo[ip][s->pfifo_tail[ip]++] = k;
        if (!s->prun_on[ip]) {
            int rc = start_prefill_batch(s, ip, t);
            if (rc) return rc;
        }
    } else {
        /* serial FCFS: the prefill's start, end and KV-ready time in closed form */
        int64_t start = s->busy[ip] > t ? s->busy[ip] : t;
        int64_t end = start + cfg->pre_base + cfg->pre_per_tok * pk;
        int64_t ready = end + cfg->xfer_per_tok * pk;
        if (ready >= T_LIMIT) return ORC_EOVERFLOW;
        s->busy[ip] = end;
        ev_t e1 = {end, EV_PREFILL_END, k, ip};
        ev_t e2 = {ready, EV_KV_READY, k, id};
        if (heap_push(&s->heap, e1) || heap_push(&s->heap, e2)) return ORC_ENOMEM;
        s->pre_end[k] = end;
        s->t_ready[k] = ready;
    }
    s->committed[id][s->n_committed[id]++] = k;
    int64_t pend = dec_pending(s, id);
    if (pend > s->st->max_pending) s->st->max_pending = pend;
    if (cfg->cap_pending > 0 && pend > cfg->cap_pending) return ORC_EOVERFLOW;
    (void)ok;

    s->i_pre[k] = (uint8_t)ip;
    s->i_dec[k] = (uint8_t)id;
    return ORC_OK;
}

static int validate_requests(const orc_sim_cfg* cfg, int64_t n, const int64_t* arr, const int32_t* p,
                             const int32_t* o, const int32_t* oh, const uint8_t* cls)
{
    for (int64_t k = 0; k < n; ++k) {
        if (arr[k] < 0 || arr[k] >= ARR_LIMIT) return ORC_EINVAL;
        if (k > 0 && arr[k] < arr[k - 1]) return ORC_EINVAL;
        if (p[k] < 0 || p[k] > (1 << 20)) return ORC_EINVAL;
        if (o[k] < 1 || o[k] > (1 << 20)) return ORC_EINVAL;
        if ((int64_t)p[k] + (int64_t)o[k] > cfg->kv_cap) return ORC_EINVAL;
        if (oh[k] < 0 || oh[k] > (1 << 17)) return ORC_EINVAL;
        if ((int64_t)cls[k] >= cfg->n_classes) return ORC_EINVAL;
    }
    return ORC_OK;
}

static int validate_cfg(const orc_sim_cfg* cfg, const orc_consts* cc, int64_t policy)
{
    if (cfg->n_prefill < 1 || cfg->n_decode < 1 || cfg->n_prefill + cfg->n_decode > 32) return ORC_EINVAL;
    if (cfg->kv_cap < 1 || cfg->kv_cap > 2147483647LL) return ORC_EINVAL;
    if (cfg->dec_kv_div < 1 || cfg->pre_base < 1 || cfg->dec_base < 1) return ORC_EINVAL;
    if (cfg->n_classes < 1 || cfg->n_classes > 4) return ORC_EINVAL;
    if (policy < 0 || policy > 4) return ORC_EINVAL;
    if (cfg->pre_batch_tokens < 0 || cfg->pre_batch_tokens > ((int64_t)1 << 30)) return ORC_EINVAL;
    if (cc->ablate < 0 || cc->ablate > 7) return ORC_EINVAL;
    if (cc->proxy_backlog < 0 || cc->proxy_backlog > 1) return ORC_EINVAL;
    if (cc->poll_us < 0 || cc->poll_us > ARR_LIMIT) return ORC_EINVAL;
    if (cc->w_b_q8 < 0 || cc->w_b_q8 > 1023 || cc->w_s_q8 < 0 || cc->w_s_q8 > 1023) return ORC_EINVAL;
    if (cc->rho_q8 < 0 || cc->rho_q8 > 1023) return ORC_EINVAL;
    for (int i = 0; i < 4; ++i)
        if (cc->sigma_q8[i] < 0 || cc->sigma_q8[i] > 1023) return ORC_EINVAL;
    return ORC_OK;
}

/* Simulate one row (one replica under one policy and one constant set).
 * Outputs per request: prefill / decode instance, first-token and completion
 * times, and (for tests) prefill end and KV-ready times.  Returns a status. */
int orc_simulate(const orc_sim_cfg* cfg, const orc_consts* cc, int64_t policy, int64_t n, const int64_t* arr,
                 const int32_t* p, const int32_t* o, const int32_t* oh, const uint8_t* cls, uint8_t* i_pre,
                 uint8_t* i_dec, int64_t* t_first, int64_t* t_done, int64_t* pre_end, int64_t* t_ready,
                 uint64_t* hash, orc_stats* st)
{
    memset(st, 0, sizeof(*st));
    *hash = 0;
    int rc = validate_cfg(cfg, cc, policy);
    if (rc) return rc;
    rc = validate_requests(cfg, n, arr, p, o, oh, cls);
    if (rc) return rc;

    sim_t s;
    memset(&s, 0, sizeof(s));
    s.cfg = cfg; s.cc = cc; s.policy = policy; s.n = n;
    s.arr = arr; s.p = p; s.o = o; s.oh = oh; s.cls = cls;
    s.i_pre = i_pre; s.i_dec = i_dec; s.t_first = t_first; s.t_done = t_done; s.pre_end = pre_end;
    s.t_ready = t_ready; s.st = st;
    int64_t nd = cfg->n_decode, np = cfg->n_prefill;
    int64_t nn = n > 0 ? n : 1;
    s.stage = (int64_t*)calloc((size_t)nn, 8);
    s.gen = (int64_t*)calloc((size_t)nn, 8);
    s.dec_of = (int64_t*)calloc((size_t)nn, 8);
    s.admitted = (int64_t*)calloc((size_t)nn, 8);
    s.committed = (int64_t**)calloc((size_t)nd, sizeof(int64_t*));
    s.fifo = (int64_t**)calloc((size_t)nd, sizeof(int64_t*));
    s.n_committed = (int64_t*)calloc((size_t)nd, 8);
    s.fifo_head = (int64_t*)calloc((size_t)nd, 8);
    s.fifo_tail = (int64_t*)calloc((size_t)nd, 8);
    s.stepping = (int64_t*)calloc((size_t)nd, 8);
    s.steps = (int64_t*)calloc((size_t)nd, 8);
    s.busy = (int64_t*)calloc((size_t)np, 8);
    s.inflight = (int64_t*)calloc((size_t)np, 8);
    s.pre_list = (int64_t**)calloc((size_t)np, sizeof(int64_t*));
    s.polled_kv = (int64_t*)calloc((size_t)nd, 8);
    s.pfifo = (int64_t**)calloc((size_t)np, sizeof(int64_t*));
    s.prun = (int64_t**)calloc((size_t)np, sizeof(int64_t*));
    s.pfifo_head = (int64_t*)calloc((size_t)np, 8);
    s.pfifo_tail = (int64_t*)calloc((size_t)np, 8);
    s.prun_n = (int64_t*)calloc((size_t)np, 8);
    s.prun_end = (int64_t*)calloc((size_t)np, 8);
    s.prun_on = (int64_t*)calloc((size_t)np, 8);
    rc = ORC_OK;
    if (!s.stage || !s.gen || !s.dec_of || !s.admitted || !s.committed || !s.fifo || !s.n_committed ||
        !s.fifo_head || !s.fifo_tail || !s.stepping || !s.steps || !s.busy || !s.inflight || !s.pre_list ||
        !s.polled_kv || !s.pfifo || !s.prun || !s.pfifo_head || !s.pfifo_tail || !s.prun_n || !s.prun_end ||
        !s.prun_on)
        rc = ORC_ENOMEM;
    for (int64_t i = 0; i < np && rc == ORC_OK; ++i) {
        s.pre_list[i] = (int64_t*)calloc((size_t)nn, 8);
        s.pfifo[i] = (int64_t*)calloc((size_t)nn, 8);
        s.prun[i] = (int64_t*)calloc((size_t)nn, 8);
        if (!s.pre_list[i] || !s.pfifo[i] || !s.prun[i]) rc = ORC_ENOMEM;
    }
    for (int64_t d = 0; d < nd && rc == ORC_OK; ++d) {
        s.committed[d] = (int64_t*)calloc((size_t)nn, 8);
        s.fifo[d] = (int64_t*)calloc((size_t)nn, 8);
        if (!s.committed[d] || !s.fifo[d]) rc = ORC_ENOMEM;
    }
    for (int64_t k = 0; k < n; ++k) t_first[k] = t_done[k] = pre_end[k] = t_ready[k] = -1;

    int64_t ia = 0;
    int64_t next_poll = 0; /* occupancy polls at 0, poll_us, 2 poll_us, ... while arrivals remain */
    while (rc == ORC_OK) {
        int64_t t = INT64_MAX;
        if (s.heap.n > 0) t = s.heap.a[0].t;
        if (ia < n && arr[ia] < t) t = arr[ia];
        if (ia < n && cc->poll_us > 0 && next_poll < t) t = next_poll;
        if (t == INT64_MAX) break;
        /* (1) step ends, prefill ends and KV-ready events at t, KV-ready in
         * order of request index [reading: equal-time order] */
        while (s.heap.n > 0 && s.heap.a[0].t == t) {
            ev_t e = heap_pop(&s.heap);
            st->events += 1;
            if (e.kind == EV_STEP_END) {
                on_step_end(&s, e.inst, t);
            } else if (e.kind == EV_PREFILL_END && e.k < 0) {
                /* a prefill batch ends: all its members leave the instance */
                int64_t pi = e.inst;
                for (int64_t m = 0; m < s.prun_n[pi]; ++m) {
                    int64_t i = 0;
                    while (s.pre_list[pi][i] != s.prun[pi][m]) ++i;
                    s.pre_list[pi][i] = s.pre_list[pi][--s.inflight[pi]];
                }
                s.prun_n[pi] = 0;
                s.prun_on[pi] = 0;
            } else if (e.kind == EV_PREFILL_END) {
                int64_t i = 0;
                while (s.pre_list[e.inst][i] != e.k) ++i;
                s.pre_list[e.inst][i] = s.pre_list[e.inst][--s.inflight[e.inst]];
            } else {
                int64_t d = e.inst;
                s.stage[e.k] = ST_WAITING;
                s.fifo[d][s.fifo_tail[d]++] = e.k;
                int64_t w = s.fifo_tail[d] - s.fifo_head[d];
                if (w > st->max_waiting) st->max_waiting = w;
                if (cfg->cap_waiting > 0 && w > cfg->cap_waiting) rc = ORC_EOVERFLOW;
            }
        }
        if (rc) break;
        /* (2) admissions and step starts on every decode instance not mid-step,
         * and the next batch on every idle prefill instance with a queue */
        for (int64_t d = 0; d < nd && rc == ORC_OK; ++d)
            if (!s.stepping[d]) rc = admit_and_start(&s, d, t);
        for (int64_t i = 0; i < np && rc == ORC_OK && cfg->pre_batch_tokens > 0; ++i)
            if (!s.prun_on[i] && s.pfifo_head[i] < s.pfifo_tail[i]) rc = start_prefill_batch(&s, i, t);
        if (rc) break;
        /* the occupancy poll at t sees the state after every event at t and
         * before the arrivals at t [reading: equal-time order] */
        if (cc->poll_us > 0 && t == next_poll) {
            for (int64_t d = 0; d < nd; ++d) s.polled_kv[d] = dec_resident(&s, d);
            next_poll += cc->poll_us;
        }
        /* (3) arrivals at t, in order of request index */
        while (ia < n && arr[ia] == t && rc == ORC_OK) {
            rc = route(&s, ia, t);
            ia++;
        }
    }
    if (rc == ORC_OK) *hash = orc_row_hash(n, i_pre, i_dec, t_first, t_done);

    for (int64_t d = 0; d < nd; ++d) {
        if (s.committed) free(s.committed[d]);
        if (s.fifo) free(s.fifo[d]);
    }
    free(s.stage); free(s.gen); free(s.dec_of); free(s.admitted); free(s.committed); free(s.fifo);
    free(s.n_committed); free(s.fifo_head); free(s.fifo_tail); free(s.stepping); free(s.steps);
    for (int64_t i = 0; i < np; ++i) {
        if (s.pre_list) free(s.pre_list[i]);
        if (s.pfifo) free(s.pfifo[i]);
        if (s.prun) free(s.prun[i]);
    }
    free(s.busy); free(s.inflight); free(s.pre_list); free(s.polled_kv); free(s.heap.a);
    free(s.pfifo); free(s.prun); free(s.pfifo_head); free(s.pfifo_tail); free(s.prun_n); free(s.prun_end);
    free(s.prun_on);
    return rc;
}

/* ======================================================================
 * SLO goodput and P99 TTFT (sec. IV-B SLO targets; Table 2 columns).
 * met = TTFT <= TTFT_c and (o == 1 or t_done - t_first <= TPOT_c * (o - 1));
 * P99 is the nearest-rank value, sorted index ceil(0.99 N) - 1.
 * ==================================================================== */
static int cmp_i64(const void* a, const void* b)
{
    int64_t x = *(const int64_t*)a, y = *(const int64_t*)b;
    return (x > y) - (x < y);
}

int orc_goodput(const orc_sim_cfg* cfg, int64_t n, const int64_t* arr, const int32_t* o, const uint8_t* cls,
                const int64_t* t_first, const int64_t* t_done, int64_t* met_out, int64_t* p99_out)
{
    *met_out = 0;
    *p99_out = -1;
    if (n <= 0) return ORC_OK;
    int64_t* ttft = (int64_t*)malloc((size_t)n * 8);
    if (!ttft) return ORC_ENOMEM;
    int64_t met = 0;
    for (int64_t k = 0; k < n; ++k) {
        int64_t c = cls[k] < cfg->n_classes ? cls[k] : cfg->n_classes - 1;
        ttft[k] = t_first[k] - arr[k];
        int ok_ttft = ttft[k] <= cfg->ttft[c];
        int ok_tpot = o[k] == 1 || (t_done[k] - t_first[k]) <= cfg->tpot[c] * ((int64_t)o[k] - 1);
        met += ok_ttft && ok_tpot;
    }
    qsort(ttft, (size_t)n, 8, cmp_i64);
    *met_out = met;
    *p99_out = ttft[(99 * n + 99) / 100 - 1];
    free(ttft);
    return ORC_OK;
}

/* ======================================================================
 * P99 TPOT of one row (Table 2's third column; sec. IV-B names TPOT targets).
 * [reading] A request's time per output token counts the tokens after its
 * first: TPOT = floor((t_done - t_first) / (o - 1)) us for o >= 2; a request of
 * one output token has none.  The row's P99 is the nearest rank, sorted index
 * ceil(0.99 M) - 1, over its M requests with o >= 2; M = 0 gives -1.
 * ==================================================================== */
int orc_p99_tpot(int64_t n, const int32_t* o, const int64_t* t_first, const int64_t* t_done, int64_t* p99_out)
{
    *p99_out = -1;
    if (n <= 0) return ORC_OK;
    int64_t* tpot = (int64_t*)malloc((size_t)n * 8);
    if (!tpot) return ORC_ENOMEM;
    int64_t m = 0;
    for (int64_t k = 0; k < n; ++k) {
        if (o[k] >= 2) tpot[m++] = (t_done[k] - t_first[k]) / ((int64_t)o[k] - 1);
    }
    if (m > 0) {
        qsort(tpot, (size_t)m, 8, cmp_i64);
        *p99_out = tpot[(99 * m + 99) / 100 - 1];
    }
    free(tpot);
    return ORC_OK;
}

/* ======================================================================
 * Standalone batch scorer: the cost(d) display of sec. III-A for a mixed
 * per-instance state (queued prefill tokens Q, active decode sequences A,
 * KV occupancy kappa), in fp64 over the same fp32 inputs, by brute force:
 *   press = kappa_d + (p + oh) / C
 *   cost  = sigma_s * (w_b * (tau_pre Q_d + tau_act A_d)
 *                      + w_s * (tau_pre0 + tau_pre p + tau_dec oh (1 + rho press)))
 *           + w_q * A_d
 * consts = [w_b, w_s, w_q, rho, tau_pre0, tau_pre, tau_dec, tau_act, 1/C,
 *           sigma_0, sigma_1, sigma_2, sigma_3]; a class >= 4 yields index -1
 * and cost NaN.  Ties go to the lowest index.  [reading: the paper prices a
 * pure decode pool; this mixed state is the spec's standalone workload.]
 * ==================================================================== */
static double score_one(const float* c, double p, double oh, int64_t s, double Q, double A, double kap)
{
    double w_b = c[0], w_s = c[1], w_q = c[2], rho = c[3], tau_pre0 = c[4], tau_pre = c[5], tau_dec = c[6];
    double tau_act = c[7], inv_cap = c[8], sigma = c[9 + s];
    double press = kap + (p + oh) * inv_cap;
    double backlog = tau_pre * Q + tau_act * A;
    double own = tau_pre0 + tau_pre * p + tau_dec * oh * (1.0 + rho * press);
    return sigma * (w_b * backlog + w_s * own) + w_q * A;
}

void orc_score_batch(const float* p, const float* oh, const uint8_t* cls, int64_t n, const float* Q,
                     const float* A, const float* kap, int64_t n_inst, const float* consts, int32_t* argmin,
                     double* best, double* second)
{
    for (int64_t r = 0; r < n; ++r) {
        if (cls[r] >= 4) {
            argmin[r] = -1;
            best[r] = NAN;
            second[r] = NAN;
            continue;
        }
        double b1 = INFINITY, b2 = INFINITY;
        int64_t i1 = -1;
        for (int64_t d = 0; d < n_inst; ++d) {
            double v = score_one(consts, p[r], oh[r], cls[r], Q[d], A[d], kap[d]);
            if (v < b1) {
                b2 = b1;
                b1 = v;
                i1 = d;
            } else if (v < b2) {
                b2 = v;
            }
        }
        argmin[r] = (int32_t)i1;
        best[r] = b1;
        second[r] = b2;
    }
}

/* fp64 cost of chosen (request, instance) pairs */
void orc_score_pairs(const float* p, const float* oh, const uint8_t* cls, const int64_t* req_idx,
                     const int64_t* inst_idx, int64_t m, const float* Q, const float* A, const float* kap,
                     const float* consts, double* out)
{
    for (int64_t i = 0; i < m; ++i) {
        int64_t r = req_idx[i], d = inst_idx[i];
        out[i] = cls[r] >= 4 ? NAN : score_one(consts, p[r], oh[r], cls[r], Q[d], A[d], kap[d]);
    }
}
