/*
 * ctr.h -- C ABI of the GB300 marginal-cost routing simulator
 * ("Calibrate, Then Route", arXiv 2609.16206).
 *
 * Exported by paper_2609_16206_gb300/libctr.so (CUDA, sm_103a).  Conventions
 * for every entry point:
 *   - Return 0 (CTR_OK) or a negative CTR_E* code.  Arguments are validated on
 *     the host before any launch; a rejected call launches nothing.
 *   - Arrays are DEVICE pointers owned by the caller unless marked "host".
 *     The library allocates nothing and keeps no state between calls, so calls
 *     on different streams are independent and thread-safe (the one exception,
 *     ctr_simulate_noalloc, documents its shared scratch array).
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued asynchronously; nothing synchronises unless
 *     stated.  Launch failures are reported as CTR_ECUDA.
 *   - All simulated times are int64 microseconds.
 */
#ifndef CTR_H
#define CTR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define CTR_OK 0
#define CTR_EINVAL (-1)    /* bad argument, enum, bound or request data */
#define CTR_ECUDA (-2)     /* CUDA launch / driver error */
#define CTR_EOVERFLOW (-3) /* a fixed-capacity structure filled up, or a time reached 2^40 us */
#define CTR_ETIMEOUT (-4)  /* the per-instance decode-step budget ran out */
#define CTR_EBOUNDS (-5)   /* bounds-checked build only: an index fell outside its buffer (a library defect) */

#define CTR_MAX_INSTANCES 32      /* prefill + decode instances of one simulated cluster */
#define CTR_MAX_CLASSES 4         /* SLO classes */
#define CTR_MAX_CONST_SETS 128    /* cost-constant sets per ctr_simulate call */
#define CTR_MAX_REQUESTS (1 << 23) /* requests per replica */
#define CTR_MAX_STEPS_PER_INSTANCE ((1LL << 31) - (1LL << 21)) /* bound on the decode-step budget */
#define CTR_SCORE_N_CONST 13      /* length of the standalone scorer's constant vector */
#define CTR_SCORE_MAX_INST 256    /* instances per standalone scoring call */
#define CTR_SCORE_MAX_REQ (1LL << 40) /* requests per standalone scoring call */

enum ctr_policy {
    CTR_POLICY_LEARNED = 0,          /* marginal-cost argmin, sec. III-A / Algorithm 1 */
    CTR_POLICY_ROUND_ROBIN = 1,      /* request k -> instance k mod N, sec. IV-C */
    CTR_POLICY_LEAST_LOADED = 2,     /* argmin of in-flight count (JSQ), sec. IV-C */
    CTR_POLICY_LENGTH_HEURISTIC = 3, /* predicted-length threshold heuristic, sec. IV-C */
    CTR_POLICY_LEARNED_P2 = 4        /* marginal cost over two sampled candidates per pool, sec. V-D / VI */
};

/* Feature ablation (sec. V-F): bits of ctr_cost_consts.ablate.  A removed
 * feature takes its neutral value in the learned cost. */
#define CTR_ABLATE_PREDICTED_LENGTH 1u /* o_hat := 0 (no own decode work, pressure without it) */
#define CTR_ABLATE_PRESSURE 2u         /* P := 0 */
#define CTR_ABLATE_SLO 4u              /* sigma := 1.0 (256) for every class */

/* Where the learned router's backlog signal comes from (ctr_cost_consts.backlog_signal). */
#define CTR_BACKLOG_TRUE 0u  /* the cluster's true remaining work (the simulator's own clock) */
#define CTR_BACKLOG_PROXY 1u /* the deployed proxy's in-flight ledger priced with the router's constants */

enum ctr_workspace_kind { CTR_WS_SIMULATE = 0 };

/* A batch of requests in structure-of-arrays form: element [r * n_req + k] is
 * request k (0-based arrival index) of replica r.  Device memory, caller-owned.
 * The request features are the four admission-time signals of sec. III-A:
 * exact prompt length p, predicted output length o_hat, SLO class, plus the
 * true output length o (known to the simulated cluster only) and the arrival. */
typedef struct ctr_requests {
    int64_t* arrival_us; /* non-decreasing within a replica, < 2^39 */
    int32_t* prompt_len; /* p, 0..2^20 */
    int32_t* true_out;   /* o, 1..2^20, p + o <= kv_cap_tokens */
    int32_t* pred_out;   /* o_hat, 0..2^17 */
    uint8_t* slo_class;  /* 0..n_classes-1 */
} ctr_requests;

/* Synthetic trace law (a host struct).  Replica g (global index) draws from the
 * Philox4x32-10 key seed + (g mod n_seeds), sub-stream g / n_seeds; counter
 * (k, sub, stream, group).  Lengths are rounded lognormals, o_hat = o * exp(N(0,
 * noise_sigma)) rounded, class from cumulative 32-bit thresholds, arrivals the
 * integer Poisson (arrival_kind 0) or two-state MMPP (1, low state first)
 * construction.  All doubles must be finite. */
typedef struct ctr_trace_cfg {
    uint64_t seed;
    int32_t n_seeds;          /* >= 1 */
    int32_t arrival_kind;     /* 0 Poisson at rate_mreq[0]; 1 MMPP rate_mreq[0] / [1] */
    int64_t rate_mreq[2];     /* milli-requests per second, 1..10^7 */
    int64_t dwell_mean_us;    /* MMPP mean state dwell, 1..10^10 */
    double prompt_mu, prompt_sigma;   /* ln-space mean / sd of the prompt length */
    int32_t prompt_min, prompt_max;   /* clip range, 0 <= min <= max <= 2^20 */
    uint64_t mix_short_thr;           /* P(short output component) * 2^32, <= 2^32 */
    double short_mu, short_sigma, long_mu, long_sigma;
    int32_t out_min, out_max;         /* 1 <= min <= max <= 2^20 */
    double noise_sigma;               /* predictor noise, >= 0 */
    int32_t pred_min, pred_max;       /* 0 <= min <= max <= 2^17 */
    int32_t n_classes;                /* 1..4 */
    int32_t reserved0;
    uint64_t class_thr[3];            /* cumulative class probabilities * 2^32, non-decreasing */
} ctr_trace_cfg;

/* Simulated cluster (a host struct): explicit prefill and decode pools, KV
 * transfer, continuous decode batching with KV reservation, SLO classes, and
 * the capacities of the per-instance structures the GPU keeps.
 * Prefill is serial FCFS per instance (prefill_batch_tokens = 0) or batched
 * (sec. VI implements continuous batching in both stages): an instance runs
 * one batch at a time, taking FCFS the head of its queue and then every next
 * request while the batch's prompt tokens stay <= prefill_batch_tokens; a
 * batch lasts pre_base + pre_per_tok * (its prompt tokens), every member's KV
 * transfer starts at its end, and a batch starts when the previous one ends
 * (before arrivals at that instant are routed) or when a request reaches an
 * idle instance.  The learned router's true prefill backlog is then the rest
 * of the running batch plus the queue cut into batches by the same rule. */
typedef struct ctr_sim_cfg {
    int32_t n_prefill, n_decode;      /* >= 1 each, n_prefill + n_decode <= 32 */
    int64_t kv_cap_tokens;            /* C per decode instance, 1..2^31-1 */
    int64_t pre_base_us;              /* prefill = base + per_tok * p; base 1..2^30 */
    int64_t pre_us_per_tok;           /* 0..2^20 */
    int64_t xfer_us_per_tok;          /* KV transfer delay = per_tok * p; 0..2^20 */
    int64_t dec_base_us;              /* decode step = base + per_seq * n + floor(KV / kv_div); base 1..2^24 */
    int64_t dec_us_per_seq;           /* 0..2^16 */
    int64_t dec_kv_tokens_per_us;     /* kv_div, 1..2^31 */
    int32_t n_classes;                /* 1..4 */
    int32_t heuristic_threshold_tokens; /* length heuristic: o_hat >= threshold uses predicted-token load */
    int64_t ttft_slo_us[4];           /* per class, >= 0 */
    int64_t tpot_slo_us[4];
    int64_t max_steps_per_instance;   /* decode-step budget per instance and row, 1..CTR_MAX_STEPS_PER_INSTANCE */
    int32_t cap_pending;              /* requests routed to a decode instance whose KV is not ready, 1..2^20 */
    int32_t cap_waiting;              /* KV-ready requests not yet admitted, 1..2^20 */
    int32_t cap_active;               /* decode batch size, 1..2^20 */
    int32_t cap_prefill_ring;         /* requests in flight on a prefill instance, 1..2^20 */
    int64_t prefill_batch_tokens;     /* 0: serial FCFS prefill; 1..2^30: batched prefill (below) */
} ctr_sim_cfg;

/* Fixed-point constants of the learned router (a host struct).  Weights carry
 * 8 fractional bits (256 = 1.0).  Decode cost, in us * 2^16:
 *   P     = min(2^18, floor((KV_res + p + o_hat) * 2^16 / C))     post-admission pressure
 *   own   = o_hat * tau_dec
 *   T2    = own + floor(floor(own * P / 2^16) * rho / 2^8)
 *   cost  = (w_b * min(B_d, 2^40) + w_s * T2) * sigma[class] + w_q * queue * 2^16
 * Prefill cost: (w_b * B_p + w_s * (tau_pre0 + p * tau_pre)) * sigma[class] + w_q * queue * 2^16,
 * with backlog B_p = max(0, busy_until - t) and B_d = floor(R_d * step_d / max(1, n_d)).
 * CTR_POLICY_LEARNED_P2 prices only two candidates per pool: Philox4x32-10
 * with key (0x243F6A88, 0x85A308D3) and counter (k, t lo, t hi, 0x5032) gives
 * u0..u3; a pool of n offers c0 = floor(u n / 2^32) and
 * c1 = (c0 + 1 + floor(u' (n - 1) / 2^32)) mod n (decode (u0, u1), prefill
 * (u2, u3)), and the cheaper one wins (ties to the lower index).
 * Signals as the deployed proxy sees them (sec. IV-A; sec. VI explains why
 * they matter for calibration):
 *   backlog_signal = CTR_BACKLOG_PROXY replaces B_p and B_d by the in-flight
 *     ledger, each request priced once when routed and dropped when it leaves:
 *     B_p = min(2^40, sum over requests whose prefill on p has not ended of
 *     tau_pre0 + tau_pre * p), B_d = min(2^40, tau_dec * sum of o_hat over
 *     requests routed to d and not completed) (0 when o_hat is ablated).
 *   occupancy_poll_us = D > 0 makes P use the resident KV of d as it was at
 *     the last poll instant floor(t / D) * D (after every event at that
 *     instant) instead of its live value; 0 = live. */
typedef struct ctr_cost_consts {
    int64_t tau_pre0_us, tau_pre_us, tau_dec_us; /* 0..2^20 */
    int64_t w_q_us;                              /* 0..2^20, us per in-flight request */
    int32_t w_b_q8, w_s_q8, rho_q8;              /* 0..1023 */
    int32_t sigma_q8[4];                         /* 0..1023 */
    uint32_t ablate;                             /* CTR_ABLATE_* bits, 0 = every feature */
    uint32_t backlog_signal;                     /* CTR_BACKLOG_TRUE or CTR_BACKLOG_PROXY */
    int64_t occupancy_poll_us;                   /* 0..2^39; 0 = live occupancy */
} ctr_cost_consts;

/* ctr_gen_trace -- synthetic request trace (Table 1 length profiles as
 * lognormal laws; the sec. III-C predictor with sec. V-G injected noise;
 * bursty arrivals).  Fills out[r * n_req + k] for replicas
 * g = replica_offset + r, r < n_replicas.  The result is bit-identical to the
 * CPU reference construction: the variates are computed in fp32 (the trace
 * is defined in fp32, each step correctly rounded in a fixed order, with the
 * log / exp / normal-quantile functions written out from named methods and
 * the distribution parameters rounded once from the caller's doubles), and
 * arrivals are integer prefix sums.
 * n_req 0..CTR_MAX_REQUESTS; n_replicas >= 0; replica_offset >= 0. */
int ctr_gen_trace(const ctr_trace_cfg* cfg /* host */, int32_t n_replicas, int64_t replica_offset,
                  int64_t n_req, ctr_requests out, void* stream);

/* ctr_score_batch -- standalone marginal-cost scorer (sec. III-A display) of
 * every request x instance pair over a mixed per-instance state: queued
 * prefill tokens Q, active decode sequences A, KV occupancy kappa.
 *   cost(r,d) = sigma_s * (w_b * (tau_pre Q_d + tau_act A_d)
 *               + w_s * (tau_pre0 + tau_pre p + tau_dec o_hat (1 + rho (kappa_d + (p + o_hat) / C))))
 *               + w_q A_d
 * consts (host, CTR_SCORE_N_CONST floats, finite, >= 0):
 *   [w_b, w_s, w_q, rho, tau_pre0, tau_pre, tau_dec, tau_act, 1/C, sigma_0..sigma_3].
 * Per request r: out_argmin[r] = argmin_d (ties -> lowest d) and out_cost[r]
 * its fp32 cost; a slo_class >= 4 gives -1 and NaN.  Inputs must be finite and
 * non-negative.  0 <= n_req <= CTR_SCORE_MAX_REQ, 1 <= n_inst <= CTR_SCORE_MAX_INST.  status is an
 * optional device int32 (NULL ok) set to CTR_ETIMEOUT if the shared-memory
 * staging wait of a block ran past its bound (never expected); that block then
 * scores nothing, so out_argmin and out_cost are unspecified for the call.
 * The kernel is launched as a programmatic dependent launch: it reads nothing
 * before the preceding work in the stream has completed, and it lets a
 * following kernel launched the same way be scheduled while it drains (such a
 * kernel must wait for its grid dependencies before reading this call's
 * outputs, as kernels launched that way do). */
int ctr_score_batch(const float* prompt_len, const float* pred_out, const uint8_t* slo_class, int64_t n_req,
                    const float* q_tokens, const float* n_active, const float* kv_occ, int32_t n_inst,
                    const float* consts /* host */, int32_t* out_argmin, float* out_cost, int32_t* status,
                    void* stream);

/* ctr_score_stream_probe -- a measurement aid, not a step of the method (the
 * paper has no counterpart): the memory traffic of ctr_score_batch without its
 * arithmetic, on the same grid with the same loads and stores, writing
 * out_argmin[r] = slo_class[r] and out_cost[r] = prompt_len[r] + pred_out[r].
 * Timed beside the scorer it gives the HBM throughput a kernel of this shape
 * reaches at that size.  n_req a multiple of 4, at most CTR_SCORE_MAX_REQ; float arrays 16-byte aligned,
 * slo_class 4-byte aligned (CTR_EINVAL otherwise). */
int ctr_score_stream_probe(const float* prompt_len, const float* pred_out, const uint8_t* slo_class, int64_t n_req,
                           int32_t* out_argmin, float* out_cost, void* stream);

/* ctr_workspace_bytes -- device workspace ctr_simulate needs to run its
 * widest grid for these sizes on the current device (0 on bad arguments).
 * A smaller workspace is accepted and runs fewer concurrent rows. */
size_t ctr_workspace_bytes(int32_t which, const ctr_sim_cfg* cfg /* host */, int64_t n_rows, int64_t n_req);

/* ctr_simulate -- batched discrete-event simulation of the routing policies
 * (Algorithm 1 inside the sec. III-D simulator with sec. VI batching).
 * Rows are (replica, const set, policy), row-major:
 *   row = (replica * n_const_sets + set) * n_policies + policy_index.
 * Replica r reads trace[r * n_req + k]; outputs are [row * n_req + k].
 * consts: n_const_sets host structs (1..CTR_MAX_CONST_SETS); policy_ids:
 * n_policies host ints (1..5 of them), values of enum ctr_policy.
 * Outputs: i_pre / i_dec (optional, NULL ok) chosen prefill / decode instance;
 * t_first_us (end of the first decode step) and t_done_us (required);
 * row_hash the order-independent 64-bit checksum of each row's routing and
 * times; row_status CTR_OK or the row's CTR_EINVAL / CTR_EOVERFLOW /
 * CTR_ETIMEOUT (outputs of a failed row are unspecified).
 * met_count / p99_ttft_us: optional (both or neither, else CTR_EINVAL): each
 * row's SLO goodput inputs exactly as ctr_goodput defines them, computed in
 * the same pass over t_first_us / t_done_us that completes row_hash (the
 * outputs are then read once, not twice).
 * workspace: device, >= 256 bytes, ideally ctr_workspace_bytes(); its contents
 * need no initialisation and are clobbered. */
int ctr_simulate(const ctr_sim_cfg* cfg /* host */, const ctr_cost_consts* consts /* host */, int32_t n_const_sets,
                 const int32_t* policy_ids /* host */, int32_t n_policies, ctr_requests trace, int32_t n_replicas,
                 int64_t n_req, uint8_t* i_pre, uint8_t* i_dec, int64_t* t_first_us, int64_t* t_done_us,
                 uint64_t* row_hash, int32_t* row_status, int64_t* met_count, int64_t* p99_ttft_us, void* workspace,
                 size_t workspace_bytes, void* stream);

/* ctr_simulate_noalloc -- ctr_simulate for callers that cannot allocate
 * device memory (the paper has no counterpart: this is a deployment aid).
 * Some callers run where a device allocation is not theirs to make -- a
 * plugin inside a serving process whose memory pool owns the GPU, code
 * between someone else's stream-capture calls, a loop that must never reach
 * the driver's allocator.  This entry point takes the simulator's scratch
 * from a fixed array of CTR_NOALLOC_SCRATCH_BYTES that the library keeps on
 * every GPU it is loaded on until the process exits; the caller still owns
 * and passes the trace and every output, exactly as for ctr_simulate, and the
 * results are identical.  The first call on a device looks the array up (once
 * per device); make it before any stream capture.  All calls share the array:
 * calls that overlap on the GPU (two streams, two threads) race and must be
 * serialised.  A configuration whose per-warp structures (the cap_* fields)
 * do not fit the array returns CTR_EINVAL; otherwise fewer rows run at once
 * than with a full workspace.  Allocates nothing. */
#define CTR_NOALLOC_SCRATCH_BYTES ((size_t)64 << 20)
int ctr_simulate_noalloc(const ctr_sim_cfg* cfg /* host */, const ctr_cost_consts* consts /* host */,
                         int32_t n_const_sets, const int32_t* policy_ids /* host */, int32_t n_policies,
                         ctr_requests trace, int32_t n_replicas, int64_t n_req, uint8_t* i_pre, uint8_t* i_dec,
                         int64_t* t_first_us, int64_t* t_done_us, uint64_t* row_hash, int32_t* row_status,
                         void* stream);

/* ctr_goodput -- SLO goodput inputs per row (sec. IV-B targets, Table 2
 * columns): met_count[row] = #{k : TTFT <= TTFT_c and (o == 1 or
 * t_done - t_first <= TPOT_c (o - 1))} and p99_ttft_us[row] = the nearest-rank
 * P99 (sorted index ceil(0.99 n) - 1; -1 when n_req == 0).  Row r uses replica
 * r / rows_per_replica of the trace.  A class >= n_classes counts as the last
 * class.
 * p99_tpot_us: optional (NULL: not computed).  Table 2's P99 TPOT: over the
 * row's M requests with o >= 2, each one's (t_done - t_first) / (o - 1)
 * rounded toward zero, the nearest-rank P99 (sorted index ceil(0.99 M) - 1;
 * -1 when M == 0), computed in a pass of its own after the goodput pass. */
int ctr_goodput(const ctr_sim_cfg* cfg /* host */, ctr_requests trace, int32_t n_replicas, int32_t rows_per_replica,
                int64_t n_req, const int64_t* t_first_us, const int64_t* t_done_us, int64_t* met_count,
                int64_t* p99_ttft_us, int64_t* p99_tpot_us, void* stream);

/* ctr_strerror -- static description of a CTR_* code. */
const char* ctr_strerror(int code);

/* ctr_abi_version -- increments on any change to the structs, the signatures or
 * the accepted ranges. */
int ctr_abi_version(void);

/* ctr_bounds_checked -- 1 in libctr_checked.so, 0 in libctr.so.  Both export
 * the same entry points with the same results.  The checked build compiles the
 * simulator's event loop and the goodput pass with a bounds check on every
 * index into the workspace, the trace, the outputs and goodput's shared-memory
 * tables: an index outside its buffer skips the access (a load reads 0) and the
 * row reports CTR_EBOUNDS -- in row_status from the simulator, in both met_count
 * and p99_ttft_us from the goodput pass -- with no fault and no trap.  With
 * valid arguments that value never occurs; the checked build exists to show it
 * on the GPU, where no memory checker runs.  It is slower and not meant for
 * production. */
int ctr_bounds_checked(void);

#ifdef __cplusplus
}
#endif

#endif /* CTR_H */
