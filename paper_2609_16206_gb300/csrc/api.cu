// api.cu -- the extern "C" entry points of libctr.so (include/ctr.h):
// host-side validation, parameter packing and kernel launches.  Nothing here
// allocates device memory or synchronises.
#include <cmath>
#include <cstring>

#include "ctr_internal.cuh"

using namespace ctr;

namespace {

constexpr int kAbiVersion = 8;

bool in_range(int64_t v, int64_t lo, int64_t hi) { return v >= lo && v <= hi; }

bool finite_all(std::initializer_list<double> xs)
{
    for (double x : xs)
        if (!std::isfinite(x)) return false;
    return true;
}

int cuda_status(cudaError_t e) { return e == cudaSuccess ? CTR_OK : CTR_ECUDA; }

bool valid_sim_cfg(const ctr_sim_cfg* c)
{
    if (!c) return false;
    if (c->n_prefill < 1 || c->n_decode < 1 || c->n_prefill > CTR_MAX_INSTANCES || c->n_decode > CTR_MAX_INSTANCES)
        return false;
    if (c->n_prefill + c->n_decode > CTR_MAX_INSTANCES) return false;  // no overflow: each is <= 32
    if (!in_range(c->kv_cap_tokens, 1, 2147483647LL)) return false;
    if (!in_range(c->pre_base_us, 1, 1LL << 30) || !in_range(c->pre_us_per_tok, 0, 1LL << 20)) return false;
    if (!in_range(c->xfer_us_per_tok, 0, 1LL << 20)) return false;
    if (!in_range(c->dec_base_us, 1, 1LL << 24) || !in_range(c->dec_us_per_seq, 0, 1LL << 16)) return false;
    if (!in_range(c->dec_kv_tokens_per_us, 1, 1LL << 31)) return false;
    if (!in_range(c->n_classes, 1, CTR_MAX_CLASSES)) return false;
    if (c->heuristic_threshold_tokens < 0) return false;
    for (int i = 0; i < CTR_MAX_CLASSES; ++i)
        if (c->ttft_slo_us[i] < 0 || c->tpot_slo_us[i] < 0) return false;
    if (!in_range(c->max_steps_per_instance, 1, CTR_MAX_STEPS_PER_INSTANCE)) return false;
    if (!in_range(c->prefill_batch_tokens, 0, 1LL << 30)) return false;
    const int64_t cap_max = 1LL << 20;
    if (!in_range(c->cap_pending, 1, cap_max) || !in_range(c->cap_waiting, 1, cap_max) ||
        !in_range(c->cap_active, 1, cap_max) || !in_range(c->cap_prefill_ring, 1, cap_max))
        return false;
    return true;
}

bool valid_consts(const ctr_cost_consts& k)
{
    const int64_t t = 1LL << 20;
    if (!in_range(k.tau_pre0_us, 0, t) || !in_range(k.tau_pre_us, 0, t) || !in_range(k.tau_dec_us, 0, t) ||
        !in_range(k.w_q_us, 0, t))
        return false;
    if (!in_range(k.w_b_q8, 0, 1023) || !in_range(k.w_s_q8, 0, 1023) || !in_range(k.rho_q8, 0, 1023)) return false;
    for (int i = 0; i < 4; ++i)
        if (!in_range(k.sigma_q8[i], 0, 1023)) return false;
    if (k.ablate > 7u) return false;
    if (k.backlog_signal > CTR_BACKLOG_PROXY) return false;
    if (!in_range(k.occupancy_poll_us, 0, kArrivalLimit)) return false;
    return true;
}

bool requests_present(const ctr_requests& r)
{
    return r.arrival_us && r.prompt_len && r.true_out && r.pred_out && r.slo_class;
}

}  // namespace

extern "C" {

int ctr_abi_version(void) { return kAbiVersion; }

int ctr_bounds_checked(void) { return CTR_BOUNDS_CHECK; }

const char* ctr_strerror(int code)
{
    switch (code) {
    case CTR_OK: return "ok";
    case CTR_EINVAL: return "invalid argument, bound or request data";
    case CTR_ECUDA: return "CUDA launch or driver error";
    case CTR_EOVERFLOW: return "a fixed-capacity structure filled up or a time reached 2^40 us";
    case CTR_ETIMEOUT: return "decode-step budget exhausted";
    case CTR_EBOUNDS: return "an index fell outside its buffer (bounds-checked build)";
    default: return "unknown ctr status";
    }
}

int ctr_gen_trace(const ctr_trace_cfg* cfg, int32_t n_replicas, int64_t replica_offset, int64_t n_req,
                  ctr_requests out, void* stream)
{
    if (!cfg || n_replicas < 0 || replica_offset < 0 || !in_range(n_req, 0, CTR_MAX_REQUESTS)) return CTR_EINVAL;
    if (n_replicas > 0 && n_req > 0 && !requests_present(out)) return CTR_EINVAL;
    if (cfg->n_seeds < 1 || (cfg->arrival_kind != 0 && cfg->arrival_kind != 1)) return CTR_EINVAL;
    if (!in_range(cfg->rate_mreq[0], 1, 10000000) || !in_range(cfg->rate_mreq[1], 1, 10000000)) return CTR_EINVAL;
    if (!in_range(cfg->dwell_mean_us, 1000, 10000000000LL)) return CTR_EINVAL;
    if (!finite_all({cfg->prompt_mu, cfg->prompt_sigma, cfg->short_mu, cfg->short_sigma, cfg->long_mu,
                     cfg->long_sigma, cfg->noise_sigma}))
        return CTR_EINVAL;
    if (cfg->noise_sigma < 0.0 || cfg->prompt_sigma < 0.0 || cfg->short_sigma < 0.0 || cfg->long_sigma < 0.0)
        return CTR_EINVAL;
    if (!(0 <= cfg->prompt_min && cfg->prompt_min <= cfg->prompt_max && cfg->prompt_max <= (1 << 20))) return CTR_EINVAL;
    if (!(1 <= cfg->out_min && cfg->out_min <= cfg->out_max && cfg->out_max <= (1 << 20))) return CTR_EINVAL;
    if (!(0 <= cfg->pred_min && cfg->pred_min <= cfg->pred_max && cfg->pred_max <= (1 << 17))) return CTR_EINVAL;
    if (cfg->mix_short_thr > (1ull << 32)) return CTR_EINVAL;
    if (!in_range(cfg->n_classes, 1, CTR_MAX_CLASSES)) return CTR_EINVAL;
    for (int i = 0; i + 1 < cfg->n_classes; ++i) {
        if (cfg->class_thr[i] > (1ull << 32)) return CTR_EINVAL;
        if (i > 0 && cfg->class_thr[i] < cfg->class_thr[i - 1]) return CTR_EINVAL;
    }
    if (replica_offset > (1LL << 40) - (int64_t)n_replicas) return CTR_EINVAL;  // offset + count <= 2^40

    TraceParams p;
    std::memset(&p, 0, sizeof(p));
    p.seed = cfg->seed;
    p.n_seeds = cfg->n_seeds;
    p.arrival_kind = cfg->arrival_kind;
    p.n_classes = cfg->n_classes;
    p.rate[0] = cfg->rate_mreq[0];
    p.rate[1] = cfg->rate_mreq[1];
    p.rate_recip[0] = ~0ull / (uint64_t)cfg->rate_mreq[0];
    p.rate_recip[1] = ~0ull / (uint64_t)cfg->rate_mreq[1];
    p.dwell_mean_us = cfg->dwell_mean_us;
    p.dwell_mean_f = (float)cfg->dwell_mean_us;
    // the trace is defined in fp32: each parameter is rounded once from the caller's double
    p.prompt_mu = (float)cfg->prompt_mu;
    p.prompt_sigma = (float)cfg->prompt_sigma;
    p.short_mu = (float)cfg->short_mu;
    p.short_sigma = (float)cfg->short_sigma;
    p.long_mu = (float)cfg->long_mu;
    p.long_sigma = (float)cfg->long_sigma;
    p.noise_sigma = (float)cfg->noise_sigma;
    p.prompt_min = cfg->prompt_min;
    p.prompt_max = cfg->prompt_max;
    p.out_min = cfg->out_min;
    p.out_max = cfg->out_max;
    p.pred_min = cfg->pred_min;
    p.pred_max = cfg->pred_max;
    p.mix_short_thr = cfg->mix_short_thr;
    for (int i = 0; i < 3; ++i) p.class_thr[i] = cfg->class_thr[i];
    p.n_replicas = n_replicas;
    p.replica_offset = replica_offset;
    p.n_req = n_req;
    p.out = out;
    return cuda_status(launch_trace(p, (cudaStream_t)stream));
}

int ctr_score_batch(const float* prompt_len, const float* pred_out, const uint8_t* slo_class, int64_t n_req,
                    const float* q_tokens, const float* n_active, const float* kv_occ, int32_t n_inst,
                    const float* consts, int32_t* out_argmin, float* out_cost, int32_t* status, void* stream)
{
    if (n_req < 0 || n_req > CTR_SCORE_MAX_REQ || n_inst < 1 || n_inst > CTR_SCORE_MAX_INST || !consts)
        return CTR_EINVAL;
    if (!q_tokens || !n_active || !kv_occ) return CTR_EINVAL;
    if (n_req > 0 && (!prompt_len || !pred_out || !slo_class || !out_argmin || !out_cost)) return CTR_EINVAL;
    ScoreParams p;
    std::memset(&p, 0, sizeof(p));
    for (int i = 0; i < CTR_SCORE_N_CONST; ++i) {
        if (!std::isfinite(consts[i]) || consts[i] < 0.0f) return CTR_EINVAL;
        p.c[i] = consts[i];
    }
    p.p = prompt_len;
    p.oh = pred_out;
    p.cls = slo_class;
    p.n = n_req;
    p.Q = q_tokens;
    p.A = n_active;
    p.kap = kv_occ;
    p.n_inst = n_inst;
    p.argmin = out_argmin;
    p.cost = out_cost;
    p.status = status;
    return cuda_status(launch_score(p, (cudaStream_t)stream));
}

int ctr_score_stream_probe(const float* prompt_len, const float* pred_out, const uint8_t* slo_class, int64_t n_req,
                           int32_t* out_argmin, float* out_cost, void* stream)
{
    if (n_req < 0 || n_req > CTR_SCORE_MAX_REQ || n_req % 4 != 0) return CTR_EINVAL;
    if (n_req > 0 && (!prompt_len || !pred_out || !slo_class || !out_argmin || !out_cost)) return CTR_EINVAL;
    if ((((uintptr_t)prompt_len | (uintptr_t)pred_out | (uintptr_t)out_argmin | (uintptr_t)out_cost) % 16u) != 0 ||
        (uintptr_t)slo_class % 4u != 0)
        return CTR_EINVAL;
    ScoreParams p;
    std::memset(&p, 0, sizeof(p));
    p.p = prompt_len;
    p.oh = pred_out;
    p.cls = slo_class;
    p.n = n_req;
    p.argmin = out_argmin;
    p.cost = out_cost;
    return cuda_status(launch_stream_probe(p, (cudaStream_t)stream));
}

size_t ctr_workspace_bytes(int32_t which, const ctr_sim_cfg* cfg, int64_t n_rows, int64_t n_req)
{
    (void)n_req;
    if (which != CTR_WS_SIMULATE || !valid_sim_cfg(cfg) || n_rows < 0) return 0;
    int64_t off_act = 0, off_wait = 0;
    int32_t cap_pr = 0;
    const int64_t slot = sim_slot_bytes(*cfg, &off_act, &off_wait, &cap_pr);
    int wpb = 0, blocks = 0;
    const int64_t resident = sim_max_resident_warps(&wpb, &blocks);
    if (resident <= 0) return 0;
    // one slot per persistent warp, and a warp carries 32 / width rows
    const int64_t rows_per_warp = 32 / sim_group_width(cfg->n_prefill + cfg->n_decode);
    const int64_t warps = (n_rows + rows_per_warp - 1) / rows_per_warp;
    const int64_t slots = warps < resident ? (warps > 0 ? warps : 1) : resident;
    return (size_t)(256 + slots * slot);
}

int ctr_simulate(const ctr_sim_cfg* cfg, const ctr_cost_consts* consts, int32_t n_const_sets,
                 const int32_t* policy_ids, int32_t n_policies, ctr_requests trace, int32_t n_replicas, int64_t n_req,
                 uint8_t* i_pre, uint8_t* i_dec, int64_t* t_first_us, int64_t* t_done_us, uint64_t* row_hash,
                 int32_t* row_status, int64_t* met_count, int64_t* p99_ttft_us, void* workspace,
                 size_t workspace_bytes, void* stream)
{
    if (!valid_sim_cfg(cfg) || !consts || !policy_ids) return CTR_EINVAL;
    if (!in_range(n_const_sets, 1, CTR_MAX_CONST_SETS) || !in_range(n_policies, 1, 5)) return CTR_EINVAL;
    if (n_replicas < 0 || !in_range(n_req, 0, CTR_MAX_REQUESTS)) return CTR_EINVAL;
    for (int i = 0; i < n_const_sets; ++i)
        if (!valid_consts(consts[i])) return CTR_EINVAL;
    for (int i = 0; i < n_policies; ++i)
        if (!in_range(policy_ids[i], 0, 4)) return CTR_EINVAL;
    const int64_t n_rows = (int64_t)n_replicas * n_const_sets * n_policies;
    if (n_rows >= (1LL << 31)) return CTR_EINVAL;
    if (n_rows == 0) return CTR_OK;
    if (!row_hash || !row_status || !workspace) return CTR_EINVAL;
    if ((met_count == nullptr) != (p99_ttft_us == nullptr)) return CTR_EINVAL;  // both goodput outputs or neither
    if (n_req > 0 && (!requests_present(trace) || !t_first_us || !t_done_us)) return CTR_EINVAL;
    if ((uintptr_t)workspace % 256 != 0) return CTR_EINVAL;

    SimParams p;
    std::memset(&p, 0, sizeof(p));
    p.n_pre = cfg->n_prefill;
    p.n_dec = cfg->n_decode;
    p.kv_cap = cfg->kv_cap_tokens;
    p.kv_cap_recip = ~0ull / (uint64_t)cfg->kv_cap_tokens;
    p.pre_base = cfg->pre_base_us;
    p.pre_tok = cfg->pre_us_per_tok;
    p.xfer_tok = cfg->xfer_us_per_tok;
    p.dec_base = cfg->dec_base_us;
    p.dec_seq = cfg->dec_us_per_seq;
    p.kv_div = cfg->dec_kv_tokens_per_us;
    p.pre_batch = cfg->prefill_batch_tokens;
    // ceil(2^64 / kv_div) = floor((2^64 - 1) / kv_div) + 1 for kv_div >= 2 (not a power of two
    // or otherwise: the +1 rounds up whenever kv_div does not divide 2^64 exactly)
    if (p.kv_div >= 2) {
        const uint64_t d = (uint64_t)p.kv_div;
        uint64_t m = ~0ull / d;
        if ((d & (d - 1)) != 0) m += 1;                 // d does not divide 2^64
        else m = (uint64_t)1 << (64 - __builtin_ctzll(d)); // exact power of two
        p.kv_div_magic = m;
    }
    p.n_classes = cfg->n_classes;
    p.heur_thresh = cfg->heuristic_threshold_tokens;
    p.max_steps = cfg->max_steps_per_instance;
    p.cap_pend = cfg->cap_pending;
    p.cap_wait = cfg->cap_waiting;
    p.cap_act = cfg->cap_active;
    p.cap_ring = cfg->cap_prefill_ring;
    p.cap_pend_store = cfg->cap_pending + cfg->cap_waiting + 1;
    p.n_sets = n_const_sets;
    p.n_pols = n_policies;
    for (int i = 0; i < n_policies; ++i) p.pols[i] = policy_ids[i];
    p.n_req = n_req;
    p.n_rows = n_rows;
    p.trace = trace;
    p.i_pre = i_pre;
    p.i_dec = i_dec;
    p.t_first = t_first_us;
    p.t_done = t_done_us;
    p.row_hash = row_hash;
    p.row_status = row_status;
    p.trace_len = (int64_t)n_replicas * n_req;
    p.out_len = n_rows * n_req;
    for (int i = 0; i < n_const_sets; ++i) {
        const ctr_cost_consts& k = consts[i];
        ConstsDev& d = p.sets[i];
        d.tau_pre0 = k.tau_pre0_us;
        d.tau_pre = k.tau_pre_us;
        d.tau_dec = k.tau_dec_us;
        d.w_q = k.w_q_us;
        d.w_b = k.w_b_q8;
        d.w_s = k.w_s_q8;
        d.rho = k.rho_q8;
        for (int c = 0; c < 4; ++c) d.sigma[c] = k.sigma_q8[c];
        d.ablate = k.ablate;
        d.proxy = k.backlog_signal;
        d.poll_us = k.occupancy_poll_us;
        d.poll_recip = k.occupancy_poll_us > 0 ? ~0ull / (uint64_t)k.occupancy_poll_us : 0;
    }

    p.slot_bytes = sim_slot_bytes(*cfg, &p.off_act, &p.off_wait, &p.cap_pr);
    int wpb = 0, blocks_max = 0;
    const int64_t resident = sim_max_resident_warps(&wpb, &blocks_max);
    if (resident <= 0) return CTR_ECUDA;
    if (workspace_bytes < 256 + (size_t)p.slot_bytes) return CTR_EINVAL;
    int64_t slots = (int64_t)((workspace_bytes - 256) / (size_t)p.slot_bytes);
    if (slots > resident) slots = resident;
    const int64_t rows_per_warp = 32 / sim_group_width(cfg->n_prefill + cfg->n_decode);
    const int64_t warps_needed = (n_rows + rows_per_warp - 1) / rows_per_warp;
    if (slots > warps_needed) slots = warps_needed;
    p.n_slots = (int32_t)slots;
    p.ws = static_cast<unsigned char*>(workspace) + 256;
    p.next_row = static_cast<uint32_t*>(workspace);
    cudaStream_t s = (cudaStream_t)stream;
    cudaError_t e = cudaMemsetAsync(workspace, 0, 256, s);
    if (e != cudaSuccess) return CTR_ECUDA;
    const int blocks = (int)((slots + wpb - 1) / wpb);
    const bool goodput = met_count != nullptr;
    e = launch_sim(p, blocks, wpb, s);
    if (e != cudaSuccess) return cuda_status(e);
    // Once the simulation has ended its per-warp structures are dead, so the slots hold, when they have
    // room, the table of the checksum terms' request-only halves for the pass that follows.
    uint64_t* kmix = nullptr;
    if (n_rows > 0 && n_req > 0 && slots * p.slot_bytes >= 16 * n_req) {
        kmix = reinterpret_cast<uint64_t*>(p.ws);
        e = launch_mix_table(kmix, n_req, s);
        if (e != cudaSuccess) return cuda_status(e);
    }
    if (!goodput) return cuda_status(launch_hash(p, kmix, blocks, s));
    // each row's goodput, in the same pass that adds its checksum's first-token and completion terms
    GoodputParams g;
    std::memset(&g, 0, sizeof(g));
    g.trace = trace;
    g.n_req = n_req;
    g.n_rows = n_rows;
    g.rows_per_replica = n_const_sets * n_policies;
    g.n_classes = cfg->n_classes;
    for (int i = 0; i < 4; ++i) {
        g.ttft[i] = cfg->ttft_slo_us[i];
        g.tpot[i] = cfg->tpot_slo_us[i];
    }
    g.t_first = t_first_us;
    g.t_done = t_done_us;
    g.met = met_count;
    g.p99 = p99_ttft_us;
    g.row_hash = row_hash;
    g.row_status = row_status;
    g.kmix = kmix;
    return cuda_status(launch_goodput(g, s));
}

int ctr_goodput(const ctr_sim_cfg* cfg, ctr_requests trace, int32_t n_replicas, int32_t rows_per_replica, int64_t n_req,
                const int64_t* t_first_us, const int64_t* t_done_us, int64_t* met_count, int64_t* p99_ttft_us,
                int64_t* p99_tpot_us, void* stream)
{
    if (!cfg || !in_range(cfg->n_classes, 1, CTR_MAX_CLASSES)) return CTR_EINVAL;
    if (n_replicas < 0 || rows_per_replica < 1 || !in_range(n_req, 0, CTR_MAX_REQUESTS)) return CTR_EINVAL;
    const int64_t n_rows = (int64_t)n_replicas * rows_per_replica;
    if (n_rows == 0) return CTR_OK;
    if (!met_count || !p99_ttft_us) return CTR_EINVAL;
    if (n_req > 0 && (!requests_present(trace) || !t_first_us || !t_done_us)) return CTR_EINVAL;
    GoodputParams p;
    std::memset(&p, 0, sizeof(p));
    p.trace = trace;
    p.n_req = n_req;
    p.n_rows = n_rows;
    p.rows_per_replica = rows_per_replica;
    p.n_classes = cfg->n_classes;
    for (int i = 0; i < 4; ++i) {
        p.ttft[i] = cfg->ttft_slo_us[i];
        p.tpot[i] = cfg->tpot_slo_us[i];
    }
    p.t_first = t_first_us;
    p.t_done = t_done_us;
    p.met = met_count;
    p.p99 = p99_ttft_us;
    const cudaError_t e = launch_goodput(p, (cudaStream_t)stream);
    if (e != cudaSuccess || !p99_tpot_us) return cuda_status(e);
    return cuda_status(launch_tpot(p, p99_tpot_us, (cudaStream_t)stream));
}

}  // extern "C"
