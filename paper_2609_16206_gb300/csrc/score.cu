// score.cu -- standalone request x instance scorer (ctr_score_batch).
//
// The sec. III-A cost of request r on instance d splits into a part shared by
// every instance and a part that depends on d:
//   cost(r,d) = sigma_s * const_r + [sigma_s * w_b * backlog_d + w_q * A_d]
//               + (sigma_s * w_s * tau_dec * rho * kappa_d) * o_hat_r
// so for a fixed class s the argmin over d is the lower envelope of the lines
// a_d^s + m_d^s * o_hat with a_d^s = sigma_s w_b backlog_d + w_q A_d and
// m_d^s = sigma_s w_s tau_dec rho kappa_d >= 0.  Each block stages the
// instance state into shared memory with a TMA bulk copy (cp.async.bulk +
// mbarrier) while its first request vectors are already in flight, builds the
// four per-class envelopes (one thread per (class, line): a division-free
// Pareto test -- a line with both a larger intercept and a larger slope than
// another can never win -- then, for the few surviving lines, the interval of
// o_hat on which the line wins and its rank), and streams requests with
// 128-bit loads, software-pipelined one vector ahead: a binary search over the
// envelope's breakpoints gives the argmin, whose fp32 cost is then evaluated
// from the full formula.  The work per request is O(log envelope size) instead
// of O(instances), which keeps the kernel on the HBM roofline.  One block per
// SM, so the envelope is built 152 times, not once per request tile.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

constexpr int kThreads = 1024;
constexpr int kMaxInst = CTR_SCORE_MAX_INST;
constexpr unsigned kWaitLimit = 1u << 22;  // bounded mbarrier polling

struct __align__(16) Smem {
    float q[kMaxInst];
    float a[kMaxInst];
    float kap[kMaxInst];
    float bk[kMaxInst];   // w_b * (tau_pre Q + tau_act A)
    float wqa[kMaxInst];  // w_q * A
    float la[4][kMaxInst];   // line intercept per class
    float lm[4][kMaxInst];   // line slope (per unit o_hat) per class
    float lo_tmp[4][kMaxInst];
    int valid_tmp[4][kMaxInst];
    int pareto[4][kMaxInst];
    float seg_lo[4][kMaxInst];
    int seg_id[4][kMaxInst];
    int nseg[4];
    unsigned long long bar;
};

__device__ __forceinline__ uint32_t smem_addr(const void* p)
{
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ float4 ld_stream(const float4* p)
{
    float4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.f32 {%0,%1,%2,%3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ uint32_t ld_stream_u32(const uint32_t* p)
{
    uint32_t v;
    asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(v) : "l"(p));
    return v;
}

// the d-dependent line of class s at instance d
__device__ __forceinline__ void line_of(const Smem& sm, const ScoreParams& P, int s, int d, float& a, float& m)
{
    const float sig = P.c[9 + s];
    a = fmaf(sig, sm.bk[d], sm.wqa[d]);
    m = sig * P.c[1] * P.c[6] * P.c[3] * sm.kap[d];
}

__device__ __forceinline__ float cost_of(const Smem& sm, const ScoreParams& P, float p, float oh, int s, int d)
{
    const float x2 = fmaf(p + oh, P.c[8], sm.kap[d]);       // post-admission pressure
    const float x3 = fmaf(P.c[3], x2, 1.0f);                // 1 + rho * press
    const float own = fmaf(P.c[6] * oh, x3, fmaf(P.c[5], p, P.c[4]));
    const float y = fmaf(P.c[1], own, sm.bk[d]);
    return fmaf(P.c[9 + s], y, sm.wqa[d]);
}

__device__ __forceinline__ void score_one(const Smem& sm, const ScoreParams& P, float p, float oh, uint32_t s,
                                          int& arg, float& cost)
{
    if (s >= 4) {
        arg = -1;
        cost = __int_as_float(0x7fc00000);
        return;
    }
    const int ns = sm.nseg[s];
    int lo = 0;
    int span = ns;
    while (span > 1) {  // last segment whose left end is <= o_hat
        const int half = span >> 1;
        if (sm.seg_lo[s][lo + half] <= oh) lo += half;
        span -= half;
    }
    const int d = sm.seg_id[s][lo];
    arg = d;
    cost = cost_of(sm, P, p, oh, (int)s, d);
}

template <bool kVec>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const ScoreParams P)
{
    extern __shared__ __align__(128) unsigned char smem_raw[];
    Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
    const int tid = threadIdx.x;
    const int n_inst = P.n_inst;

    // first request vector of this thread, in flight while the block builds its envelopes
    const int64_t nv = kVec ? (P.n >> 2) : 0;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    int64_t v = (int64_t)blockIdx.x * kThreads + tid;
    bool has = kVec && v < nv;
    const float4* p4 = reinterpret_cast<const float4*>(P.p);
    const float4* o4 = reinterpret_cast<const float4*>(P.oh);
    const uint32_t* c4 = reinterpret_cast<const uint32_t*>(P.cls);
    float4 pv = make_float4(0.f, 0.f, 0.f, 0.f), ov = pv;
    uint32_t cv = 0;
    if (has) {
        pv = ld_stream(p4 + v);
        ov = ld_stream(o4 + v);
        cv = ld_stream_u32(c4 + v);
    }

    // ---- stage the instance state: TMA bulk copy when aligned, else plain loads
    const uint32_t bytes = (uint32_t)n_inst * 4u;
    const bool bulk = kVec && (bytes % 16u == 0) && (((uintptr_t)P.Q | (uintptr_t)P.A | (uintptr_t)P.kap) % 16u == 0);
    if (bulk) {
        const uint32_t bar = smem_addr(&sm.bar);
        if (tid == 0) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
        if (tid == 0) {
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(3u * bytes)
                         : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             smem_addr(sm.q)),
                         "l"(P.Q), "r"(bytes), "r"(bar)
                         : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             smem_addr(sm.a)),
                         "l"(P.A), "r"(bytes), "r"(bar)
                         : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             smem_addr(sm.kap)),
                         "l"(P.kap), "r"(bytes), "r"(bar)
                         : "memory");
        }
        uint32_t done = 0;
        for (unsigned it = 0; it < kWaitLimit && !done; ++it) {
            asm volatile(
                "{\n\t.reg .pred p;\n\t"
                "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n\t"
                "selp.u32 %0, 1, 0, p;\n\t}"
                : "=r"(done)
                : "r"(bar)
                : "memory");
        }
        if (__syncthreads_or(!done)) {  // block-uniform decision
            // never expected: report it and read the state with plain loads instead
            if (tid == 0 && P.status) atomicExch(P.status, CTR_ETIMEOUT);
            for (int d = tid; d < n_inst; d += kThreads) {
                sm.q[d] = P.Q[d];
                sm.a[d] = P.A[d];
                sm.kap[d] = P.kap[d];
            }
        }
    } else {
        for (int d = tid; d < n_inst; d += kThreads) {
            sm.q[d] = P.Q[d];
            sm.a[d] = P.A[d];
            sm.kap[d] = P.kap[d];
        }
    }
    __syncthreads();
    for (int d = tid; d < n_inst; d += kThreads) {
        sm.bk[d] = P.c[0] * fmaf(P.c[5], sm.q[d], P.c[7] * sm.a[d]);
        sm.wqa[d] = P.c[2] * sm.a[d];
    }
    __syncthreads();

    // ---- per-class lower envelope
    for (int idx = tid; idx < 4 * n_inst; idx += kThreads) {
        const int s = idx / n_inst, d = idx - s * n_inst;
        line_of(sm, P, s, d, sm.la[s][d], sm.lm[s][d]);
    }
    __syncthreads();
    for (int idx = tid; idx < 4 * n_inst; idx += kThreads) {  // Pareto filter (ties: lowest index survives)
        const int s = idx / n_inst, d = idx - s * n_inst;
        const float ad = sm.la[s][d], md = sm.lm[s][d];
        bool dominated = false;
        for (int e = 0; e < n_inst; ++e) {
            const float ae = sm.la[s][e], me = sm.lm[s][e];
            dominated |= ae <= ad && me <= md && (ae < ad || me < md || e < d);
        }
        sm.pareto[s][d] = !dominated;
    }
    __syncthreads();
    for (int idx = tid; idx < 4 * n_inst; idx += kThreads) {  // winning o_hat interval of each surviving line
        const int s = idx / n_inst, d = idx - s * n_inst;
        bool valid = false;
        float lo = 0.0f;
        if (sm.pareto[s][d]) {
            const float ad = sm.la[s][d], md = sm.lm[s][d];
            float hi = __int_as_float(0x7f800000);
            for (int e = 0; e < n_inst; ++e) {
                if (e == d || !sm.pareto[s][e]) continue;
                const float ae = sm.la[s][e], me = sm.lm[s][e];
                if (me > md) {
                    lo = fmaxf(lo, (ad - ae) / (me - md));
                } else if (me < md) {
                    hi = fminf(hi, (ae - ad) / (md - me));
                }
            }
            valid = lo < hi;
        }
        sm.valid_tmp[s][d] = valid;
        sm.lo_tmp[s][d] = lo;
    }
    if (tid < 4) sm.nseg[tid] = 0;
    __syncthreads();
    for (int idx = tid; idx < 4 * n_inst; idx += kThreads) {
        const int s = idx / n_inst, d = idx - s * n_inst;
        if (!sm.valid_tmp[s][d]) continue;
        const float lo = sm.lo_tmp[s][d];
        int rank = 0;
        for (int e = 0; e < n_inst; ++e)
            rank += sm.valid_tmp[s][e] && (sm.lo_tmp[s][e] < lo || (sm.lo_tmp[s][e] == lo && e < d));
        sm.seg_lo[s][rank] = lo;
        sm.seg_id[s][rank] = d;
        atomicAdd(&sm.nseg[s], 1);
    }
    __syncthreads();
    if (tid < 4 && sm.nseg[tid] == 0) {  // rounding left no winner (never with finite inputs): brute force line
        int best = 0;
        float bv = 0.0f;
        for (int d = 0; d < n_inst; ++d) {
            float a, m;
            line_of(sm, P, tid, d, a, m);
            if (d == 0 || a < bv) {
                bv = a;
                best = d;
            }
        }
        sm.seg_lo[tid][0] = 0.0f;
        sm.seg_id[tid][0] = best;
        sm.nseg[tid] = 1;
    }
    __syncthreads();

    // ---- stream the requests (the first vector was loaded before the prologue)
    if (kVec) {
        int4* a4 = reinterpret_cast<int4*>(P.argmin);
        float4* f4 = reinterpret_cast<float4*>(P.cost);
        while (has) {
            const int64_t vn = v + stride;
            const bool hn = vn < nv;
            float4 pn = make_float4(0.f, 0.f, 0.f, 0.f), on = pn;
            uint32_t cn = 0;
            if (hn) {
                pn = ld_stream(p4 + vn);
                on = ld_stream(o4 + vn);
                cn = ld_stream_u32(c4 + vn);
            }
            int4 ai;
            float4 fc;
            score_one(sm, P, pv.x, ov.x, cv & 0xFFu, ai.x, fc.x);
            score_one(sm, P, pv.y, ov.y, (cv >> 8) & 0xFFu, ai.y, fc.y);
            score_one(sm, P, pv.z, ov.z, (cv >> 16) & 0xFFu, ai.z, fc.z);
            score_one(sm, P, pv.w, ov.w, cv >> 24, ai.w, fc.w);
            __stcs(a4 + v, ai);
            __stcs(f4 + v, fc);
            v = vn;
            has = hn;
            pv = pn;
            ov = on;
            cv = cn;
        }
        if (blockIdx.x == 0 && tid < (int)(P.n & 3)) {
            const int64_t i = (nv << 2) + tid;
            int ai;
            float fc;
            score_one(sm, P, P.p[i], P.oh[i], P.cls[i], ai, fc);
            P.argmin[i] = ai;
            P.cost[i] = fc;
        }
    } else {
        for (int64_t i = (int64_t)blockIdx.x * kThreads + tid; i < P.n; i += (int64_t)gridDim.x * kThreads) {
            int ai;
            float fc;
            score_one(sm, P, P.p[i], P.oh[i], P.cls[i], ai, fc);
            P.argmin[i] = ai;
            P.cost[i] = fc;
        }
    }
}

}  // namespace

cudaError_t launch_score(const ScoreParams& p, cudaStream_t stream)
{
    if (p.n == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    const bool vec = (((uintptr_t)p.p | (uintptr_t)p.oh | (uintptr_t)p.cost | (uintptr_t)p.argmin) % 16u == 0) &&
                     ((uintptr_t)p.cls % 4u == 0);
    const int smem = (int)sizeof(Smem);
    const int64_t per_block = vec ? 4 * kThreads : kThreads;
    int64_t blocks = (p.n + per_block - 1) / per_block;
    const int64_t cap = (int64_t)sms;
    if (blocks > cap) blocks = cap;
    if (vec) {
        err = cudaFuncSetAttribute(score_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (err != cudaSuccess) return err;
        score_kernel<true><<<(unsigned)blocks, kThreads, smem, stream>>>(p);
    } else {
        err = cudaFuncSetAttribute(score_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (err != cudaSuccess) return err;
        score_kernel<false><<<(unsigned)blocks, kThreads, smem, stream>>>(p);
    }
    return cudaGetLastError();
}

}  // namespace ctr
