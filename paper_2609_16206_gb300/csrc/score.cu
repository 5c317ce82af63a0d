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
// mbarrier) while its first request vectors are already in flight, then builds
// the four per-class envelopes: for pools of up to 64 instances one warp per
// class walks the envelope from o_hat = 0 by gift wrapping (one warp argmin
// per segment); wider pools use every thread (a Pareto test, the o_hat
// interval on which each surviving line wins, and its rank).  Each segment
// keeps its instance's cost terms, sigma_s folded in, in one 16-byte entry.
// Requests stream with 128-bit loads, software-pipelined two vectors ahead,
// each block over an equal contiguous range: the count of breakpoints at or
// below o_hat (4 or 7 compares, chosen per block from its longest envelope; a
// binary search past 8 segments) gives the argmin, whose fp32 cost is then
// evaluated from the full formula.  The work
// per request is O(log envelope size) instead of O(instances), which keeps the
// kernel on the HBM roofline.  One block per SM, so the envelope is built 152
// times, not once per request tile.
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
    // per segment: sigma w_s kappa tau_dec rho, sigma w_s, sigma BK + WQA, index (as bits); row 4 holds
    // the one entry of the invalid classes (slo_class >= 4): (0, 0, NaN, -1)
    float4 seg_e[5][kMaxInst];
    float4 brk[5][2];  // breakpoints 1..7 of each class (seg_lo[s][1..7]), +inf past the last; row 4 all +inf
    int nseg[5];
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

// The request-only part of the cost: own = G + H kappa_d with
// G = tau_pre0 + tau_pre p + o_hat (tau_dec + tau_dec rho / C (p + o_hat)) and H = tau_dec rho o_hat,
// so cost = sigma_s (BK_d + w_s (G + H kappa_d)) + WQA_d.  The constant tau_dec rho / C is
// folded once per thread (kg) and tau_dec rho into the segment entries.
__device__ __forceinline__ float req_g(const ScoreParams& P, float kg, float p, float oh)
{
    return fmaf(oh, fmaf(kg, p + oh, P.c[6]), fmaf(P.c[5], p, P.c[4]));
}

// The full cost at the segment's instance, e = (sigma_s w_s tau_dec rho kappa_d, sigma_s w_s,
// sigma_s BK_d + WQA_d, d): e.x o_hat + e.y G + e.z, every term non-negative, each path
// at most 9 roundings of 2^-24.
__device__ __forceinline__ float cost_at(float g, float oh, float4 e) { return fmaf(e.x, oh, fmaf(e.y, g, e.z)); }

// the segment entry of instance d in class s
__device__ __forceinline__ float4 seg_entry(const Smem& sm, const ScoreParams& P, int s, int d)
{
    const float A = sm.a[d];
    const float sig = P.c[9 + s];
    const float sws = sig * P.c[1];
    const float bk = P.c[0] * fmaf(P.c[5], sm.q[d], P.c[7] * A);
    return make_float4(sws * sm.kap[d] * P.c[6] * P.c[3], sws, fmaf(sig, bk, P.c[2] * A), __int_as_float(d));
}

// kB = 4 or 8: every class has at most kB + 1 segments (block-uniform), and the
// segment is the count of its padded breakpoints <= o_hat; kB = 0: binary search
// (an invalid class reads row 4: no breakpoints, one entry (0, 0, NaN, -1))
template <int kB>
__device__ __forceinline__ void score_one(const Smem& sm, const ScoreParams& P, float kg, float p, float oh,
                                          uint32_t s, int& arg, float& cost)
{
    s = s < 4u ? s : 4u;
    int seg;
    if (kB > 0) {  // segments start at 0 and at the sorted breakpoints: count those <= o_hat
        const float4 b0 = sm.brk[s][0];
        seg = (int)(b0.x <= oh) + (int)(b0.y <= oh) + (int)(b0.z <= oh) + (int)(b0.w <= oh);
        if (kB > 4) {
            const float4 b1 = sm.brk[s][1];
            seg += (int)(b1.x <= oh) + (int)(b1.y <= oh) + (int)(b1.z <= oh);
        }
    } else {
        int lo = 0, span = sm.nseg[s];
        while (span > 1) {  // last segment whose left end is <= o_hat
            const int half = span >> 1;
            if (sm.seg_lo[s][lo + half] <= oh) lo += half;
            span -= half;
        }
        seg = lo;
    }
    const float4 e = sm.seg_e[s][seg];
    arg = __float_as_int(e.w);
    cost = cost_at(req_g(P, kg, p, oh), oh, e);
}

// (intercept, slope, index) lexicographic order of envelope lines
__device__ __forceinline__ bool line_less(float a, float m, int i, float b, float n, int j)
{
    return a < b || (a == b && (m < n || (m == n && i < j)));
}

// An order-preserving 32-bit key of a float: (key(a) < key(b)) == (a < b) for
// non-NaN a, b (negative values have every bit flipped, others the sign bit set).
__device__ __forceinline__ uint32_t fkey(float x)
{
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// The warp's least (x, j) over each lane's candidate, returned to every lane as
// the winning index j (-1 when no lane has one): a redux.sync minimum on the
// key of x, then one on j among the lanes holding that x.
__device__ __forceinline__ int warp_argmin_x(bool has, float x, int j)
{
    const uint32_t kx = has ? fkey(x) : 0xffffffffu;
    const uint32_t mx = __reduce_min_sync(0xffffffffu, kx);
    const uint32_t kj = has && kx == mx ? (uint32_t)j : 0xffffffffu;
    return (int)__reduce_min_sync(0xffffffffu, kj);
}

// Lower envelope of one class's lines over o_hat >= 0 with one warp, for up to
// 64 lines (two per lane), by gift wrapping: the first segment's line has the
// least intercept; from the current line the next one is, among the lines of
// smaller slope, the one whose crossing with it comes first, and the crossing
// is that segment's left end.  Each step lowers the slope, so the loop ends
// within n_inst steps, one warp minimum each (a handful for the states seen in
// practice: the envelope of n random lines has O(log n) segments).  Ties need
// no slope rule: of two lines meeting the current one at the same point, the
// steeper one taken first meets the other there again at the next step, which
// leaves it a segment of zero length (a crossing a rounding step off leaves a
// sliver where the two costs agree to rounding).  A lane's two lines are
// compared first (least crossing, then smaller slope), then the warp takes
// the least (crossing, index) with two redux.sync reductions.  Crossings use
// the fast reciprocal divide (a few ulp, which moves a breakpoint only among
// near-equal costs).  Left ends are kept non-decreasing against
// rounding.  Segment t stays in lane t % 32, slot t / 32, until the warp writes
// the segment arrays and the padded breakpoints.
__device__ void warp_envelope(Smem& sm, const ScoreParams& P, int s, int n_inst, int lane)
{
    const float inf = __int_as_float(0x7f800000);
    const float sig = P.c[9 + s];
    const float ks = sig * P.c[1] * P.c[6] * P.c[3];
    float a[2], m[2];
    bool live[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) {  // the line of instance j (the expression line_of evaluates)
        const int j = lane + 32 * r;
        const float A = j < n_inst ? sm.a[j] : 0.0f;
        a[r] = j < n_inst ? fmaf(sig, P.c[0] * fmaf(P.c[5], sm.q[j], P.c[7] * A), P.c[2] * A) : inf;
        m[r] = j < n_inst ? ks * sm.kap[j] : inf;
        // a non-finite line (outside the input contract) takes no part, which keeps
        // every comparison below a total order and the warp's decisions uniform
        live[r] = fabsf(a[r]) < inf && fabsf(m[r]) < inf;
    }
    // the lane's least line (intercept, slope, index), then the warp's (intercept, index)
    int r0 = live[0] ? 0 : 1;
    if (live[0] && live[1] && line_less(a[1], m[1], lane + 32, a[0], m[0], lane)) r0 = 1;
    int ci = warp_argmin_x(live[0] || live[1], r0 ? a[1] : a[0], lane + 32 * r0);
    bool more = ci >= 0;
    if (!more) ci = 0;  // no finite line at all (outside the input contract): line 0
    float ca = __shfl_sync(0xffffffffu, ci >= 32 ? a[1] : a[0], ci & 31);
    float cm = __shfl_sync(0xffffffffu, ci >= 32 ? m[1] : m[0], ci & 31);
    float lo0 = 0.0f, lo1 = 0.0f;
    int id0 = ci, id1 = 0;
    float x_cur = 0.0f;
    int nseg = 1;
    while (more && nseg < n_inst) {
        // the lane's first crossing among its lines of smaller slope (x, slope, index),
        // branch-free: both crossings, then selects
        const float d0 = cm - m[0], d1 = cm - m[1];
        const float x0 = __fdividef(a[0] - ca, d0), x1 = __fdividef(a[1] - ca, d1);
        const bool c0 = live[0] && m[0] < cm && x0 == x0;
        const bool c1 = live[1] && m[1] < cm && x1 == x1;
        const bool p1 = c1 && (!c0 || x1 < x0 || (x1 == x0 && m[1] < m[0]));  // slot 0 (lower index) on full ties
        const bool has = c0 || c1;
        const float bx = p1 ? x1 : x0, bm = p1 ? m[1] : m[0], ba = p1 ? a[1] : a[0];
        const int bi = warp_argmin_x(has, bx, lane + 32 * (int)p1);  // the warp's first crossing
        if (bi < 0) break;  // warp-uniform: no line of smaller slope is left
        const int wl = bi & 31;
        ca = __shfl_sync(0xffffffffu, ba, wl);
        cm = __shfl_sync(0xffffffffu, bm, wl);
        x_cur = fmaxf(__shfl_sync(0xffffffffu, bx, wl), x_cur);
        if (lane == (nseg & 31)) {
            if (nseg < 32) {
                lo0 = x_cur;
                id0 = bi;
            } else {
                lo1 = x_cur;
                id1 = bi;
            }
        }
        ++nseg;
    }
    if (lane < nseg) {
        sm.seg_lo[s][lane] = lo0;
        sm.seg_e[s][lane] = seg_entry(sm, P, s, id0);
    }
    if (lane + 32 < nseg) {
        sm.seg_lo[s][lane + 32] = lo1;
        sm.seg_e[s][lane + 32] = seg_entry(sm, P, s, id1);
    }
    if (lane >= 1 && lane <= 8) {  // padded breakpoints for the branch-free segment count
        float* b = reinterpret_cast<float*>(&sm.brk[s][0]);
        b[lane - 1] = lane < nseg ? lo0 : inf;
    }
    if (lane == 0) sm.nseg[s] = nseg;
}

// A thread's request vectors (4 requests each): block b owns the contiguous
// range [n_vec * b / blocks, n_vec * (b + 1) / blocks), so every block streams
// the same number of vectors within one, and its threads take every
// kThreads-th vector from the block's start; the current vector and the next
// are loaded ahead of their use.
struct ReqPipe {
    int64_t v, end;
    bool has, hn;
    float4 pv, ov, pn, on;
    uint32_t cv, cn;
};

__device__ __forceinline__ void pipe_start(ReqPipe& q, const ScoreParams& P, int64_t n_vec, int tid)
{
    const float4* p4 = reinterpret_cast<const float4*>(P.p);
    const float4* o4 = reinterpret_cast<const float4*>(P.oh);
    const uint32_t* c4 = reinterpret_cast<const uint32_t*>(P.cls);
    q.v = n_vec * blockIdx.x / gridDim.x + tid;
    q.end = n_vec * (blockIdx.x + 1) / gridDim.x;
    q.pv = q.ov = q.pn = q.on = make_float4(0.f, 0.f, 0.f, 0.f);
    q.cv = q.cn = 0;
    q.has = q.v < q.end;
    if (q.has) {
        q.pv = ld_stream(p4 + q.v);
        q.ov = ld_stream(o4 + q.v);
        q.cv = ld_stream_u32(c4 + q.v);
    }
    q.hn = q.v + kThreads < q.end;
    if (q.hn) {
        q.pn = ld_stream(p4 + q.v + kThreads);
        q.on = ld_stream(o4 + q.v + kThreads);
        q.cn = ld_stream_u32(c4 + q.v + kThreads);
    }
}

// score the thread's vectors, two ahead: vector v is priced while v + kThreads
// and v + 2 kThreads load
template <int kB>
__device__ __forceinline__ void pipe_score(ReqPipe& q, const Smem& sm, const ScoreParams& P)
{
    const float4* p4 = reinterpret_cast<const float4*>(P.p);
    const float4* o4 = reinterpret_cast<const float4*>(P.oh);
    const uint32_t* c4 = reinterpret_cast<const uint32_t*>(P.cls);
    int4* a4 = reinterpret_cast<int4*>(P.argmin);
    float4* f4 = reinterpret_cast<float4*>(P.cost);
    const float kg = P.c[6] * P.c[3] * P.c[8];
    while (q.has) {
        const int64_t vf = q.v + 2 * kThreads;
        const bool hf = vf < q.end;
        float4 pf = make_float4(0.f, 0.f, 0.f, 0.f), of = pf;
        uint32_t cf = 0;
        if (hf) {
            pf = ld_stream(p4 + vf);
            of = ld_stream(o4 + vf);
            cf = ld_stream_u32(c4 + vf);
        }
        int4 ai;
        float4 fc;
        score_one<kB>(sm, P, kg, q.pv.x, q.ov.x, q.cv & 0xFFu, ai.x, fc.x);
        score_one<kB>(sm, P, kg, q.pv.y, q.ov.y, (q.cv >> 8) & 0xFFu, ai.y, fc.y);
        score_one<kB>(sm, P, kg, q.pv.z, q.ov.z, (q.cv >> 16) & 0xFFu, ai.z, fc.z);
        score_one<kB>(sm, P, kg, q.pv.w, q.ov.w, q.cv >> 24, ai.w, fc.w);
        __stcs(a4 + q.v, ai);
        __stcs(f4 + q.v, fc);
        q.v += kThreads;
        q.has = q.hn;
        q.pv = q.pn;
        q.ov = q.on;
        q.cv = q.cn;
        q.hn = hf;
        q.pn = pf;
        q.on = of;
        q.cn = cf;
    }
}

template <bool kVec>
__global__ void __launch_bounds__(kThreads, 1) score_kernel(const ScoreParams P)
{
    extern __shared__ __align__(128) unsigned char smem_raw[];
    Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
    const int tid = threadIdx.x;
    const int n_inst = P.n_inst;
    if (tid == kThreads - 1) {  // row 4: the invalid classes (visible after the first barrier)
        const float inf = __int_as_float(0x7f800000);
        sm.brk[4][0] = sm.brk[4][1] = make_float4(inf, inf, inf, inf);
        sm.seg_e[4][0] = make_float4(0.0f, 0.0f, __int_as_float(0x7fc00000), __int_as_float(-1));
        sm.nseg[4] = 1;
    }

    // ---- stage the instance state first: it heads the critical path (state -> envelopes -> scoring), so
    // its TMA bulk copy is issued before the request prefetch (plain loads when unaligned)
    const uint32_t bytes = (uint32_t)n_inst * 4u;
    const bool bulk = kVec && (bytes % 16u == 0) && (((uintptr_t)P.Q | (uintptr_t)P.A | (uintptr_t)P.kap) % 16u == 0);
    const uint32_t bar = smem_addr(&sm.bar);
    if (bulk && tid == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(bar) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // launched as a programmatic dependent: nothing the previous kernel in the stream
    // writes is read before it has completed; the next launch may be scheduled at once
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    if (bulk && tid == 0) {
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(3u * bytes) : "memory");
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

    // the first two request vectors of this thread, in flight while the block builds its envelopes
    const int64_t nv = kVec ? (P.n >> 2) : 0;
    ReqPipe q;
    pipe_start(q, P, nv, tid);

    if (bulk) {
        __syncthreads();  // the barrier is initialised before any thread polls it
        auto staged = [&]() {  // bounded polling of the staging barrier
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
            return done != 0;
        };
        if (__syncthreads_or(!staged())) {  // block-uniform decision
            // never expected: report it, give the copies in flight a second bounded wait
            // (the block must not leave with them still writing its shared memory),
            // and score nothing: the call's outputs are unspecified
            if (tid == 0 && P.status) atomicExch(P.status, CTR_ETIMEOUT);
            (void)__syncthreads_or(!staged());
            return;
        }
    } else {
        for (int d = tid; d < n_inst; d += kThreads) {
            sm.q[d] = P.Q[d];
            sm.a[d] = P.A[d];
            sm.kap[d] = P.kap[d];
        }
    }
    __syncthreads();
    if (n_inst <= 64) {  // warps 0-3 build the four class envelopes from the staged state
        if (tid < 128) warp_envelope(sm, P, tid >> 5, n_inst, tid & 31);
        __syncthreads();
    } else {
        for (int d = tid; d < n_inst; d += kThreads) {
            sm.bk[d] = P.c[0] * fmaf(P.c[5], sm.q[d], P.c[7] * sm.a[d]);
            sm.wqa[d] = P.c[2] * sm.a[d];
        }
        __syncthreads();
        // ---- per-class lower envelope over all lines
        for (int idx = tid; idx < 4 * n_inst; idx += kThreads) {
            const int s = idx / n_inst, d = idx - s * n_inst;
            line_of(sm, P, s, d, sm.la[s][d], sm.lm[s][d]);
        }
        if (tid < 4) sm.nseg[tid] = 0;
        __syncthreads();
        // wider pools: each (class, line) pair is handled by tpp threads that
        // split its scans over the other lines and combine them with butterfly
        // shuffles, so all 32 warps of the block share the O(n^2) work
        int tpp = kThreads / (4 * n_inst);  // threads per pair: a power of two in [1, 32]
        tpp = tpp >= 32 ? 32 : tpp >= 16 ? 16 : tpp >= 8 ? 8 : tpp >= 4 ? 4 : tpp >= 2 ? 2 : 1;
        const int pair = tid / tpp, part = tid - pair * tpp;
        const bool act = pair < 4 * n_inst;
        const int es = act ? pair / n_inst : 0;
        const int ed = act ? pair - es * n_inst : 0;
        const float ad = sm.la[es][ed], md = sm.lm[es][ed];
        // Pareto filter: a line with a smaller-or-equal intercept and slope (ties: lowest index) hides it
        bool dominated = false;
        if (act) {
#pragma unroll 4
            for (int e = part; e < n_inst; e += tpp) {
                const float ae = sm.la[es][e], me = sm.lm[es][e];
                dominated |= ae <= ad && me <= md && (ae < ad || me < md || e < ed);
            }
        }
        for (int off = 1; off < tpp; off <<= 1) dominated |= __shfl_xor_sync(0xffffffffu, dominated, off, tpp);
        if (act && part == 0) sm.pareto[es][ed] = !dominated;
        __syncthreads();
        // the o_hat interval on which a surviving line wins
        const bool cand = act && sm.pareto[es][ed];
        float lo = 0.0f, hi = __int_as_float(0x7f800000);
        if (cand) {
#pragma unroll 4
            for (int e = part; e < n_inst; e += tpp) {
                if (e == ed || !sm.pareto[es][e]) continue;
                const float ae = sm.la[es][e], me = sm.lm[es][e];
                if (me > md) {
                    lo = fmaxf(lo, (ad - ae) / (me - md));
                } else if (me < md) {
                    hi = fminf(hi, (ae - ad) / (md - me));
                }
            }
        }
        for (int off = 1; off < tpp; off <<= 1) {
            lo = fmaxf(lo, __shfl_xor_sync(0xffffffffu, lo, off, tpp));
            hi = fminf(hi, __shfl_xor_sync(0xffffffffu, hi, off, tpp));
        }
        const bool valid = cand && lo < hi;
        if (act && part == 0) {
            sm.valid_tmp[es][ed] = valid;
            sm.lo_tmp[es][ed] = lo;
        }
        __syncthreads();
        // rank of each winning interval by its left end
        int rank = 0;
        if (valid) {
#pragma unroll 4
            for (int e = part; e < n_inst; e += tpp) {
                const float le = sm.lo_tmp[es][e];
                rank += sm.valid_tmp[es][e] && (le < lo || (le == lo && e < ed));
            }
        }
        for (int off = 1; off < tpp; off <<= 1) rank += __shfl_xor_sync(0xffffffffu, rank, off, tpp);
        if (valid && part == 0) {
            sm.seg_lo[es][rank] = lo;
            sm.seg_e[es][rank] = seg_entry(sm, P, es, ed);
            atomicAdd(&sm.nseg[es], 1);
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
            sm.seg_e[tid][0] = seg_entry(sm, P, tid, best);
            sm.nseg[tid] = 1;
        }
        __syncthreads();

        if (tid < 4 * 8) {  // padded breakpoints for the branch-free segment count
            const int cs = tid >> 3, t = (tid & 7) + 1;
            float* b = reinterpret_cast<float*>(&sm.brk[cs][0]);
            b[t - 1] = t < sm.nseg[cs] ? sm.seg_lo[cs][t] : __int_as_float(0x7f800000);
        }
        __syncthreads();
    }

    // ---- stream the requests (the first vectors were loaded before the prologue); the
    // segment search is chosen once per block from the longest envelope
    int maxseg = sm.nseg[0];
    for (int c = 1; c < 4; ++c) maxseg = sm.nseg[c] > maxseg ? sm.nseg[c] : maxseg;
    if (kVec) {
        if (maxseg <= 5)
            pipe_score<4>(q, sm, P);
        else if (maxseg <= 8)
            pipe_score<8>(q, sm, P);
        else
            pipe_score<0>(q, sm, P);
        if (blockIdx.x == 0 && tid < (int)(P.n & 3)) {
            const int64_t i = (nv << 2) + tid;
            int ai;
            float fc;
            score_one<0>(sm, P, P.c[6] * P.c[3] * P.c[8], P.p[i], P.oh[i], P.cls[i], ai, fc);
            P.argmin[i] = ai;
            P.cost[i] = fc;
        }
    } else {
        for (int64_t i = (int64_t)blockIdx.x * kThreads + tid; i < P.n; i += (int64_t)gridDim.x * kThreads) {
            int ai;
            float fc;
            score_one<0>(sm, P, P.c[6] * P.c[3] * P.c[8], P.p[i], P.oh[i], P.cls[i], ai, fc);
            P.argmin[i] = ai;
            P.cost[i] = fc;
        }
    }
}

// The scorer's memory traffic without its arithmetic or prologue: the same
// grid, launch attributes, 128-bit streaming loads two vectors ahead and
// streaming stores, writing class and p + o_hat.  It measures the HBM ceiling
// the scorer can reach at a given size.  It takes the vectors in grid-stride
// order, which streams faster on its own than the scorer's contiguous block
// ranges, so the ceiling it gives is the stricter of the two.
__global__ void __launch_bounds__(kThreads, 1) stream_probe_kernel(const ScoreParams P)
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    const int64_t nv = P.n >> 2;
    const int64_t stride = (int64_t)gridDim.x * kThreads;
    const float4* p4 = reinterpret_cast<const float4*>(P.p);
    const float4* o4 = reinterpret_cast<const float4*>(P.oh);
    const uint32_t* c4 = reinterpret_cast<const uint32_t*>(P.cls);
    int4* a4 = reinterpret_cast<int4*>(P.argmin);
    float4* f4 = reinterpret_cast<float4*>(P.cost);
    int64_t v = (int64_t)blockIdx.x * kThreads + threadIdx.x;
    bool has = v < nv;
    float4 pv = make_float4(0.f, 0.f, 0.f, 0.f), ov = pv, pn = pv, on = pv;
    uint32_t cv = 0, cn = 0;
    if (has) {
        pv = ld_stream(p4 + v);
        ov = ld_stream(o4 + v);
        cv = ld_stream_u32(c4 + v);
    }
    bool hn = v + stride < nv;
    if (hn) {
        pn = ld_stream(p4 + v + stride);
        on = ld_stream(o4 + v + stride);
        cn = ld_stream_u32(c4 + v + stride);
    }
    while (has) {
        const int64_t vf = v + 2 * stride;
        const bool hf = vf < nv;
        float4 pf = make_float4(0.f, 0.f, 0.f, 0.f), of = pf;
        uint32_t cf = 0;
        if (hf) {
            pf = ld_stream(p4 + vf);
            of = ld_stream(o4 + vf);
            cf = ld_stream_u32(c4 + vf);
        }
        __stcs(a4 + v, make_int4((int)(cv & 0xFFu), (int)((cv >> 8) & 0xFFu), (int)((cv >> 16) & 0xFFu),
                                 (int)(cv >> 24)));
        __stcs(f4 + v, make_float4(pv.x + ov.x, pv.y + ov.y, pv.z + ov.z, pv.w + ov.w));
        v += stride;
        has = hn;
        pv = pn;
        ov = on;
        cv = cn;
        hn = hf;
        pn = pf;
        on = of;
        cn = cf;
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
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = (size_t)smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (vec) {
        err = cudaFuncSetAttribute(score_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (err != cudaSuccess) return err;
        err = cudaLaunchKernelEx(&cfg, score_kernel<true>, p);
    } else {
        err = cudaFuncSetAttribute(score_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (err != cudaSuccess) return err;
        err = cudaLaunchKernelEx(&cfg, score_kernel<false>, p);
    }
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
}

cudaError_t launch_stream_probe(const ScoreParams& p, cudaStream_t stream)
{
    if (p.n < 4) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    int64_t blocks = ((p.n >> 2) + kThreads - 1) / kThreads;
    if (blocks > sms) blocks = sms;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)blocks);
    cfg.blockDim = dim3(kThreads);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    err = cudaLaunchKernelEx(&cfg, stream_probe_kernel, p);
    if (err != cudaSuccess) return err;
    return cudaGetLastError();
}

}  // namespace ctr
