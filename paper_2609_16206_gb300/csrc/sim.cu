// sim.cu -- batched discrete-event simulation of request routing
// (ctr_simulate): Algorithm 1 of the paper inside the sec. III-D simulator,
// with the continuous decode batching of sec. VI, the marginal-cost score of
// sec. III-A and the sec. IV-C baselines.
//
// Layout: a row is (replica x cost-constant set x policy); a lane group of G
// lanes (G = the next power of two >= the pool size) simulates one row, lane
// i < n_pre being prefill instance i and lane n_pre + d decode instance d, and
// a warp carries 32 / G rows side by side (the policies of one replica, which
// share arrival times).  Warps are persistent and pull row groups from an
// atomic counter in the workspace.  For every arrival k:
//   1. each decode lane advances its own instance's event loop to t_k
//      (runs of plain steps in closed form, step ends, KV-ready requests,
//      FCFS admissions, step starts); each prefill lane retires prefills that
//      ended by t_k (or, with batched prefill, ends and starts its batches
//      first and hands the members' KV-ready times to the decode lanes);
//   2. every lane prices its instance for the row's policy, and two argmins
//      within the lane group (ties to the lowest lane) pick i_pre and i_dec;
//   3. the i_pre lane commits the prefill, broadcasts the KV-ready time when
//      it is known, and the i_dec lane queues the request.
// All time and cost arithmetic is int64 fixed point, so every decision is
// deterministic.  Instances never interact except through routing, so the
// per-lane event loops reproduce the global event order exactly (events at
// an arrival's own time are processed before it is routed).
//
// Per-lane structures live in the workspace slot of the warp, each lane's
// entries contiguous (a heap's top levels then share cache lines; the heaps
// are 4-ary, a node's four children two 16-byte words and a heap of n keys
// about log4 n levels deep, except with batched prefill: see heap_push_bin): a min-heap of
// pending KV-ready keys (t_ready << 23 | k) per decode lane (the prefill
// lanes use the same region as their in-flight ring of prefill end times,
// packed with the prompt length as end << 21 | p), a min-heap of active
// requests keyed by finishing step (finish << 23 | k), and a FIFO ring of
// KV-ready requests awaiting admission.  Heap tops are cached in registers,
// so a run of plain decode steps touches no memory.  The row checksum's
// routing terms are summed here; its first-token and completion terms are
// summed by hash_kernel from the outputs.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

constexpr uint64_t kEmpty = ~0ull;
constexpr unsigned kFull = 0xffffffffu;
constexpr int kWarpsPerBlock = 4;
constexpr int64_t kNever = INT64_MAX;
constexpr int64_t kBacklogClamp = int64_t(1) << 40;
constexpr int64_t kPressureClamp = int64_t(1) << 18;
constexpr int kRecipN = 1024;  // batch sizes with a tabulated reciprocal
constexpr int kRingPBits = 21;  // prefill ring entry: end << 21 | p (p <= 2^20)
constexpr int64_t kRingPMask = (int64_t(1) << kRingPBits) - 1;
constexpr int kRingKShift = 26;  // batched prefill ring entry: k << 26 | d << 21 | p

// floor((2^64 - 1) / n) for n = 1..kRecipN, for the decode backlog's division
// by the batch size (built at compile time, read through the read-only path)
struct RecipTable {
    uint64_t v[kRecipN + 1];
};
constexpr RecipTable make_recip_table()
{
    RecipTable t{};
    for (int i = 1; i <= kRecipN; ++i) t.v[i] = ~0ull / (uint64_t)i;
    return t;
}
__device__ const RecipTable kRecipTable = make_recip_table();

// floor(num / d) with r = floor((2^64 - 1) / d): the estimate is low by at most 2
__device__ __forceinline__ uint64_t div_recip(uint64_t num, uint64_t d, uint64_t recip)
{
    uint64_t q = __umul64hi(num, recip);
    uint64_t r = num - q * d;
    if (r >= d) {
        ++q;
        r -= d;
    }
    if (r >= d) ++q;
    return q;
}

// floor(x / d) for 0 <= x < 2^56 and 0 < d < 2^37: an fp32 estimate (both
// operands rounded to fp32, relative error of the quotient a few 2^-24), then
// exact integer correction (the estimate is within one unit of the quotient
// whenever the quotient is below 2^20, the only case the simulator asks for;
// larger quotients fall back to division).
__device__ __forceinline__ int64_t floor_div_small(int64_t x, int64_t d)
{
    const float xf = __ll2float_rn(x);
    const float df = __ll2float_rn(d);
    const float qf = __fdividef(xf, df);
    if (!(qf < 1048576.0f)) return x / d;
    int32_t q = __float2int_rz(qf);  // within one of the quotient, below 2^20
    int64_t r = x - (int64_t)q * d;
    while (r < 0) {
        --q;
        r += d;
    }
    while (r >= d) {
        ++q;
        r -= d;
    }
    return q;
}

// floor(x / kv_div) for 0 <= x < 2^32 with magic = ceil(2^64 / kv_div), exact: the
// 96-bit product x * magic shifted right by 64, from two 32 x 32-bit products
__device__ __forceinline__ int64_t kv_term(int64_t x, const SimParams& P)
{
    if (P.kv_div == 1) return x;
    const uint32_t xl = (uint32_t)x;
    const uint64_t lo = (uint64_t)xl * (uint32_t)P.kv_div_magic;
    const uint64_t hi = (uint64_t)xl * (uint32_t)(P.kv_div_magic >> 32);
    return (int64_t)((hi + (lo >> 32)) >> 32);  // no overflow: hi <= 2^64 - 2^33 + 1
}

// Entries per lane of a heap region holding up to cap keys.  The heaps are
// 4-ary: node j (0-based) sits at position j + 3, so its children 4j + 1 ..
// 4j + 4 sit at positions 4j + 4 .. 4j + 7, a 32-byte aligned block read as
// two 16-byte words; the region has cap + 3 entries rounded up to 4.
__host__ __device__ __forceinline__ int64_t heap_stride(int64_t cap) { return (cap + 6) & ~int64_t(3); }

constexpr int kHeapRoot = 3;

// min-heap of unique 64-bit keys; each lane's heap is contiguous
__device__ __forceinline__ void heap_push(uint64_t* h, int32_t& n, uint64_t& top, uint64_t key, int64_t lim,
                                          bool& bad)
{
    int i = kHeapRoot + n++;
    while (i > kHeapRoot) {
        const int parent = (i >> 2) + 2;
        const uint64_t pv = ck_ld(h, parent, lim, bad);
        if (pv < key) break;
        ck_st(h, i, lim, pv, bad);
        i = parent;
    }
    ck_st(h, i, lim, key, bad);
    if (i == kHeapRoot) top = key;
}

__device__ __forceinline__ void heap_pop(uint64_t* h, int32_t& n, uint64_t& top, int64_t lim, bool& bad)
{
    const int m = n--;  // the last key moves into the hole left at the root
    if (m == 1) {
        top = kEmpty;
        return;
    }
    const int lastp = kHeapRoot + m - 1;
    const uint64_t last = ck_ld(h, lastp, lim, bad);
    const int endp = lastp - 1;  // position of the last key that stays
    int i = kHeapRoot;
    for (;;) {
        const int c = (i - 2) << 2;  // first child
        if (c > endp) break;
        const ulonglong2 c01 = ck_ld2(h + c, 0, lim - c, bad);  // the block of four as two 16-byte words
        const ulonglong2 c23 = ck_ld2(h + c, 2, lim - c, bad);
        uint64_t cv = c01.x;
        int ci = c;
        if (c + 1 <= endp && c01.y < cv) {
            cv = c01.y;
            ci = c + 1;
        }
        if (c + 2 <= endp && c23.x < cv) {
            cv = c23.x;
            ci = c + 2;
        }
        if (c + 3 <= endp && c23.y < cv) {
            cv = c23.y;
            ci = c + 3;
        }
        if (last < cv) break;
        ck_st(h, i, lim, cv, bad);
        i = ci;
    }
    ck_st(h, i, lim, last, bad);
    top = ck_ld(h, kHeapRoot, lim, bad);
}

// Binary 1-based variants (children 2i and 2i + 1 in one 16-byte word), kept
// for batched prefill: its short-output document workload keeps decode batches
// small, where the extra compares of a 4-ary level cost more than the saved
// levels (4,096 x 10,000: 97.6 ms binary, 104.1 ms 4-ary; the replica sweep and
// the large pool are 2 % and 6 % faster 4-ary).  Same region stride.
__device__ __forceinline__ void heap_push_bin(uint64_t* h, int32_t& n, uint64_t& top, uint64_t key, int64_t lim,
                                              bool& bad)
{
    int i = ++n;
    while (i > 1) {
        const int parent = i >> 1;
        const uint64_t pv = ck_ld(h, parent, lim, bad);
        if (pv < key) break;
        ck_st(h, i, lim, pv, bad);
        i = parent;
    }
    ck_st(h, i, lim, key, bad);
    if (i == 1) top = key;
}

__device__ __forceinline__ void heap_pop_bin(uint64_t* h, int32_t& n, uint64_t& top, int64_t lim, bool& bad)
{
    const int m = n--;
    if (m == 1) {
        top = kEmpty;
        return;
    }
    const uint64_t last = ck_ld(h, m, lim, bad);
    const int sz = m - 1;
    int i = 1;
    for (;;) {
        const int c = 2 * i;
        if (c > sz) break;
        const ulonglong2 ch = ck_ld2(h, c, lim, bad);  // c even: a 16-byte word
        uint64_t cv = ch.x;
        int ci = c;
        if (c < sz && ch.y < cv) {
            cv = ch.y;
            ci = c + 1;
        }
        if (last < cv) break;
        ck_st(h, i, lim, cv, bad);
        i = ci;
    }
    ck_st(h, i, lim, last, bad);
    top = ck_ld(h, 1, lim, bad);
}

// the heap operations of a kernel instantiation: binary with batched prefill, else 4-ary
template <bool kBin>
__device__ __forceinline__ void hpush(uint64_t* h, int32_t& n, uint64_t& top, uint64_t key, int64_t lim, bool& bad)
{
    if constexpr (kBin)
        heap_push_bin(h, n, top, key, lim, bad);
    else
        heap_push(h, n, top, key, lim, bad);
}
template <bool kBin>
__device__ __forceinline__ void hpop(uint64_t* h, int32_t& n, uint64_t& top, int64_t lim, bool& bad)
{
    if constexpr (kBin)
        heap_pop_bin(h, n, top, lim, bad);
    else
        heap_pop(h, n, top, lim, bad);
}

// argmin over the lanes of 64-bit values (ties -> lowest lane)
__device__ __forceinline__ int warp_argmin(uint64_t v)
{
    const uint32_t hi = (uint32_t)(v >> 32), lo = (uint32_t)v;
    const uint32_t mhi = __reduce_min_sync(kFull, hi);
    const uint32_t mlo = __reduce_min_sync(kFull, hi == mhi ? lo : 0xffffffffu);
    const uint32_t ball = __ballot_sync(kFull, hi == mhi && lo == mlo);
    return __ffs(ball) - 1;
}

// A decode lane's state.  `sum` is the one in-flight sum the row's policy
// reads: the true remaining output tokens R for the learned router on the true
// backlog, the predicted lengths o_hat for the length heuristic and the proxy's
// ledger (sum_is_o_hat), nothing for the others.
struct Decode {
    int64_t step_end, sum;
    int32_t step_idx;        // steps ended; the step budget keeps it and every completion step below 2^31
    int32_t kv_res, kv_rsv;  // resident <= reserved <= C < 2^31 tokens
    uint64_t pend_top, act_top;
    int32_t n_act, q, pend_n, w_head, w_n;  // n_act is also the active heap's size
    bool stepping;
};

// Move every pending request whose KV is ready by t into the waiting FIFO, in
// (time, index) order; the FIFO's size is checked after each insertion.
template <int kArity>
__device__ __forceinline__ int flush_ready(Decode& s, int64_t t, const SimParams& P, uint64_t* pend, uint32_t* wait,
                                           bool& bad)
{
    while (s.pend_n > 0 && (int64_t)(s.pend_top >> kKeyBits) <= t) {
        const uint32_t k = (uint32_t)(s.pend_top & kKeyMask);
        hpop<kArity == 2>(pend, s.pend_n, s.pend_top, heap_stride(P.cap_pr), bad);
        if (s.w_n == P.cap_wait) return CTR_EOVERFLOW;
        int pos = s.w_head + s.w_n;
        if (pos >= P.cap_wait) pos -= P.cap_wait;
        ck_st(wait, pos, P.cap_wait, k, bad);
        s.w_n += 1;
    }
    return CTR_OK;
}

// Advance one decode instance through every event at times <= T.  The pending
// heap may hold requests already KV-ready (taken at the next step end); it has
// room for cap_pend + cap_wait + 1 entries, so a full heap means the waiting
// FIFO has overflowed.  kSnap: when tsnap >= 0, also record in kv_snap the
// resident KV as it is after every event at times <= tsnap (an occupancy
// poll; tsnap <= T), then set tsnap to -1.
template <bool kSnap, int kArity>
__device__ __forceinline__ int decode_advance(Decode& s, int64_t T, const SimParams& P, uint64_t* pend, uint64_t* act,
                                              uint32_t* wait, int64_t tb, int64_t ob, int64_t& tsnap, int64_t& kv_snap,
                                              bool sum_is_o_hat, bool& bad)
{
    for (;;) {
        // Plain step ends first: the step ends by T, no request finishes with
        // it, nothing has become KV-ready by then and nobody waits for
        // admission, so the batch is unchanged and the next step starts at
        // once.  Lanes leave this loop at their next non-plain event, which
        // the handler below takes.
        const int64_t tp = s.pend_n > 0 ? (int64_t)(s.pend_top >> kKeyBits) : kNever;
        const int64_t limit = tp <= T ? tp - 1 : T;  // plain step ends lie at or before limit
        // The run is taken in closed form: while the floor(KV / kv_div) term of
        // the step time is unchanged every step lasts S, so the number of plain
        // ends is the least of the steps before the next completion, the steps
        // before that term changes, and the steps that end by the limit.
        while (s.stepping && s.step_end <= limit && s.w_n == 0) {
            const int32_t m_fin = (int32_t)(s.act_top >> kKeyBits) - s.step_idx - 1;  // <= 2^20
            if (m_fin <= 0) break;
            const int32_t n = s.n_act;
            const int64_t q1 = kv_term(s.kv_res + n, P);  // KV term of the next step
            const int64_t S = P.dec_base + (int64_t)(int32_t)P.dec_seq * n + q1;
            // plain end j happens at step_end + (j - 1) S <= limit (usually the binding bound)
            int32_t m = (int32_t)m_fin;
            const int64_t span = limit - s.step_end;
            if ((int64_t)(m - 1) * S > span) {  // then span < 2^20 * 2^37
                m = (int32_t)(span < (int64_t(1) << 56) ? floor_div_small(span, S) : span / S) + 1;
            }
            // the term stays q1 while j n <= room; q1 + 1 <= 2^31 and kv_div <= 2^31
            const int64_t room = (int64_t)((uint64_t)(uint32_t)(q1 + 1) * (uint32_t)P.kv_div) - 1 - s.kv_res;
            if ((int64_t)m * n > room) {  // the KV term changes first: m = floor(room / n) >= 1
                m = n <= kRecipN ? (int32_t)div_recip((uint64_t)room, (uint64_t)n, __ldg(&kRecipTable.v[n]))
                                 : (int32_t)(room / n);
            }
            if constexpr (kSnap) {
                // the poll instant falls before this run or inside it: the occupancy
                // there follows from the number of the run's ends by then
                if (tsnap >= 0) {
                    if (tsnap < s.step_end) {
                        kv_snap = s.kv_res;
                        tsnap = -1;
                    } else if (tsnap < s.step_end + (int64_t)(m - 1) * S) {
                        const int64_t d = tsnap - s.step_end;  // < (m - 1) S < 2^57
                        const int64_t j = (d < (int64_t(1) << 56) ? floor_div_small(d, S) : d / S) + 1;
                        kv_snap = s.kv_res + j * (int64_t)n;
                        tsnap = -1;
                    }
                }
            }
            const int64_t mn = (int64_t)m * n;
            s.step_idx += m;
            s.kv_res += (int32_t)mn;  // stays within the reservation
            if (!sum_is_o_hat) s.sum -= mn;  // R: every active request is one token closer
            if (s.step_idx >= (int32_t)P.max_steps) return CTR_ETIMEOUT;
            s.step_end += (int64_t)m * S;
            if (s.step_end >= kTimeLimit) return CTR_EOVERFLOW;
        }
        // A KV-ready event while a step runs only matters at the step's end (the
        // next admission), so it is taken there, in the same pass: the next
        // event is the running step's end, or the next KV-ready when idle.
        const int64_t tev = s.stepping ? s.step_end : tp;
        if constexpr (kSnap) {
            if (tsnap >= 0 && tev > tsnap) {  // every event by the poll instant is done
                kv_snap = s.kv_res;
                tsnap = -1;
            }
        }
        if (tev > T) return CTR_OK;
        if (s.stepping) {  // (1) the running step ends: one token for every active request
            s.step_idx += 1;
            s.kv_res += s.n_act;
            if (!sum_is_o_hat) s.sum -= s.n_act;
            s.stepping = false;
            while (s.n_act > 0 && (int32_t)(s.act_top >> kKeyBits) == s.step_idx) {
                const int64_t k = (int64_t)(s.act_top & kKeyMask);
                hpop<kArity == 2>(act, s.n_act, s.act_top, heap_stride(P.cap_act), bad);
                const int64_t pk = ck_ldg(P.trace.prompt_len, tb + k, P.trace_len, bad);
                const int64_t ok = ck_ldg(P.trace.true_out, tb + k, P.trace_len, bad);
                s.q -= 1;
                s.kv_res -= (int32_t)(pk + ok);
                s.kv_rsv -= (int32_t)(pk + ok);
                if (sum_is_o_hat) s.sum -= ck_ldg(P.trace.pred_out, tb + k, P.trace_len, bad);
                ck_st(P.t_done, ob + k, P.out_len, tev, bad);
            }
        }
        // (2) every request KV-ready by now joins the waiting FIFO in (time, index) order
        const int rc = flush_ready<kArity>(s, tev, P, pend, wait, bad);
        if (rc != CTR_OK) return rc;
        // (3) not mid-step: strict FCFS admission while the reservation fits, then start a step
        if (!s.stepping) {
            const int pos0 = s.w_head;
            int admitted = 0;
            while (s.w_n > 0) {
                const uint32_t k = ck_ld(wait, s.w_head, P.cap_wait, bad);
                const int64_t pk = ck_ldg(P.trace.prompt_len, tb + k, P.trace_len, bad);
                const int64_t ok = ck_ldg(P.trace.true_out, tb + k, P.trace_len, bad);
                if ((uint32_t)s.kv_rsv + (uint32_t)(pk + ok) > (uint32_t)P.kv_cap) break;  // < 2^31 + 2^21
                if (s.n_act == P.cap_act) return CTR_EOVERFLOW;
                s.w_head = s.w_head + 1 == P.cap_wait ? 0 : s.w_head + 1;
                s.w_n -= 1;
                s.kv_rsv += (int32_t)(pk + ok);
                s.kv_res += (int32_t)pk;
                hpush<kArity == 2>(act, s.n_act, s.act_top, ((uint64_t)(s.step_idx + ok) << kKeyBits) | k,
                                   heap_stride(P.cap_act), bad);
                admitted += 1;
            }
            if (s.n_act > 0) {
                if (s.step_idx >= (int32_t)P.max_steps) return CTR_ETIMEOUT;  // steps started on this instance
                s.step_end = tev + P.dec_base + (int64_t)(int32_t)P.dec_seq * s.n_act + kv_term(s.kv_res, P);
                if (s.step_end >= kTimeLimit) return CTR_EOVERFLOW;
                s.stepping = true;
                int pos = pos0;
                for (int i = 0; i < admitted; ++i) {  // first token at the end of this step
                    const uint32_t k = ck_ld(wait, pos, P.cap_wait, bad);
                    ck_st(P.t_first, ob + k, P.out_len, s.step_end, bad);
                    pos = pos + 1 == P.cap_wait ? 0 : pos + 1;
                }
            }
            if (s.w_n == 0) s.w_head = 0;  // an empty ring restarts at its first entry (stays cache-resident)
        }
    }
}

// Per-request bounds, arrival order (CTR_EINVAL before anything is simulated).
__device__ __forceinline__ bool row_valid(const SimParams& P, int64_t tb, int lane, bool& bad)
{
    int64_t prev_last = 0;
    for (int64_t base = 0; base < P.n_req; base += 32) {
        const int64_t k = base + lane;
        const bool live = k < P.n_req;
        int64_t t = 0;
        bool bad = false;
        if (live) {
            t = ck_ld(P.trace.arrival_us, tb + k, P.trace_len, bad);
            const int64_t p = ck_ld(P.trace.prompt_len, tb + k, P.trace_len, bad);
            const int64_t o = ck_ld(P.trace.true_out, tb + k, P.trace_len, bad);
            const int64_t oh = ck_ld(P.trace.pred_out, tb + k, P.trace_len, bad);
            const int64_t c = ck_ld(P.trace.slo_class, tb + k, P.trace_len, bad);
            bad = t < 0 || t >= kArrivalLimit || p < 0 || p > (1 << 20) || o < 1 || o > (1 << 20) ||
                  p + o > P.kv_cap || oh < 0 || oh > (1 << 17) || c >= P.n_classes;
        }
        int64_t before = __shfl_up_sync(kFull, t, 1);
        if (lane == 0) before = prev_last;
        if (live && t < before) bad = true;
        if (__any_sync(kFull, bad)) return false;
        prev_last = __shfl_sync(kFull, t, 31);
    }
    return true;
}

// argmin of 64-bit values within aligned groups of G lanes (ties -> lowest lane),
// returned as the lane index inside the group: a butterfly minimum, then one
// ballot for the lanes that hold it (every lane of the warp calls it)
template <int G>
__device__ __forceinline__ int group_argmin(uint64_t v, int gl)
{
    if constexpr (G == 32) {
        return warp_argmin(v);
    } else {
        uint64_t m = v;  // the group's minimum, then its lowest lane holding it
#pragma unroll
        for (int off = G / 2; off > 0; off >>= 1) {
            const uint64_t o = __shfl_xor_sync(kFull, m, off, G);
            m = o < m ? o : m;
        }
        const uint32_t ball = __ballot_sync(kFull, v == m);
        return __ffs((ball >> ((threadIdx.x & 31) - gl)) & ((1u << G) - 1u)) - 1;
    }
}

// One warp carries 32 / G rows side by side: lanes [g*G, g*G + G) simulate
// row base_row + g, lane g*G + i being instance i of that row.  All rows of a
// workload have the same number of requests, so the groups walk their
// arrivals in lockstep (request k of every row at once, each at its own time);
// the per-lane event loops, the per-group argmins and the commits are
// independent across groups.  kMode 1 compiles in the deployed proxy's
// signals (ledger backlog, polled occupancy), kMode 2 batched prefill as
// well; the host launches the least instantiation a launch needs.
//
// Batched prefill: a prefill lane's ring holds its in-flight requests as
// k << 26 | d << 21 | p (running batch first, then the queue).  Before the
// decode lanes advance to an arrival, the prefill lanes end every batch that
// ends by then and start the next at that instant; each newly started batch
// (contiguous at the ring's head) is published to the group, and every
// decode lane copies its own members, now with known KV-ready times, into its
// pending heap.  Repeated until no prefill lane has another batch ending.
template <int G, int kMode, int kBlocksPerSM>
__global__ void __launch_bounds__(kWarpsPerBlock * 32, kBlocksPerSM) sim_kernel(const __grid_constant__ SimParams P)
{
    constexpr bool kSig = kMode >= 1;  // the proxy's signals: ledger backlog, polled occupancy
    constexpr bool kBat = kMode == 2;  // batched prefill
    constexpr int kArity = kBat ? 2 : 4;  // heap arity: binary with batched prefill (see heap_push_bin)
    constexpr int kRowsPerWarp = 32 / G;
    const int lane = threadIdx.x & 31;
    const int grp = lane / G;
    const int gl = lane % G;
    const uint32_t gmask = G == 32 ? kFull : (((1u << G) - 1u) << (grp * G));
    const int64_t slot = (int64_t)blockIdx.x * kWarpsPerBlock + (threadIdx.x >> 5);
    if (slot >= P.n_slots) return;
    unsigned char* sb = P.ws + slot * P.slot_bytes;
    const int64_t pr_stride = heap_stride(P.cap_pr);
    uint64_t* pend = reinterpret_cast<uint64_t*>(sb) + lane * pr_stride;  // decode lanes: 4-ary heap
    int64_t* ring = reinterpret_cast<int64_t*>(sb) + lane * pr_stride;    // prefill lanes: ring from 0
    uint64_t* act = reinterpret_cast<uint64_t*>(sb + P.off_act) + lane * heap_stride(P.cap_act);
    uint32_t* wait = reinterpret_cast<uint32_t*>(sb + P.off_wait) + lane * P.cap_wait;

    const bool is_pre = gl < P.n_pre;
    const bool is_dec = gl >= P.n_pre && gl < P.n_pre + P.n_dec;
    const int64_t per_rep = (int64_t)P.n_sets * P.n_pols;
    const int64_t n = P.n_req;

    for (;;) {
        uint32_t base32 = 0;
        if (lane == 0) base32 = atomicAdd(P.next_row, (uint32_t)kRowsPerWarp);
        const int64_t base_row = __shfl_sync(kFull, base32, 0);
        if (base_row >= P.n_rows) break;
        const int64_t row = base_row + grp;
        const bool has_row = row < P.n_rows;
        const int64_t rep = has_row ? row / per_rep : 0;
        const int set = has_row ? (int)((row / P.n_pols) % P.n_sets) : 0;
        const int pol = has_row ? P.pols[row % P.n_pols] : CTR_POLICY_ROUND_ROBIN;
        const ConstsDev& cc = P.sets[set];
        // the in-flight sum the row's decode pricing reads: predicted lengths for the length
        // heuristic and the proxy's ledger, else true remaining tokens (unread by JSQ / RR)
        const bool learned_row = pol == CTR_POLICY_LEARNED || pol == CTR_POLICY_LEARNED_P2;
        const bool sum_is_o_hat = pol == CTR_POLICY_LENGTH_HEURISTIC || (kSig && learned_row && cc.proxy);
        const int64_t tb = rep * n;
        const int64_t ob = row * n;

        // per-request bounds, one row at a time with the whole warp
        bool oob = false;  // bounds-checked builds: an index of this lane fell outside its buffer
        bool valid = false;
        for (int g = 0; g < kRowsPerWarp; ++g) {
            const int64_t r = base_row + g;
            if (r >= P.n_rows) break;
            bool oob_g = false;
            const bool ok = row_valid(P, (r / per_rep) * n, lane, oob_g);
            if (g == grp) oob = oob_g;
            if (g == grp) valid = ok;
        }
        bool live = has_row && valid;

        Decode s;
        s.step_end = 0; s.step_idx = 0; s.kv_res = 0; s.kv_rsv = 0; s.sum = 0;
        s.pend_top = kEmpty; s.act_top = kEmpty;
        s.n_act = 0; s.q = 0; s.pend_n = 0; s.w_head = 0; s.w_n = 0;
        s.stepping = false;
        // A lane simulates a prefill or a decode instance, never both, so a prefill
        // lane keeps its state in decode fields it does not use (fewer live registers).
        int64_t& busy = s.step_end;    // end of the last prefill (of the running batch, when batched)
        uint64_t& ring_front = s.act_top;  // the ring's front entry (end << 21 | p), read while ring_n > 0
        int64_t& ring_sum_p = s.sum;       // prompt tokens of the prefills in the ring
        int32_t& ring_head = s.w_head;
        int32_t& ring_n = s.w_n;
        int64_t kv_seen = 0, last_poll = -1;     // decode lanes: occupancy at the last poll instant
        int32_t rr_p = 0, rr_d = 0;
        uint64_t h = 0;
        int err = CTR_OK;
        // batched prefill lanes: busy = end of the running batch of run_n members (run_p tokens); the
        // queue behind it, cut FCFS into budget-limited batches, forms q_batches, the last of q_tail tokens
        int32_t run_n = 0, q_batches = 0;
        int64_t run_p = 0, q_tail = 0;
        const bool batched = kBat && P.pre_batch > 0;

        // Batched prefill: end every batch that ends by T, start the next at that
        // instant, and hand the members' KV-ready times to their decode lanes
        // (warp-collective: every lane of the warp calls it).
        auto prefill_batches = [&](int64_t T) {
            for (;;) {
                int32_t pub_n = 0, pub_head = 0;
                int64_t pub_end = 0;
                if (live && err == CTR_OK && is_pre && run_n > 0 && busy <= T) {
                    ring_head += run_n;
                    if (ring_head >= P.cap_ring) ring_head -= P.cap_ring;
                    ring_n -= run_n;
                    ring_sum_p -= run_p;
                    run_n = 0;
                    run_p = 0;
                    if (ring_n > 0) {  // the next batch: the head, then FCFS while the budget holds
                        int pos = ring_head;
                        int64_t pmax = 0;
                        while (run_n < ring_n) {
                            const int64_t pj = ck_ld(ring, pos, (int64_t)P.cap_ring, oob) & kRingPMask;
                            if (run_n > 0 && run_p + pj > P.pre_batch) break;
                            run_p += pj;
                            pmax = pj > pmax ? pj : pmax;
                            run_n += 1;
                            pos = pos + 1 == P.cap_ring ? 0 : pos + 1;
                        }
                        busy += P.pre_base + P.pre_tok * run_p;
                        q_batches -= 1;
                        if (q_batches == 0) q_tail = 0;
                        if (busy + P.xfer_tok * pmax >= kTimeLimit) {
                            err = CTR_EOVERFLOW;
                        } else {
                            pub_n = run_n;
                            pub_head = ring_head;
                            pub_end = busy;
                        }
                    }
                }
                if (!__any_sync(kFull, pub_n > 0)) break;
                const int64_t* const rings = reinterpret_cast<const int64_t*>(sb);
                for (int i = 0; i < P.n_pre; ++i) {
                    const int src = grp * G + i;
                    const int32_t m_i = __shfl_sync(kFull, pub_n, src);
                    const int32_t h_i = __shfl_sync(kFull, pub_head, src);
                    const int64_t e_i = __shfl_sync(kFull, pub_end, src);
                    if (is_dec && live) {
                        int pos = h_i;
                        for (int32_t m = 0; m < m_i; ++m) {
                            const int64_t v = ck_ld(rings + src * pr_stride, pos, (int64_t)P.cap_ring, oob);
                            if ((int)((v >> kRingPBits) & 31) == gl - P.n_pre) {
                                const int64_t ready = e_i + P.xfer_tok * (v & kRingPMask);
                                if (s.pend_n == P.cap_pend_store) {
                                    err = CTR_EOVERFLOW;  // the waiting FIFO has overflowed
                                } else {
                                    hpush<kArity == 2>(pend, s.pend_n, s.pend_top,
                                              ((uint64_t)ready << kKeyBits) | (uint64_t)(v >> kRingKShift), pr_stride,
                                              oob);
                                }
                            }
                            pos = pos + 1 == P.cap_ring ? 0 : pos + 1;
                        }
                    }
                }
            }
        };

        for (int64_t base = 0; base < n; base += G) {
            if (!__any_sync(kFull, live)) break;
            const int64_t kl = base + gl;
            const bool mine = live && kl < n;
            int64_t my_t = 0;
            uint32_t my_pc = 0, my_o = 0, my_oh = 0;
            if (mine) {
                my_t = ck_ld(P.trace.arrival_us, tb + kl, P.trace_len, oob);
                my_pc = (uint32_t)ck_ld(P.trace.prompt_len, tb + kl, P.trace_len, oob) |
                        ((uint32_t)ck_ld(P.trace.slo_class, tb + kl, P.trace_len, oob) << 24);
                my_o = (uint32_t)ck_ld(P.trace.true_out, tb + kl, P.trace_len, oob);
                my_oh = (uint32_t)ck_ld(P.trace.pred_out, tb + kl, P.trace_len, oob);
            }
            uint32_t my_route = 0;
            const int cnt = (int)(n - base < G ? n - base : G);
            for (int j = 0; j < cnt; ++j) {
                const int64_t T = __shfl_sync(kFull, my_t, j, G);

                // 1. advance every instance to the arrival time
                if constexpr (kBat) {
                    if (batched) prefill_batches(T);
                }
                if (live) {
                    if (is_dec) {
                        int64_t tsnap = -1;
                        if (kSig && cc.poll_us > 0) {
                            // the router sees the occupancy of the last poll instant floor(T / D) D,
                            // taken after every event at that instant, on the way to T
                            const int64_t tp = (int64_t)div_recip((uint64_t)T, (uint64_t)cc.poll_us, cc.poll_recip) *
                                               cc.poll_us;
                            if (tp > last_poll) {
                                tsnap = tp;
                                last_poll = tp;
                            }
                        }
                        if (err == CTR_OK)
                            err = decode_advance<kSig, kArity>(s, T, P, pend, act, wait, tb, ob, tsnap, kv_seen,
                                                               sum_is_o_hat, oob);
                    } else if (is_pre && !batched) {
                        const int64_t thr = ((T + 1) << kRingPBits) - 1;  // entries whose prefill ended by T
                        while (ring_n > 0 && ring_front <= (uint64_t)thr) {
                            if constexpr (kSig) ring_sum_p -= ring_front & kRingPMask;
                            ring_head = ring_head + 1 == P.cap_ring ? 0 : ring_head + 1;
                            ring_n -= 1;
                            ring_front = ring_n > 0 ? (uint64_t)ck_ld(ring, ring_head, (int64_t)P.cap_ring, oob)
                                                    : (uint64_t)kNever;
                        }
                        if (ring_n == 0) ring_head = 0;
                    }
                }
                if (__ballot_sync(kFull, err != CTR_OK) & gmask) live = false;

                __syncwarp();  // the lanes leave their event loops at different passes: regroup
                // the request's features (read after the advance, which does not need them)
                const int64_t k = base + j;
                const uint32_t pc = __shfl_sync(kFull, my_pc, j, G);
                const int64_t pk = pc & 0xFFFFFFu;
                const int ck = (int)(pc >> 24);
                const int64_t ok = __shfl_sync(kFull, my_o, j, G);
                const int64_t ohk = __shfl_sync(kFull, my_oh, j, G);
                // 2. price the candidates and take the argmin of each pool
                uint64_t cost = kEmpty;
                if (live && pol != CTR_POLICY_ROUND_ROBIN) {
                    const bool learned = pol == CTR_POLICY_LEARNED || pol == CTR_POLICY_LEARNED_P2;
                    // feature ablation (sec. V-F): a removed feature takes its neutral value
                    const int64_t oh_f = (cc.ablate & CTR_ABLATE_PREDICTED_LENGTH) ? 0 : ohk;
                    const int64_t sig = (cc.ablate & CTR_ABLATE_SLO) ? 256 : cc.sigma[ck];
                    if (is_pre) {
                        if (learned) {
                            int64_t b = busy > T ? busy - T : 0;
                            if (batched) {  // the running batch's rest, then the queue's batches
                                b = (run_n > 0 && busy > T ? busy - T : 0) + P.pre_base * (int64_t)q_batches +
                                    P.pre_tok * (ring_sum_p - run_p);
                                if (b > kBacklogClamp) b = kBacklogClamp;
                            }
                            if (kSig && cc.proxy) {  // the ledger: tau_pre0 + tau_pre p per prefill not yet ended
                                b = cc.tau_pre0 * (int64_t)ring_n + cc.tau_pre * ring_sum_p;
                                if (b > kBacklogClamp) b = kBacklogClamp;
                            }
                            const int64_t load = cc.w_b * b + cc.w_s * (cc.tau_pre0 + pk * cc.tau_pre);
                            cost = (uint64_t)(load * sig + cc.w_q * (int64_t)ring_n * 65536);
                        } else {
                            cost = (uint64_t)ring_n;
                        }
                    } else if (is_dec) {
                        if (learned) {
                            const int64_t na = s.n_act;
                            const int64_t step = P.dec_base + (int64_t)(int32_t)P.dec_seq * s.n_act + kv_term(s.kv_res, P);
                            const uint64_t hi = __umul64hi((uint64_t)s.sum, (uint64_t)step);
                            const uint64_t lo = (uint64_t)s.sum * (uint64_t)step;
                            int64_t b;
                            if (hi != 0 || lo >= (1ull << 62)) {
                                b = kBacklogClamp;
                            } else {
                                const uint64_t nd = (uint64_t)(na > 1 ? na : 1);
                                b = (int64_t)(nd <= (uint64_t)kRecipN ? div_recip(lo, nd, __ldg(&kRecipTable.v[nd]))
                                                                      : lo / nd);
                                if (b > kBacklogClamp) b = kBacklogClamp;
                            }
                            if (kSig && cc.proxy) {  // the ledger: tau_dec o_hat per request routed here and not done
                                b = (cc.ablate & CTR_ABLATE_PREDICTED_LENGTH) ? 0 : cc.tau_dec * s.sum;
                                if (b > kBacklogClamp) b = kBacklogClamp;
                            }
                            const int64_t kv = kSig && cc.poll_us > 0 ? kv_seen : s.kv_res;
                            int64_t press = (int64_t)div_recip((uint64_t)(kv + pk + oh_f) << 16,
                                                               (uint64_t)P.kv_cap, P.kv_cap_recip);
                            if (press > kPressureClamp) press = kPressureClamp;
                            if (cc.ablate & CTR_ABLATE_PRESSURE) press = 0;
                            const int64_t own = oh_f * cc.tau_dec;
                            const int64_t priced = own + ((((own * press) >> 16) * cc.rho) >> 8);
                            const int64_t load = cc.w_b * b + cc.w_s * priced;
                            cost = (uint64_t)(load * sig + cc.w_q * (int64_t)s.q * 65536);
                        } else if (pol == CTR_POLICY_LENGTH_HEURISTIC && ohk >= P.heur_thresh) {
                            cost = (uint64_t)s.sum;
                        } else {
                            cost = (uint64_t)s.q;
                        }
                    }
                    if (pol == CTR_POLICY_LEARNED_P2 && (is_pre || is_dec)) {
                        // power of two choices: only two sampled candidates per pool are priced
                        const Philox4 u = philox4x32_10((uint32_t)k, (uint32_t)T, (uint32_t)((uint64_t)T >> 32),
                                                        0x5032u, 0x243F6A88u, 0x85A308D3u);
                        const uint32_t n_pool = is_pre ? (uint32_t)P.n_pre : (uint32_t)P.n_dec;
                        const uint32_t a0 = is_pre ? u.v[2] : u.v[0], a1 = is_pre ? u.v[3] : u.v[1];
                        const uint32_t c0 = (uint32_t)(((uint64_t)a0 * n_pool) >> 32);
                        uint32_t c1 = c0;
                        if (n_pool > 1) {
                            c1 = c0 + 1 + (uint32_t)(((uint64_t)a1 * (n_pool - 1)) >> 32);
                            if (c1 >= n_pool) c1 -= n_pool;
                        }
                        const uint32_t me = is_pre ? (uint32_t)gl : (uint32_t)(gl - P.n_pre);
                        if (me != c0 && me != c1) cost = kEmpty;
                    }
                }
                const int amin_p = group_argmin<G>(is_pre ? cost : kEmpty, gl);
                const int amin_d = group_argmin<G>(is_dec ? cost : kEmpty, gl);
                int ip, id;
                if (pol == CTR_POLICY_ROUND_ROBIN) {
                    ip = rr_p;
                    id = rr_d;
                } else {
                    ip = amin_p;
                    id = amin_d - P.n_pre;
                }
                rr_p = rr_p + 1 == P.n_pre ? 0 : rr_p + 1;
                rr_d = rr_d + 1 == P.n_dec ? 0 : rr_d + 1;

                // 3. commit: FCFS prefill, KV transfer, queue at the decode instance
                int64_t ready = 0;
                if (batched && live && gl == ip) {
                    if (ring_n == P.cap_ring) {
                        err = CTR_EOVERFLOW;
                        ready = kTimeLimit;
                    } else {
                        int pos = ring_head + ring_n;
                        if (pos >= P.cap_ring) pos -= P.cap_ring;
                        ck_st(ring, pos, (int64_t)P.cap_ring, (k << kRingKShift) | ((int64_t)id << kRingPBits) | pk, oob);
                        ring_n += 1;
                        ring_sum_p += pk;
                        if (run_n == 0) {  // an idle instance starts a batch of this request at once
                            busy = T + P.pre_base + (int64_t)(int32_t)P.pre_tok * (int32_t)pk;
                            run_n = 1;
                            run_p = pk;
                            ready = busy + (int64_t)(int32_t)P.xfer_tok * (int32_t)pk;
                            if (ready >= kTimeLimit) err = CTR_EOVERFLOW;
                        } else {  // queued: its KV-ready time is known when its batch starts
                            if (q_batches > 0 && q_tail + pk <= P.pre_batch) {
                                q_tail += pk;
                            } else {
                                q_batches += 1;
                                q_tail = pk;
                            }
                            ready = -1;
                        }
                    }
                } else if (live && gl == ip) {
                    const int64_t start = busy > T ? busy : T;
                    const int64_t end = start + P.pre_base + (int64_t)(int32_t)P.pre_tok * (int32_t)pk;
                    ready = end + (int64_t)(int32_t)P.xfer_tok * (int32_t)pk;
                    if (ready >= kTimeLimit) {
                        err = CTR_EOVERFLOW;
                    } else if (ring_n == P.cap_ring) {
                        err = CTR_EOVERFLOW;
                    } else {
                        busy = end;
                        int pos = ring_head + ring_n;
                        if (pos >= P.cap_ring) pos -= P.cap_ring;
                        const int64_t e = (end << kRingPBits) | pk;
                        ck_st(ring, pos, (int64_t)P.cap_ring, e, oob);
                        if (ring_n == 0) ring_front = (uint64_t)e;
                        ring_n += 1;
                        if constexpr (kSig) ring_sum_p += pk;
                    }
                }
                ready = __shfl_sync(kFull, ready, ip, G);
                if (live && gl == P.n_pre + id && ready < kTimeLimit) {
                    // requests routed here whose KV is not ready yet, exactly: first move
                    // those already ready (kept in the heap until the step end) if it matters
                    if (s.q - s.w_n - s.n_act >= P.cap_pend) err = flush_ready<kArity>(s, T, P, pend, wait, oob);
                    if (err != CTR_OK || s.q - s.w_n - s.n_act == P.cap_pend ||
                        (ready >= 0 && s.pend_n == P.cap_pend_store)) {
                        err = CTR_EOVERFLOW;
                    } else {
                        if (ready >= 0)
                            hpush<kArity == 2>(pend, s.pend_n, s.pend_top, ((uint64_t)ready << kKeyBits) | (uint64_t)k,
                                               pr_stride, oob);
                        s.q += 1;
                        s.sum += sum_is_o_hat ? ohk : ok;
                    }
                }
                if (gl == j) my_route = ((uint32_t)ip << 8) | (uint32_t)id;
                if (__ballot_sync(kFull, err != CTR_OK) & gmask) live = false;
            }
            if (mine && live) {
                // the routing term of the row checksum, all lanes at once (the
                // first-token and completion terms are added by hash_kernel)
                h += hterm(kl, 1, (uint64_t)my_route);
                if (P.i_pre) ck_st(P.i_pre, ob + kl, P.out_len, (uint8_t)(my_route >> 8), oob);
                if (P.i_dec) ck_st(P.i_dec, ob + kl, P.out_len, (uint8_t)(my_route & 0xFF), oob);
            }
        }
        // drain: every remaining batch, then every remaining event
        if constexpr (kBat) {
            if (batched) {
                prefill_batches(kNever - 1);
                if (__ballot_sync(kFull, err != CTR_OK) & gmask) live = false;
            }
        }
        if (live && is_dec) {
            int64_t no_snap = -1;
            err = decode_advance<false, kArity>(s, kNever - 1, P, pend, act, wait, tb, ob, no_snap, kv_seen, sum_is_o_hat,
                                                oob);
        }

#pragma unroll
        for (int off = G / 2; off > 0; off >>= 1) h += __shfl_xor_sync(kFull, h, off, G);
        int status = CTR_OK;
        if (__ballot_sync(kFull, err == CTR_ETIMEOUT) & gmask) status = CTR_ETIMEOUT;
        if (__ballot_sync(kFull, err == CTR_EOVERFLOW) & gmask) status = CTR_EOVERFLOW;
        if (has_row && !valid) status = CTR_EINVAL;
#if CTR_BOUNDS_CHECK
        if (__ballot_sync(kFull, oob) & gmask) status = CTR_EBOUNDS;
#endif
        if (gl == 0 && has_row) {
            P.row_status[row] = status;
            P.row_hash[row] = status == CTR_OK ? h : 0;
        }
    }
}

// The first-token and completion terms of the row checksum, one block per
// row over the simulator's outputs (coalesced; cheaper than hashing inside
// the diverged event handlers).  Rows that failed keep the checksum 0.
constexpr int kHashThreads = 256;
__global__ void __launch_bounds__(kHashThreads) hash_kernel(const __grid_constant__ SimParams P, const uint64_t* kmix)
{
    __shared__ uint64_t part[kHashThreads / 32];
    for (int64_t row = blockIdx.x; row < P.n_rows; row += gridDim.x) {
        if (P.row_status[row] != CTR_OK) continue;  // block-uniform
        const int64_t ob = row * P.n_req;
        uint64_t h = 0;
#pragma unroll 4
        for (int64_t k = threadIdx.x; k < P.n_req; k += kHashThreads) {
            const int64_t tf = __ldcs(&P.t_first[ob + k]);
            const int64_t td = __ldcs(&P.t_done[ob + k]);
            if (kmix)  // the request-only halves, mixed once per call (launch_mix_table)
                h += mix64(__ldg(&kmix[k]) ^ (uint64_t)tf) + mix64(__ldg(&kmix[P.n_req + k]) ^ (uint64_t)td);
            else
                h += hterm(k, 2, (uint64_t)tf) + hterm(k, 3, (uint64_t)td);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) h += __shfl_xor_sync(kFull, h, off);
        if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = h;
        __syncthreads();
        if (threadIdx.x == 0) {
            uint64_t t = 0;
            for (int w = 0; w < kHashThreads / 32; ++w) t += part[w];
            P.row_hash[row] += t;
        }
        __syncthreads();  // part[] is reused by the next row
    }
}

}  // namespace

int64_t sim_slot_bytes(const ctr_sim_cfg& cfg, int64_t* off_act, int64_t* off_wait, int32_t* cap_pr)
{
    const int64_t pend_store = (int64_t)cfg.cap_pending + cfg.cap_waiting + 1;  // pending heap entries
    const int64_t pr = pend_store > cfg.cap_prefill_ring ? pend_store : cfg.cap_prefill_ring;
    const int64_t a = heap_stride(pr) * 8 * kWarp;
    const int64_t b = a + heap_stride(cfg.cap_active) * 8 * kWarp;
    const int64_t c = b + (int64_t)cfg.cap_waiting * 4 * kWarp;
    *off_act = a;
    *off_wait = b;
    *cap_pr = (int32_t)pr;
    return (c + 255) / 256 * 256;
}

int sim_group_width(int n_instances)
{
    return n_instances <= 4 ? 4 : n_instances <= 8 ? 8 : n_instances <= 16 ? 16 : 32;
}

int sim_max_resident_warps(int* warps_per_block, int* blocks)
{
    int dev = 0, sms = 0, per_sm = 0, per_sm_g = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    // the smallest occupancy over the group widths and modes at 8 blocks per
    // SM, so one workspace size fits every launch
    per_sm = 1 << 30;
    const void* kernels[12] = {
        (const void*)sim_kernel<4, 0, 8>, (const void*)sim_kernel<8, 0, 8>, (const void*)sim_kernel<16, 0, 8>,
        (const void*)sim_kernel<32, 0, 8>, (const void*)sim_kernel<4, 1, 8>, (const void*)sim_kernel<8, 1, 8>,
        (const void*)sim_kernel<16, 1, 8>, (const void*)sim_kernel<32, 1, 8>, (const void*)sim_kernel<4, 2, 8>,
        (const void*)sim_kernel<8, 2, 8>, (const void*)sim_kernel<16, 2, 8>, (const void*)sim_kernel<32, 2, 8>};
    for (const void* k : kernels) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm_g, k, kWarpsPerBlock * 32, 0) != cudaSuccess)
            return 0;
        if (per_sm_g < per_sm) per_sm = per_sm_g;
    }
    *warps_per_block = kWarpsPerBlock;
    *blocks = sms * per_sm;
    return sms * per_sm * kWarpsPerBlock;
}

namespace {

// 7 blocks per SM (72 registers a thread, fewer spills) when all of the
// launch's persistent warps fit on the GPU at that occupancy -- the common
// case of one row group per warp -- else 8 (more warps to hide latency).
template <int G, int kMode>
cudaError_t launch_width(const SimParams& p, int blocks, cudaStream_t stream)
{
    int dev = 0, sms = 0, per_sm7 = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return cudaErrorInvalidDevice;
    cudaError_t e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm7, sim_kernel<G, kMode, 7>, kWarpsPerBlock * 32, 0);
    if (e != cudaSuccess) return e;
    if ((int64_t)p.n_slots <= (int64_t)sms * per_sm7 * kWarpsPerBlock)
        sim_kernel<G, kMode, 7><<<blocks, kWarpsPerBlock * 32, 0, stream>>>(p);
    else
        sim_kernel<G, kMode, 8><<<blocks, kWarpsPerBlock * 32, 0, stream>>>(p);
    return cudaGetLastError();
}

template <int kMode>
cudaError_t launch_mode(const SimParams& p, int blocks, cudaStream_t stream)
{
    switch (sim_group_width(p.n_pre + p.n_dec)) {
    case 4: return launch_width<4, kMode>(p, blocks, stream);
    case 8: return launch_width<8, kMode>(p, blocks, stream);
    case 16: return launch_width<16, kMode>(p, blocks, stream);
    default: return launch_width<32, kMode>(p, blocks, stream);
    }
}

}  // namespace

cudaError_t launch_sim(const SimParams& p, int blocks, int warps_per_block, cudaStream_t stream)
{
    (void)warps_per_block;
    bool signals = false;  // the proxy's ledger backlog or polled occupancy in some constant set
    for (int i = 0; i < p.n_sets; ++i) signals = signals || p.sets[i].proxy != 0 || p.sets[i].poll_us > 0;
    const cudaError_t e = p.pre_batch > 0 ? launch_mode<2>(p, blocks, stream)
                          : signals       ? launch_mode<1>(p, blocks, stream)
                                          : launch_mode<0>(p, blocks, stream);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

cudaError_t launch_hash(const SimParams& p, const uint64_t* kmix, int blocks, cudaStream_t stream)
{
    if (p.n_rows == 0) return cudaSuccess;
    const int64_t hb = p.n_rows < (int64_t)blocks * 8 ? p.n_rows : (int64_t)blocks * 8;
    hash_kernel<<<(unsigned)hb, kHashThreads, 0, stream>>>(p, kmix);
    return cudaGetLastError();
}

}  // namespace ctr
