// goodput.cu -- SLO goodput inputs per simulated row (ctr_goodput):
// the count of requests meeting both SLOs of their class (sec. IV-B targets,
// Table 2 goodput), the exact nearest-rank P99 TTFT and, on request, the
// exact nearest-rank P99 TPOT (Table 2 columns; tpot_kernel at the end).
//
// One block per unit of up to kRows rows of one replica, which share the
// replica's trace and request indices.  Pass 0 reads the unit once: per
// request the trace's arrival, output length and class, then each row's
// t_first and t_done; per row the met count and, when the rows fit in shared
// memory (kStage) and every TTFT lies in [0, 2^32), a histogram of the TTFTs
// over logarithmic bins (64 per octave, monotone in the TTFT) with each
// request's bin kept in shared memory.  For each row a block scan then finds
// the bin holding the P99's rank; the requests of that bin (a few dozen in
// practice) are gathered, their exact TTFTs read back, and the value of the
// remaining rank among them counted out exactly.  A row with a TTFT outside
// [0, 2^32), more than kCand requests in the P99's bin, or too many requests
// to stage falls back to a radix select over the exact TTFTs read from global
// memory (11-bit digits, most significant first).  Called from ctr_simulate
// with kHash, pass 0 also sums each row's checksum terms of first-token and
// completion times; the request-only half of those terms is read from the
// call's table (launch_mix_table) when ctr_simulate has one, else mixed once
// per request for the unit's rows.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

constexpr int kThreads = 512;
constexpr int kLogBins = 2112;  // bin 0: a TTFT of 0; then 64 per octave of [1, 2^32)
constexpr int kCand = 512;      // requests of the P99's bin selected exactly in shared memory
constexpr int kDigit = 11;      // radix select fallback
constexpr int kBins = 1 << kDigit;
static_assert(kBins <= kLogBins, "the radix fallback reuses the histogram");

// Monotone bin of a TTFT in [0, 2^32): the exponent and the top 6 mantissa bits
// of its fp32 value rounded toward zero (exact integer to float conversion
// order is kept by round-toward-zero, so x <= y gives bin(x) <= bin(y)).
__device__ __forceinline__ uint32_t log_bin(uint32_t x)
{
    return x == 0 ? 0u : (__float_as_uint(__uint2float_rz(x)) >> 17) - (126u << 6);
}

template <typename T, typename Op>
__device__ T block_reduce(T v, T identity, Op op, T* scratch)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, off));
    if (lane == 0) scratch[wid] = v;
    __syncthreads();
    if (wid == 0) {
        v = lane < kThreads / 32 ? scratch[lane] : identity;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v = op(v, __shfl_xor_sync(0xffffffffu, v, off));
        if (lane == 0) scratch[0] = v;
    }
    __syncthreads();
    const T r = scratch[0];
    __syncthreads();
    return r;
}

// The bin of hist[0 .. nb) holding 0-based rank `rank`, and the count of the
// bins before it, to every thread: each thread sums a contiguous run of bins, a
// block scan of the sums finds the run, its thread walks it.
__device__ void find_rank_bin(const uint32_t* hist, int nb, int64_t rank, uint32_t* pick, uint32_t* wsum)
{
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int per = (nb + kThreads - 1) / kThreads;
    const int b0 = tid * per, b1 = b0 + per < nb ? b0 + per : nb;
    uint32_t sum = 0;
    for (int b = b0; b < b1; ++b) sum += hist[b];
    uint32_t incl = sum;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
        const uint32_t v = __shfl_up_sync(0xffffffffu, incl, off);
        if (lane >= off) incl += v;
    }
    if (lane == 31) wsum[wid] = incl;
    __syncthreads();
    uint32_t before = 0;
    for (int w = 0; w < wid; ++w) before += wsum[w];
    const uint32_t excl = before + incl - sum;
    if ((int64_t)excl <= rank && rank < (int64_t)(excl + sum)) {  // exactly one thread
        uint32_t acc = excl;
        int bin = b0;
        for (int b = b0; b < b1; ++b) {
            if ((int64_t)(acc + hist[b]) > rank) {
                bin = b;
                break;
            }
            acc += hist[b];
        }
        pick[0] = (uint32_t)bin;
        pick[1] = acc;
    }
    __syncthreads();
}


// Shared scratch of the per-row selection.
struct SelScratch {
    int64_t red64[kThreads / 32];
    uint32_t wsum[kThreads / 32];
    uint32_t pick[2];
    uint32_t n_cand;
    int32_t cand_k[kCand];
    int64_t cand_v[kCand];
};

// One row's P99 TTFT (and its met count, already reduced) into P.p99 / P.met:
// from its histogram and staged bins when `staged`, else by the radix select
// over the TTFTs in global memory (which reuses `hist`).  Block-collective.
#if CTR_BOUNDS_CHECK
#define CTR_CK_FLAG_PARAM , bool& bad
#define CTR_CK_FLAG_ARG , bad
#else  // the plain build's function keeps its plain signature
#define CTR_CK_FLAG_PARAM
#define CTR_CK_FLAG_ARG
#endif
__device__ void select_row(const GoodputParams& P, int64_t row, int64_t tb, int64_t n, int32_t met, bool staged,
                           uint32_t* hist, const uint16_t* bins, SelScratch& S CTR_CK_FLAG_PARAM)
{
#if !CTR_BOUNDS_CHECK
    bool bad = false;  // dead: the accessors below compile to plain accesses
#endif
    const int64_t trace_len = (P.n_rows / P.rows_per_replica) * n, out_len = P.n_rows * n;
    const int tid = threadIdx.x;
    const int64_t ob = row * n;
    const int64_t rank = (99 * n + 99) / 100 - 1;  // 0-based nearest rank
    if (staged) {
        if (tid == 0) S.n_cand = 0;
        find_rank_bin(hist, kLogBins, rank, S.pick, S.wsum);  // its barriers also publish n_cand
        const uint32_t B = S.pick[0];
        const int64_t r_in = rank - (int64_t)S.pick[1];  // rank among the bin's requests
        for (int64_t k = tid; k < n; k += kThreads) {
            if (ck_ld(bins, k, n, bad) == B) {
                const uint32_t i = atomicAdd(&S.n_cand, 1u);
                if (i < (uint32_t)kCand) S.cand_k[i] = (int32_t)k;
            }
        }
        __syncthreads();
        const int c = (int)S.n_cand;
        if (c <= kCand) {
            for (int i = tid; i < c; i += kThreads) {
                const int64_t k = S.cand_k[i];
                S.cand_v[i] = ck_ld(P.t_first, ob + k, out_len, bad) - ck_ld(P.trace.arrival_us, tb + k, trace_len, bad);
            }
            __syncthreads();
            // the candidate whose position in (value, slot) order is the remaining rank
            for (int i = tid; i < c; i += kThreads) {
                const int64_t v = S.cand_v[i];
                int64_t pos = 0;
                for (int j = 0; j < c; ++j) {
                    const int64_t w = S.cand_v[j];
                    pos += w < v || (w == v && j < i);
                }
                if (pos == r_in) P.p99[row] = v;
            }
            if (tid == 0) P.met[row] = met;
            __syncthreads();
            return;
        }
    }
    // ---- fallback: exact radix select over (TTFT - min) read from global memory
    int64_t mn = INT64_MAX, mx = INT64_MIN;
    for (int64_t k = tid; k < n; k += kThreads) {
        const int64_t t = ck_ld(P.t_first, ob + k, out_len, bad) - ck_ld(P.trace.arrival_us, tb + k, trace_len, bad);
        mn = t < mn ? t : mn;
        mx = t > mx ? t : mx;
    }
    mn = block_reduce<int64_t>(mn, INT64_MAX, [](int64_t a, int64_t b) { return a < b ? a : b; }, S.red64);
    mx = block_reduce<int64_t>(mx, INT64_MIN, [](int64_t a, int64_t b) { return a > b ? a : b; }, S.red64);
    const uint64_t range = (uint64_t)mx - (uint64_t)mn;
    int shift = range == 0 ? 0 : 64 - __clzll((long long)range);  // bits still undetermined
    uint64_t prefix = 0;                                            // chosen high bits of (ttft - mn)
    int64_t rk = rank;                                              // rank among the candidates
    while (shift > 0) {
        const int dbits = shift < kDigit ? shift : kDigit;
        const int above = shift;  // candidates agree with prefix on bits >= above
        shift -= dbits;
        for (int i = tid; i < kBins; i += kThreads) hist[i] = 0;
        __syncthreads();
        const uint32_t dmask = (1u << dbits) - 1u;
        for (int64_t k = tid; k < n; k += kThreads) {
            const uint64_t v = (uint64_t)(ck_ld(P.t_first, ob + k, out_len, bad) -
                                          ck_ld(P.trace.arrival_us, tb + k, trace_len, bad)) - (uint64_t)mn;
            const bool match = above >= 64 || (v >> above) == (prefix >> above);
            if (match) {
                const uint32_t b = (uint32_t)(v >> shift) & dmask;
                if (ck_ok(b, kBins, bad)) atomicAdd(&hist[b], 1u);
            }
        }
        __syncthreads();
        find_rank_bin(hist, kBins, rk, S.pick, S.wsum);
        prefix |= (uint64_t)S.pick[0] << shift;
        rk -= S.pick[1];
        __syncthreads();
    }
    if (tid == 0) {
        P.met[row] = met;
        P.p99[row] = (int64_t)((uint64_t)mn + prefix);
    }
    __syncthreads();
}

template <int kRows, bool kStage, bool kHash>
__global__ void __launch_bounds__(kThreads, 2) goodput_kernel(const GoodputParams P)
{
    __shared__ uint32_t hist[kRows][kLogBins];
    __shared__ SelScratch S;
    extern __shared__ uint16_t bin_s[];  // kStage: each row's TTFT bins, [kRows][n]
    const int tid = threadIdx.x;
    const int64_t n = P.n_req;
    const int64_t rpr = P.rows_per_replica;
    const int64_t upr = (rpr + kRows - 1) / kRows;  // units per replica
    const int64_t n_units = (P.n_rows / rpr) * upr;
    const int64_t trace_len = (P.n_rows / rpr) * n, out_len = P.n_rows * n;  // entries of the trace and outputs

    for (int64_t unit = blockIdx.x; unit < n_units; unit += gridDim.x) {
        const int64_t rep = unit / upr;
        const int64_t j0 = (unit - rep * upr) * kRows;
        const int nr = (int)(rpr - j0 < kRows ? rpr - j0 : kRows);  // rows of this unit
        const int64_t row0 = rep * rpr + j0;
        const int64_t tb = rep * n;
        if (kStage) {
            for (int i = tid; i < kRows * kLogBins; i += kThreads) (&hist[0][0])[i] = 0;
            __syncthreads();
        }
        int32_t met[kRows];
        uint64_t h[kRows];  // kHash: each row's first-token and completion checksum terms
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            met[r] = 0;
            h[r] = 0;
        }
        uint32_t wide = 0;  // bit r: row r has a TTFT outside [0, 2^32)
        bool bad = false;   // bounds-checked builds: an index of this thread fell outside its buffer
        for (int64_t k = tid; k < n; k += kThreads) {
            // every load of the request issued before any is used
            const int64_t ta = ck_ldg(P.trace.arrival_us, tb + k, trace_len, bad);
            const int64_t o = ck_ldg(P.trace.true_out, tb + k, trace_len, bad);
            int c = (int)ck_ldg(P.trace.slo_class, tb + k, trace_len, bad);
            int64_t tf[kRows], td[kRows];
#pragma unroll
            for (int r = 0; r < kRows; ++r) {
                if (r < nr) {
                    tf[r] = ck_ldg(P.t_first, (row0 + r) * n + k, out_len, bad);
                    td[r] = ck_ldg(P.t_done, (row0 + r) * n + k, out_len, bad);
                }
            }
            if (c >= P.n_classes) c = P.n_classes - 1;
            const int64_t ttft_slo = P.ttft[c], tpot_slo = P.tpot[c] * (o - 1);
            uint64_t m2 = 0, m3 = 0;  // the request-only halves of the checksum terms
            if (kHash) {
                if (P.kmix) {  // mixed once per call (launch_mix_table)
                    m2 = ck_ldg(P.kmix, k, 2 * n, bad);
                    m3 = ck_ldg(P.kmix, n + k, 2 * n, bad);
                } else {
                    m2 = mix64((uint64_t(2) << 56) ^ (uint64_t)k);
                    m3 = mix64((uint64_t(3) << 56) ^ (uint64_t)k);
                }
            }
#pragma unroll
            for (int r = 0; r < kRows; ++r) {
                if (r < nr) {
                    const int64_t ttft = tf[r] - ta;
                    met[r] += ttft <= ttft_slo && (o == 1 || td[r] - tf[r] <= tpot_slo);
                    const bool fits = (uint64_t)ttft < (uint64_t(1) << 32);
                    wide |= (uint32_t)!fits << r;
                    if (kStage) {
                        const uint32_t b = fits ? log_bin((uint32_t)ttft) : 0u;
                        if (ck_ok(b, kLogBins, bad)) atomicAdd(&hist[r][b], 1u);
                        ck_st(bin_s, (int64_t)r * n + k, (int64_t)kRows * n, (uint16_t)b, bad);
                    }
                    if (kHash) h[r] += mix64(m2 ^ (uint64_t)tf[r]) + mix64(m3 ^ (uint64_t)td[r]);
                }
            }
        }
        wide = (uint32_t)block_reduce<int32_t>((int32_t)wide, 0, [](int32_t a, int32_t b) { return a | b; },
                                               reinterpret_cast<int32_t*>(S.red64));
#pragma unroll
        for (int r = 0; r < kRows; ++r) {
            if (r < nr) {
                const int32_t m_r = block_reduce<int32_t>(met[r], 0, [](int32_t a, int32_t b) { return a + b; },
                                                          reinterpret_cast<int32_t*>(S.red64));
                const int64_t row = row0 + r;
                if (kHash) {
                    const uint64_t h_r = (uint64_t)block_reduce<int64_t>((int64_t)h[r], 0, [](int64_t a, int64_t b) {
                        return (int64_t)((uint64_t)a + (uint64_t)b);  // sum mod 2^64
                    }, S.red64);
                    if (tid == 0 && P.row_status[row] == CTR_OK) P.row_hash[row] += h_r;  // a failed row keeps 0
                }
                if (n == 0) {
                    if (tid == 0) {
                        P.met[row] = 0;
                        P.p99[row] = -1;
                    }
                    continue;
                }
                select_row(P, row, tb, n, m_r, kStage && !((wide >> r) & 1u), hist[r], bin_s + (int64_t)r * n,
                           S CTR_CK_FLAG_ARG);
#if CTR_BOUNDS_CHECK
                if (__syncthreads_or(bad) && tid == 0) {  // a row whose pass left a buffer: both outputs say so
                    P.met[row] = CTR_EBOUNDS;
                    P.p99[row] = CTR_EBOUNDS;
                }
#endif
            }
        }
    }
}

// P99 TPOT per row (Table 2): one block per row, each thread taking two
// requests per pass with all their loads issued first.  A request with o >= 2
// output tokens has TPOT = (t_done - t_first) / (o - 1) rounded toward zero
// (the floor, as t_done >= t_first); one-token requests have none.  Pass 1
// counts the row's M such requests and histograms their TPOTs over the same
// logarithmic bins as the TTFTs (32-bit quotients when the decode time is
// below 2^32 us); a block scan finds the bin of the nearest rank
// ceil(0.99 M) - 1; pass 2 gathers that bin's TPOTs and counts the remaining
// rank out exactly.  A decode time outside [0, 2^32) or more than kCand
// requests in the bin fall back to an exact radix select (11-bit digits) over
// the 64-bit quotients.
__device__ __forceinline__ bool tpot_of(const GoodputParams& P, int64_t tb, int64_t ob, int64_t k, int64_t& v)
{
    const int32_t o = __ldg(&P.trace.true_out[tb + k]);
    if (o < 2) return false;
    v = (__ldg(&P.t_done[ob + k]) - __ldg(&P.t_first[ob + k])) / (int64_t)(o - 1);
    return true;
}
// the same for a row whose decode times all lie in [0, 2^32): one 32-bit quotient
__device__ __forceinline__ bool tpot32_of(const GoodputParams& P, int64_t tb, int64_t ob, int64_t k, uint32_t& v)
{
    const int32_t o = __ldg(&P.trace.true_out[tb + k]);
    if (o < 2) return false;
    v = (uint32_t)(__ldg(&P.t_done[ob + k]) - __ldg(&P.t_first[ob + k])) / (uint32_t)(o - 1);
    return true;
}

__global__ void __launch_bounds__(kThreads, 2) tpot_kernel(const GoodputParams P, int64_t* p99_tpot)
{
    __shared__ uint32_t hist[kLogBins];
    __shared__ SelScratch S;
    const int tid = threadIdx.x;
    const int64_t n = P.n_req;
    for (int64_t row = blockIdx.x; row < P.n_rows; row += gridDim.x) {
        const int64_t tb = (row / P.rows_per_replica) * n, ob = row * n;
        for (int i = tid; i < kLogBins; i += kThreads) hist[i] = 0;
        __syncthreads();
        int32_t m = 0;
        int32_t wide = 0;  // a decode time outside [0, 2^32)
        for (int64_t k0 = tid; k0 < n; k0 += 2 * kThreads) {  // two requests per thread, loads first
            int32_t o[2];
            int64_t d[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int64_t k = k0 + u * kThreads < n ? k0 + u * kThreads : k0;
                o[u] = __ldg(&P.trace.true_out[tb + k]);
                d[u] = __ldg(&P.t_done[ob + k]) - __ldg(&P.t_first[ob + k]);
            }
            if (k0 + kThreads >= n) o[1] = 0;  // past the end: no request
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                if (o[u] < 2) continue;
                m += 1;
                if ((uint64_t)d[u] < (uint64_t(1) << 32)) {
                    atomicAdd(&hist[log_bin((uint32_t)d[u] / (uint32_t)(o[u] - 1))], 1u);
                } else {
                    wide = 1;
                }
            }
        }
        const int32_t M = block_reduce<int32_t>(m, 0, [](int32_t a, int32_t b) { return a + b; },
                                                reinterpret_cast<int32_t*>(S.red64));
        wide = block_reduce<int32_t>(wide, 0, [](int32_t a, int32_t b) { return a | b; },
                                     reinterpret_cast<int32_t*>(S.red64));
        if (M == 0) {
            if (tid == 0) p99_tpot[row] = -1;
            continue;
        }
        const int64_t rank = (99 * (int64_t)M + 99) / 100 - 1;  // 0-based nearest rank among the M
        if (!wide) {
            if (tid == 0) S.n_cand = 0;
            find_rank_bin(hist, kLogBins, rank, S.pick, S.wsum);  // its barriers also publish n_cand
            const uint32_t B = S.pick[0];
            const int64_t r_in = rank - (int64_t)S.pick[1];
            for (int64_t k0 = tid; k0 < n; k0 += 2 * kThreads) {
                int32_t o[2];
                uint32_t d[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    const int64_t k = k0 + u * kThreads < n ? k0 + u * kThreads : k0;
                    o[u] = __ldg(&P.trace.true_out[tb + k]);
                    d[u] = (uint32_t)(__ldg(&P.t_done[ob + k]) - __ldg(&P.t_first[ob + k]));
                }
                if (k0 + kThreads >= n) o[1] = 0;
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    if (o[u] < 2) continue;
                    const uint32_t v = d[u] / (uint32_t)(o[u] - 1);
                    if (log_bin(v) == B) {
                        const uint32_t i = atomicAdd(&S.n_cand, 1u);
                        if (i < (uint32_t)kCand) S.cand_v[i] = (int64_t)v;
                    }
                }
            }
            __syncthreads();
            const int c = (int)S.n_cand;
            if (c <= kCand) {
                for (int i = tid; i < c; i += kThreads) {
                    const int64_t v = S.cand_v[i];
                    int64_t pos = 0;
                    for (int j = 0; j < c; ++j) {
                        const int64_t w = S.cand_v[j];
                        pos += w < v || (w == v && j < i);
                    }
                    if (pos == r_in) p99_tpot[row] = v;
                }
                __syncthreads();
                continue;
            }
        }
        // exact radix select over (TPOT - min) of the row's multi-token requests
        int64_t mn = INT64_MAX, mx = INT64_MIN;
        for (int64_t k = tid; k < n; k += kThreads) {
            int64_t v;
            if (tpot_of(P, tb, ob, k, v)) {
                mn = v < mn ? v : mn;
                mx = v > mx ? v : mx;
            }
        }
        mn = block_reduce<int64_t>(mn, INT64_MAX, [](int64_t a, int64_t b) { return a < b ? a : b; }, S.red64);
        mx = block_reduce<int64_t>(mx, INT64_MIN, [](int64_t a, int64_t b) { return a > b ? a : b; }, S.red64);
        const uint64_t range = (uint64_t)mx - (uint64_t)mn;
        int shift = range == 0 ? 0 : 64 - __clzll((long long)range);
        uint64_t prefix = 0;
        int64_t rk = rank;
        while (shift > 0) {
            const int dbits = shift < kDigit ? shift : kDigit;
            const int above = shift;
            shift -= dbits;
            for (int i = tid; i < kBins; i += kThreads) hist[i] = 0;
            __syncthreads();
            const uint32_t dmask = (1u << dbits) - 1u;
            for (int64_t k = tid; k < n; k += kThreads) {
                int64_t tv;
                if (!tpot_of(P, tb, ob, k, tv)) continue;
                const uint64_t v = (uint64_t)tv - (uint64_t)mn;
                if (above >= 64 || (v >> above) == (prefix >> above)) atomicAdd(&hist[(uint32_t)(v >> shift) & dmask], 1u);
            }
            __syncthreads();
            find_rank_bin(hist, kBins, rk, S.pick, S.wsum);
            prefix |= (uint64_t)S.pick[0] << shift;
            rk -= S.pick[1];
            __syncthreads();
        }
        if (tid == 0) p99_tpot[row] = (int64_t)((uint64_t)mn + prefix);
        __syncthreads();
    }
}

__global__ void __launch_bounds__(256) mix_table_kernel(uint64_t* t, int64_t n)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < 2 * n; i += (int64_t)gridDim.x * blockDim.x) {
        const bool first = i < n;
        const int64_t k = first ? i : i - n;
        t[i] = mix64(((first ? uint64_t(2) : uint64_t(3)) << 56) ^ (uint64_t)k);
    }
}

template <int kRows, bool kStage>
cudaError_t launch_rows(const GoodputParams& p, int64_t dyn_bytes, bool hash, int sms, cudaStream_t stream)
{
    const void* k = hash ? (const void*)goodput_kernel<kRows, kStage, true>
                         : (const void*)goodput_kernel<kRows, kStage, false>;
    cudaError_t err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)dyn_bytes);
    if (err != cudaSuccess) return err;
    int per_sm = 0;
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kThreads, (size_t)dyn_bytes);
    if (err != cudaSuccess) return err;
    const int64_t rpr = p.rows_per_replica;
    int64_t blocks = (p.n_rows / rpr) * ((rpr + kRows - 1) / kRows);
    const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
    if (blocks > cap) blocks = cap;
    if (hash)
        goodput_kernel<kRows, kStage, true><<<(unsigned)blocks, kThreads, (size_t)dyn_bytes, stream>>>(p);
    else
        goodput_kernel<kRows, kStage, false><<<(unsigned)blocks, kThreads, (size_t)dyn_bytes, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_tpot(const GoodputParams& p, int64_t* p99_tpot, cudaStream_t stream)
{
    if (p.n_rows == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    const int64_t blocks = p.n_rows < (int64_t)sms * 2 ? p.n_rows : (int64_t)sms * 2;
    tpot_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(p, p99_tpot);
    return cudaGetLastError();
}

cudaError_t launch_mix_table(uint64_t* t, int64_t n, cudaStream_t stream)
{
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (2 * n + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    mix_table_kernel<<<(unsigned)blocks, 256, 0, stream>>>(t, n);
    return cudaGetLastError();
}

cudaError_t launch_goodput(const GoodputParams& p, cudaStream_t stream)
{
    if (p.n_rows == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    // Two blocks per SM when a unit's staged bins, histograms and scratch fit in half the shared memory;
    // two rows per unit when the replica has them (they share the trace's reads and, without a table, the
    // request-only checksum mixes).
    constexpr int64_t kSmemBudget = 108 * 1024;
    const int64_t fixed = (int64_t)sizeof(SelScratch) + 256;
    const bool hash = p.row_hash != nullptr;
    const int64_t n2 = p.n_req * 2;
    auto fits = [&](int rows) { return n2 > 0 && rows * (n2 + 4 * kLogBins) + fixed <= kSmemBudget; };
    if (p.rows_per_replica >= 2 && fits(2)) return launch_rows<2, true>(p, 2 * n2, hash, sms, stream);
    if (fits(1)) return launch_rows<1, true>(p, n2, hash, sms, stream);
    constexpr int64_t kStageMaxBytes = 200 * 1024;  // one row staged, one block per SM
    if (n2 > 0 && n2 + 4 * kLogBins + fixed <= kStageMaxBytes) return launch_rows<1, true>(p, n2, hash, sms, stream);
    return launch_rows<1, false>(p, 0, hash, sms, stream);  // rows too long to stage
}

}  // namespace ctr
