// goodput.cu -- SLO goodput inputs per simulated row (ctr_goodput):
// the count of requests meeting both SLOs of their class (sec. IV-B targets,
// Table 2 goodput) and the exact nearest-rank P99 TTFT (Table 2 column).
//
// One block per row.  Pass 0 reads the row once: the met count, and, when the
// row fits in shared memory (kStage) and every TTFT lies in [0, 2^32), a
// histogram of the TTFTs over logarithmic bins (64 per octave, monotone in the
// TTFT) with each request's bin kept in shared memory.  A block scan finds the
// bin holding the P99's rank; the requests of that bin (a few dozen in
// practice) are gathered, their exact TTFTs read back, and the value of the
// remaining rank among them counted out exactly.  A row with too many requests,
// a TTFT outside [0, 2^32) or more than kCand requests in the P99's bin falls
// back to a radix select over the exact TTFTs read from global memory
// (11-bit digits, most significant first).  Called from ctr_simulate with
// kHash, pass 0 also sums the row checksum's first-token and completion terms,
// so the outputs are read once for both.
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

template <bool kStage, bool kHash>
__global__ void __launch_bounds__(kThreads, 2) goodput_kernel(const GoodputParams P)
{
    __shared__ uint32_t hist[kLogBins];
    __shared__ int64_t red64[kThreads / 32];
    __shared__ uint32_t wsum[kThreads / 32];
    __shared__ uint32_t pick[2];
    __shared__ uint32_t n_cand;
    __shared__ int32_t cand_k[kCand];
    __shared__ int64_t cand_v[kCand];
    extern __shared__ uint16_t bin_s[];  // kStage: each request's TTFT bin
    const int tid = threadIdx.x;
    const int64_t n = P.n_req;

    for (int64_t row = blockIdx.x; row < P.n_rows; row += gridDim.x) {
        const int64_t tb = (row / P.rows_per_replica) * n;
        const int64_t ob = row * n;
        if (kStage) {
            for (int i = tid; i < kLogBins; i += kThreads) hist[i] = 0;
            if (tid == 0) n_cand = 0;
            __syncthreads();
        }
        int32_t met = 0;
        bool wide = false;  // some TTFT outside [0, 2^32)
        uint64_t h = 0;     // kHash: the row's first-token and completion checksum terms
        // 2 elements per thread per round, all loads issued before any is used
        for (int64_t base = tid; base < n; base += (int64_t)kThreads * 2) {
            int64_t tf[2], td[2], ta[2];
            int32_t ov[2];
            uint32_t cv[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int64_t k = base + (int64_t)u * kThreads;
                if (k < n) {
                    tf[u] = __ldg(&P.t_first[ob + k]);
                    td[u] = __ldg(&P.t_done[ob + k]);
                    ta[u] = __ldg(&P.trace.arrival_us[tb + k]);
                    ov[u] = __ldg(&P.trace.true_out[tb + k]);
                    cv[u] = __ldg(&P.trace.slo_class[tb + k]);
                }
            }
#pragma unroll
            for (int u = 0; u < 2; ++u) {
                const int64_t k = base + (int64_t)u * kThreads;
                if (k < n) {
                    const int64_t ttft = tf[u] - ta[u];
                    const int64_t o = ov[u];
                    int c = (int)cv[u];
                    if (c >= P.n_classes) c = P.n_classes - 1;
                    met += ttft <= P.ttft[c] && (o == 1 || td[u] - tf[u] <= P.tpot[c] * (o - 1));
                    const bool fits = (uint64_t)ttft < (uint64_t(1) << 32);
                    wide |= !fits;
                    if (kStage) {
                        const uint32_t b = fits ? log_bin((uint32_t)ttft) : 0u;
                        atomicAdd(&hist[b], 1u);
                        bin_s[k] = (uint16_t)b;
                    }
                    if (kHash) h += hterm(k, 2, (uint64_t)tf[u]) + hterm(k, 3, (uint64_t)td[u]);
                }
            }
        }
        met = block_reduce<int32_t>(met, 0, [](int32_t a, int32_t b) { return a + b; },
                                    reinterpret_cast<int32_t*>(red64));
        if (kHash) {
            h = (uint64_t)block_reduce<int64_t>((int64_t)h, 0, [](int64_t a, int64_t b) {
                return (int64_t)((uint64_t)a + (uint64_t)b);  // sum mod 2^64
            }, red64);
            if (tid == 0 && P.row_status[row] == CTR_OK) P.row_hash[row] += h;  // a failed row keeps 0
        }
        wide = __syncthreads_or(wide) != 0;
        if (n == 0) {
            if (tid == 0) {
                P.met[row] = 0;
                P.p99[row] = -1;
            }
            continue;
        }
        const int64_t rank = (99 * n + 99) / 100 - 1;  // 0-based nearest rank
        if (kStage && !wide) {
            find_rank_bin(hist, kLogBins, rank, pick, wsum);
            const uint32_t B = pick[0];
            const int64_t r_in = rank - (int64_t)pick[1];  // rank among the bin's requests
            for (int64_t k = tid; k < n; k += kThreads) {
                if (bin_s[k] == B) {
                    const uint32_t i = atomicAdd(&n_cand, 1u);
                    if (i < (uint32_t)kCand) cand_k[i] = (int32_t)k;
                }
            }
            __syncthreads();
            const int c = (int)n_cand;
            if (c <= kCand) {
                for (int i = tid; i < c; i += kThreads) {
                    const int64_t k = cand_k[i];
                    cand_v[i] = P.t_first[ob + k] - P.trace.arrival_us[tb + k];
                }
                __syncthreads();
                // the candidate whose position in (value, slot) order is the remaining rank
                for (int i = tid; i < c; i += kThreads) {
                    const int64_t v = cand_v[i];
                    int64_t pos = 0;
                    for (int j = 0; j < c; ++j) {
                        const int64_t w = cand_v[j];
                        pos += w < v || (w == v && j < i);
                    }
                    if (pos == r_in) P.p99[row] = v;
                }
                if (tid == 0) P.met[row] = met;
                __syncthreads();
                continue;
            }
        }
        // ---- fallback: exact radix select over (TTFT - min) read from global memory
        int64_t mn = INT64_MAX, mx = INT64_MIN;
        for (int64_t k = tid; k < n; k += kThreads) {
            const int64_t t = P.t_first[ob + k] - P.trace.arrival_us[tb + k];
            mn = t < mn ? t : mn;
            mx = t > mx ? t : mx;
        }
        mn = block_reduce<int64_t>(mn, INT64_MAX, [](int64_t a, int64_t b) { return a < b ? a : b; }, red64);
        mx = block_reduce<int64_t>(mx, INT64_MIN, [](int64_t a, int64_t b) { return a > b ? a : b; }, red64);
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
                const uint64_t v = (uint64_t)(P.t_first[ob + k] - P.trace.arrival_us[tb + k]) - (uint64_t)mn;
                const bool match = above >= 64 || (v >> above) == (prefix >> above);
                if (match) atomicAdd(&hist[(uint32_t)(v >> shift) & dmask], 1u);
            }
            __syncthreads();
            find_rank_bin(hist, kBins, rk, pick, wsum);
            prefix |= (uint64_t)pick[0] << shift;
            rk -= pick[1];
            __syncthreads();
        }
        if (tid == 0) {
            P.met[row] = met;
            P.p99[row] = (int64_t)((uint64_t)mn + prefix);
        }
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_goodput(const GoodputParams& p, cudaStream_t stream)
{
    if (p.n_rows == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    constexpr int64_t kStageMaxBytes = 200 * 1024;  // a row's TTFT bins staged in shared memory up to this
    const int64_t stage_bytes = p.n_req * 2;
    const bool hash = p.row_hash != nullptr;
    if (stage_bytes > 0 && stage_bytes <= kStageMaxBytes) {
        const void* k = hash ? (const void*)goodput_kernel<true, true> : (const void*)goodput_kernel<true, false>;
        err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)stage_bytes);
        if (err != cudaSuccess) return err;
        int per_sm = 0;
        err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kThreads, (size_t)stage_bytes);
        if (err != cudaSuccess) return err;
        int64_t blocks = p.n_rows;
        const int64_t cap = (int64_t)sms * (per_sm > 0 ? per_sm : 1);
        if (blocks > cap) blocks = cap;
        if (hash)
            goodput_kernel<true, true><<<(unsigned)blocks, kThreads, (size_t)stage_bytes, stream>>>(p);
        else
            goodput_kernel<true, false><<<(unsigned)blocks, kThreads, (size_t)stage_bytes, stream>>>(p);
        return cudaGetLastError();
    }
    int64_t blocks = p.n_rows;
    if (blocks > (int64_t)sms * 8) blocks = (int64_t)sms * 8;
    if (hash)
        goodput_kernel<false, true><<<(unsigned)blocks, kThreads, 0, stream>>>(p);
    else
        goodput_kernel<false, false><<<(unsigned)blocks, kThreads, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace ctr
