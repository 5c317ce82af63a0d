// goodput.cu -- SLO goodput inputs per simulated row (ctr_goodput):
// the count of requests meeting both SLOs of their class (sec. IV-B targets,
// Table 2 goodput) and the exact nearest-rank P99 TTFT (Table 2 column).
//
// One 512-thread block per row (two blocks per SM at 64 registers a
// thread).  Pass 0 reads the row once and reduces the met count and the TTFT
// range; the P99 is then selected exactly by a radix select over
// (TTFT - min) with 11-bit digits, most significant first, each pass
// histogramming the candidates that still match the digits chosen so far
// (2048 shared-memory bins).  When the row fits (kStage), pass 0 also keeps
// its TTFTs in shared memory as 32-bit values and the select passes read them
// there, so a row crosses HBM once; a row with a TTFT outside [0, 2^32) or too
// many requests re-reads its TTFTs from global memory instead.  Called from
// ctr_simulate with kHash, pass 0 also sums the row checksum's first-token and
// completion terms, so the outputs are read once for both.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

constexpr int kThreads = 512;
constexpr int kDigit = 11;
constexpr int kBins = 1 << kDigit;

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

template <bool kStage, bool kHash>
__global__ void __launch_bounds__(kThreads, 2) goodput_kernel(const GoodputParams P)
{
    __shared__ uint32_t hist[kBins];
    __shared__ int64_t red64[kThreads / 32];
    __shared__ uint32_t pick[2];
    extern __shared__ uint32_t ttft_s[];  // kStage: the row's TTFTs
    const int tid = threadIdx.x;
    const int64_t n = P.n_req;

    for (int64_t row = blockIdx.x; row < P.n_rows; row += gridDim.x) {
        const int64_t tb = (row / P.rows_per_replica) * n;
        const int64_t ob = row * n;
        int64_t met = 0, mn = INT64_MAX, mx = INT64_MIN;
        uint64_t h = 0;  // kHash: the row's first-token and completion checksum terms
        // 2 elements per thread per round, all loads issued before any is used (the pass is latency-bound;
        // more elements in flight spill at 64 registers and lose more than they hide)
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
                    const bool ok = ttft <= P.ttft[c] && (o == 1 || td[u] - tf[u] <= P.tpot[c] * (o - 1));
                    met += ok;
                    mn = ttft < mn ? ttft : mn;
                    mx = ttft > mx ? ttft : mx;
                    if (kStage) ttft_s[k] = (uint32_t)ttft;
                    if (kHash) h += hterm(k, 2, (uint64_t)tf[u]) + hterm(k, 3, (uint64_t)td[u]);
                }
            }
        }
        met = block_reduce<int64_t>(met, 0, [](int64_t a, int64_t b) { return a + b; }, red64);
        mn = block_reduce<int64_t>(mn, INT64_MAX, [](int64_t a, int64_t b) { return a < b ? a : b; }, red64);
        mx = block_reduce<int64_t>(mx, INT64_MIN, [](int64_t a, int64_t b) { return a > b ? a : b; }, red64);
        if (kHash) {
            h = (uint64_t)block_reduce<int64_t>((int64_t)h, 0, [](int64_t a, int64_t b) {
                return (int64_t)((uint64_t)a + (uint64_t)b);  // sum mod 2^64
            }, red64);
            if (tid == 0 && P.row_status[row] == CTR_OK) P.row_hash[row] += h;  // a failed row keeps 0
        }
        if (n == 0) {
            if (tid == 0) {
                P.met[row] = 0;
                P.p99[row] = -1;
            }
            continue;
        }
        // the staged 32-bit copies are exact when every TTFT lies in [0, 2^32)
        const bool staged = kStage && mn >= 0 && mx < (int64_t(1) << 32);
        const uint64_t range = (uint64_t)mx - (uint64_t)mn;
        int shift = range == 0 ? 0 : 64 - __clzll((long long)range);  // bits still undetermined
        uint64_t prefix = 0;                                            // chosen high bits of (ttft - mn)
        int64_t rank = (99 * n + 99) / 100 - 1;                         // 0-based rank among the candidates
        while (shift > 0) {
            const int dbits = shift < kDigit ? shift : kDigit;
            const int above = shift;  // candidates agree with prefix on bits >= above
            shift -= dbits;
            for (int i = tid; i < kBins; i += kThreads) hist[i] = 0;
            __syncthreads();
            const uint32_t dmask = (1u << dbits) - 1u;
            for (int64_t k = tid; k < n; k += kThreads) {
                const uint64_t v = (staged ? (uint64_t)ttft_s[k] : (uint64_t)(P.t_first[ob + k] - P.trace.arrival_us[tb + k])) -
                                   (uint64_t)mn;
                const bool match = above >= 64 || (v >> above) == (prefix >> above);
                if (match) atomicAdd(&hist[(uint32_t)(v >> shift) & dmask], 1u);
            }
            __syncthreads();
            if (tid < 32) {  // find the bin holding the rank: per-lane sums, then a scan
                const int per = kBins / 32;
                uint32_t sum = 0;
                for (int i = 0; i < per; ++i) sum += hist[tid * per + i];
                uint32_t incl = sum;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const uint32_t v = __shfl_up_sync(0xffffffffu, incl, off);
                    if (tid >= off) incl += v;
                }
                const uint32_t excl = incl - sum;
                const bool mine = (int64_t)excl <= rank && rank < (int64_t)incl;
                const uint32_t ball = __ballot_sync(0xffffffffu, mine);
                const int owner = __ffs(ball) - 1;
                if (tid == owner) {
                    uint32_t acc = excl;
                    int bin = tid * per;
                    for (int i = 0; i < per; ++i) {
                        const uint32_t hcount = hist[tid * per + i];
                        if ((int64_t)(acc + hcount) > rank) {
                            bin = tid * per + i;
                            break;
                        }
                        acc += hcount;
                    }
                    pick[0] = (uint32_t)bin;
                    pick[1] = acc;
                }
            }
            __syncthreads();
            prefix |= (uint64_t)pick[0] << shift;
            rank -= pick[1];
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
    constexpr int64_t kStageMaxBytes = 160 * 1024;  // a row's TTFTs staged in shared memory up to this
    const int64_t stage_bytes = p.n_req * 4;
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
