// trace.cu -- synthetic request trace on the GPU (ctr_gen_trace).
//
// One warp per replica; lane l owns request base + l of each 32-request
// chunk.  Per request: two Philox4x32-10 blocks (Salmon et al., SC'11),
// rounded lognormal prompt / output lengths (Table 1 profiles), a predicted
// output length with multiplicative lognormal noise (sec. III-C, sec. V-G),
// an SLO class, and an integer unit-rate exponential gap.  A warp-wide int64
// inclusive scan turns gaps into cumulative work; Poisson arrivals divide by
// the rate, MMPP arrivals walk the state intervals cooperatively.
//
// Bit-identity with the CPU reference construction rests on doing only IEEE
// basic operations in a fixed order, in fp32 (the precision the integer
// lengths and gaps are defined in; GB300's fp64 rate would bound the kernel):
// every operation below is an explicit round-to-nearest intrinsic (no
// contraction into FMA; the file is also compiled with -fmad=false), and
// log / exp / the normal quantile are written here from their published
// methods rather than taken from CUDA's math library.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

using U32x4 = Philox4;
__device__ __forceinline__ U32x4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                        uint32_t k1)
{
    return philox4x32_10(c0, c1, c2, c3, k0, k1);
}

// ------------------------------------------------------------- fp32 helpers
__device__ __forceinline__ float add(float a, float b) { return __fadd_rn(a, b); }
__device__ __forceinline__ float sub(float a, float b) { return __fsub_rn(a, b); }
__device__ __forceinline__ float mul(float a, float b) { return __fmul_rn(a, b); }
__device__ __forceinline__ float dvd(float a, float b) { return __fdiv_rn(a, b); }

// Integer <-> float conversions without the 64-bit conversion instructions
// (GB300 runs those on its narrow fp64 pipe).  rn_u33(n): n < 2^33 rounded
// once to fp32 -- the exact sum of two exactly representable parts, rounded by
// one fp32 addition; trunc_pos(v): the integer part of a non-negative finite
// float below 2^63, read off its exponent and mantissa.
__device__ __forceinline__ float rn_u33(uint64_t n)
{
    const float hi = __uint2float_rn((uint32_t)(n >> 9));   // < 2^24: exact
    const float lo = __uint2float_rn((uint32_t)(n & 511u));  // exact
    return add(mul(hi, 512.0f), lo);
}

__device__ __forceinline__ int64_t trunc_pos(float v)
{
    const uint32_t b = __float_as_uint(v);
    const int e = (int)((b >> 23) & 0xffu) - 127;  // -0.0 (from ln 1) has e < 0 and gives 0
    if (e < 0) return 0;
    const uint64_t mant = (uint64_t)((b & 0x007FFFFFu) | 0x00800000u);
    return (int64_t)(e >= 23 ? mant << (e - 23) : mant >> (23 - e));
}

// (u + 1/2) 2^-32 rounded once to fp32; 1 - U is the same of ~u
__device__ __forceinline__ float u01(uint32_t u)
{
    return mul(rn_u33(2ull * u + 1ull), 0x1p-33f);
}

// Natural log of a positive normal x: x = m 2^e with m in (sqrt(1/2), sqrt(2)],
// s = (m - 1)/(m + 1), ln m = 2 s sum_{i=0..5} s^(2i) / (2i + 1) by Horner,
// ln x = e * ln2_hi + (e * ln2_lo + ln m)  (ln2_hi has 16 significant bits).
__device__ float det_logf(float x)
{
    const float inv_odd[6] = {0x1p+0f, 0x1.555556p-2f, 0x1.99999ap-3f, 0x1.24924ap-3f, 0x1.c71c72p-4f, 0x1.745d18p-4f};
    const uint32_t bits = __float_as_uint(x);
    int e = (int)((bits >> 23) & 0xffu) - 127;
    float m = __uint_as_float((bits & 0x007FFFFFu) | 0x3F800000u);
    if (m > 0x1.6a09e6p+0f) {
        m = mul(m, 0.5f);
        e += 1;
    }
    const float f = sub(m, 1.0f);
    const float s = dvd(f, add(m, 1.0f));
    const float z = mul(s, s);
    float acc = inv_odd[5];
#pragma unroll
    for (int i = 4; i >= 0; --i) acc = add(mul(acc, z), inv_odd[i]);
    const float ln_m = mul(add(s, s), acc);
    const float ed = __int2float_rn(e);
    return add(mul(ed, 0x1.62e4p-1f), add(mul(ed, 0x1.7f7d1cp-20f), ln_m));
}

// exp: k = nearest integer to x / ln2 (halves away from zero),
// r = (x - k ln2_hi) - k ln2_lo, e^r by its degree-7 Taylor polynomial, times
// 2^k through the exponent field.  x is clamped to [-87, 88].
__device__ float det_expf(float x)
{
    const float inv_fact[8] = {0x1p+0f, 0x1p+0f, 0x1p-1f, 0x1.555556p-3f, 0x1.555556p-5f, 0x1.111112p-7f,
                               0x1.6c16c2p-10f, 0x1.a01a02p-13f};
    if (x > 88.0f) x = 88.0f;
    if (x < -87.0f) x = -87.0f;
    const float kf = mul(x, 0x1.715476p+0f);
    const int k = __float2int_rz(kf >= 0.0f ? add(kf, 0.5f) : sub(kf, 0.5f));
    const float kd = __int2float_rn(k);
    const float r = sub(sub(x, mul(kd, 0x1.62e4p-1f)), mul(kd, 0x1.7f7d1cp-20f));
    float acc = inv_fact[7];
#pragma unroll
    for (int i = 6; i >= 0; --i) acc = add(mul(acc, r), inv_fact[i]);
    return mul(acc, __uint_as_float((uint32_t)(k + 127) << 23));
}

// Wichura (1988), algorithm AS241 PPND16 in fp32: rational approximations of
// degree 7 in r = 0.180625 - q^2 (|q| <= 0.425, q = U - 1/2) or in
// r = sqrt(-ln min(U, 1 - U)) shifted by 1.6 (r <= 5) or by 5.
__device__ __forceinline__ float poly7(const float* c, float r)
{
    float acc = c[7];
#pragma unroll
    for (int i = 6; i >= 0; --i) acc = add(mul(acc, r), c[i]);
    return acc;
}

__device__ float det_ndtrif(uint32_t u)
{
    const float a[8] = {0x1.b18d92p+1f, 0x1.0a4888p+7f, 0x1.ece5d2p+10f, 0x1.ad1d8cp+13f,
                        0x1.66c3e8p+15f, 0x1.06c1c6p+16f, 0x1.052d26p+15f, 0x1.39a296p+11f};
    const float b[8] = {0x1p+0f, 0x1.5281b4p+5f, 0x1.5797fp+9f, 0x1.512322p+12f,
                        0x1.4b772ep+14f, 0x1.3317cap+15f, 0x1.c0e458p+14f, 0x1.46a7ecp+12f};
    const float c[8] = {0x1.6c666p+0f, 0x1.285774p+2f, 0x1.713f72p+2f, 0x1.d2ecb2p+1f,
                        0x1.453ccp+0f, 0x1.ef2abcp-3f, 0x1.744eb6p-6f, 0x1.9615acp-11f};
    const float d[8] = {0x1p+0f, 0x1.06cefcp+1f, 0x1.ad278ep+0f, 0x1.61293p-1f,
                        0x1.2f5124p-3f, 0x1.f207a8p-7f, 0x1.1f18ccp-11f, 0x1.20d3f6p-30f};
    const float e[8] = {0x1.aa1b1cp+2f, 0x1.5daea6p+2f, 0x1.c8ea64p+0f, 0x1.2fad94p-2f,
                        0x1.b2b412p-6f, 0x1.45c19p-10f, 0x1.c6ec6cp-16f, 0x1.afb74ep-23f};
    const float f[8] = {0x1p+0f, 0x1.331d34p-1f, 0x1.186eb2p-3f, 0x1.e76f94p-7f,
                        0x1.9c8bcap-11f, 0x1.35c2c4p-16f, 0x1.31447p-23f, 0x1.269cp-49f};
    const long long twice = 2ll * (long long)u + 1ll - 4294967296ll;  // 2^33 (U - 1/2), odd, |twice| < 2^32
    const float mag = __uint2float_rn((uint32_t)(twice < 0 ? -twice : twice));
    const float q = mul(twice < 0 ? -mag : mag, 0x1p-33f);
    const float aq = q < 0.0f ? -q : q;
    if (aq <= 0x1.b33334p-2f) {
        const float r = sub(0x1.71eb86p-3f, mul(q, q));
        return dvd(mul(q, poly7(a, r)), poly7(b, r));
    }
    const float tail = twice < 0 ? u01(u) : u01(~u);
    float r = __fsqrt_rn(-det_logf(tail));
    float v;
    if (r <= 5.0f) {
        r = sub(r, 0x1.99999ap+0f);
        v = dvd(poly7(c, r), poly7(d, r));
    } else {
        r = sub(r, 5.0f);
        v = dvd(poly7(e, r), poly7(f, r));
    }
    return twice < 0 ? -v : v;
}

// clip(floor(v + 1/2), lo, hi) for v >= 0 (NaN / inf / huge -> hi); hi <= 2^20
__device__ __forceinline__ int64_t round_clip(float v, int64_t lo, int64_t hi)
{
    const float y = add(v, 0.5f);
    if (!(y < __int2float_rn((int)hi))) return hi;
    const int64_t t = __float2int_rz(y);
    return t < lo ? lo : t;
}

// floor(num / d) for num >= 0 with recip = floor((2^64 - 1) / d): the estimate is low by at most 2
__device__ __forceinline__ int64_t div_rate(int64_t num, int64_t d, uint64_t recip)
{
    uint64_t q = __umul64hi((uint64_t)num, recip);
    uint64_t r = (uint64_t)num - q * (uint64_t)d;
    if (r >= (uint64_t)d) {
        ++q;
        r -= (uint64_t)d;
    }
    if (r >= (uint64_t)d) ++q;
    return (int64_t)q;
}

__device__ __forceinline__ int64_t dwell(const TraceParams& P, uint32_t k0, uint32_t k1, uint32_t sub_id,
                                         int64_t j)
{
    const U32x4 x = philox((uint32_t)j, sub_id, 1u, 0u, k0, k1);
    const float g = det_logf(u01(x.v[0]));
    return trunc_pos(mul(-g, P.dwell_mean_f));
}

__global__ void __launch_bounds__(256) trace_kernel(const TraceParams P)
{
    const int lane = threadIdx.x & 31;
    const int64_t warp = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int64_t n_warps = (int64_t)gridDim.x * (blockDim.x >> 5);
    for (int64_t r = warp; r < P.n_replicas; r += n_warps) {
        const int64_t g = P.replica_offset + r;
        const uint64_t seed = P.seed + (uint64_t)(g % P.n_seeds);
        const uint32_t k0 = (uint32_t)seed, k1 = (uint32_t)(seed >> 32);
        const uint32_t sub_id = (uint32_t)(g / P.n_seeds);
        const int64_t row = r * P.n_req;

        int64_t carry = 0;  // cumulative unit-rate work before this chunk (nano-events)
        // MMPP interval j: [T, T + D) over which cumulative work runs from A to A_next
        int64_t j = 0, T = 0, A = 0, D = 0, A_next = 0;
        if (P.arrival_kind == 1) {
            D = dwell(P, k0, k1, sub_id, 0);
            A_next = A + P.rate[0] * D;
        }
        for (int64_t base = 0; base < P.n_req; base += 32) {
            const int64_t k = base + lane;
            const bool live = k < P.n_req;
            int64_t p = 0, o = 0, oh = 0, c = 0, gap = 0;
            if (live) {
                const U32x4 x = philox((uint32_t)k, sub_id, 0u, 0u, k0, k1);
                const U32x4 y = philox((uint32_t)k, sub_id, 0u, 1u, k0, k1);
                const float zp = det_ndtrif(x.v[0]);
                p = round_clip(det_expf(add(P.prompt_mu, mul(P.prompt_sigma, zp))), P.prompt_min, P.prompt_max);
                const bool is_short = (uint64_t)x.v[1] < P.mix_short_thr;
                const float mu = is_short ? P.short_mu : P.long_mu;
                const float sg = is_short ? P.short_sigma : P.long_sigma;
                const float zo = det_ndtrif(x.v[2]);
                o = round_clip(det_expf(add(mu, mul(sg, zo))), P.out_min, P.out_max);
                const float zn = det_ndtrif(x.v[3]);
                oh = round_clip(mul(__int2float_rn((int)o), det_expf(mul(P.noise_sigma, zn))), P.pred_min, P.pred_max);
                while (c < P.n_classes - 1 && (uint64_t)y.v[0] >= P.class_thr[c]) ++c;
                gap = trunc_pos(mul(-det_logf(u01(y.v[1])), 0x1.dcd65p+29f));
            }
            // inclusive warp scan of the gaps (integers: exact in any order)
            int64_t lam = gap;
#pragma unroll
            for (int off = 1; off < 32; off <<= 1) {
                const int64_t v = __shfl_up_sync(0xffffffffu, lam, off);
                if (lane >= off) lam += v;
            }
            lam += carry;
            carry = __shfl_sync(0xffffffffu, lam, 31);

            int64_t t = 0;
            if (P.arrival_kind == 0) {
                t = div_rate(lam, P.rate[0], P.rate_recip[0]);
            } else {
                // walk the intervals until every live lane found the last j with A_j <= lam
                bool done = !live;
                for (;;) {
                    if (!done && lam < A_next) {
                        t = T + div_rate(lam - A, P.rate[j & 1], P.rate_recip[j & 1]);
                        done = true;
                    }
                    if (__all_sync(0xffffffffu, done)) break;
                    T += D;
                    A = A_next;
                    j += 1;
                    D = dwell(P, k0, k1, sub_id, j);
                    A_next = A + P.rate[j & 1] * D;
                }
            }
            if (live) {
                P.out.arrival_us[row + k] = t;
                P.out.prompt_len[row + k] = (int32_t)p;
                P.out.true_out[row + k] = (int32_t)o;
                P.out.pred_out[row + k] = (int32_t)oh;
                P.out.slo_class[row + k] = (uint8_t)c;
            }
        }
    }
}

}  // namespace

cudaError_t launch_trace(const TraceParams& p, cudaStream_t stream)
{
    if (p.n_replicas == 0 || p.n_req == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err != cudaSuccess) return err;
    // small blocks spread one warp per replica evenly over the SMs (the kernel is
    // issue-bound, so the SM holding the most warps sets its time)
    const int warps_per_block = 4;
    int64_t blocks = (p.n_replicas + warps_per_block - 1) / warps_per_block;
    const int64_t cap = (int64_t)sms * 16;
    if (blocks > cap) blocks = cap;
    trace_kernel<<<(unsigned)blocks, warps_per_block * 32, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace ctr
