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
// basic operations in a fixed order: every fp64 operation below is an
// explicit round-to-nearest intrinsic (no contraction into FMA; the file is
// also compiled with -fmad=false), and log / exp / the normal quantile are
// written here from their published methods rather than taken from CUDA's
// math library.
#include "ctr_internal.cuh"

namespace ctr {
namespace {

// ------------------------------------------------------------- Philox4x32-10
struct U32x4 {
    uint32_t v[4];
};

__device__ __forceinline__ U32x4 philox(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                        uint32_t k1)
{
#pragma unroll
    for (int round = 0; round < 10; ++round) {
        const uint32_t hi0 = __umulhi(0xD2511F53u, c0), lo0 = 0xD2511F53u * c0;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c2), lo1 = 0xCD9E8D57u * c2;
        const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
        c0 = n0;
        c1 = lo1;
        c2 = n2;
        c3 = lo0;
        k0 += 0x9E3779B9u;  // the bump after the last round is never used
        k1 += 0xBB67AE85u;
    }
    return U32x4{{c0, c1, c2, c3}};
}

// ------------------------------------------------------------- fp64 helpers
__device__ __forceinline__ double add(double a, double b) { return __dadd_rn(a, b); }
__device__ __forceinline__ double sub(double a, double b) { return __dsub_rn(a, b); }
__device__ __forceinline__ double mul(double a, double b) { return __dmul_rn(a, b); }
__device__ __forceinline__ double dvd(double a, double b) { return __ddiv_rn(a, b); }

__device__ __forceinline__ double u01(uint32_t x)  // (x + 1/2) 2^-32, exact
{
    return mul(add(__uint2double_rn(x), 0.5), 0x1p-32);
}

// Natural log for positive normal x: x = m 2^e with m in (sqrt(1/2), sqrt(2)],
// s = (m - 1)/(m + 1), ln m = 2 s sum_{i=0..10} s^(2i) / (2i + 1) by Horner,
// ln x = e * ln2_hi + (e * ln2_lo + ln m)  (ln2_hi has 32 significant bits).
__device__ double det_log(double x)
{
    const double inv_odd[11] = {0x1.0000000000000p+0, 0x1.5555555555555p-2, 0x1.999999999999ap-3,
                                0x1.2492492492492p-3, 0x1.c71c71c71c71cp-4, 0x1.745d1745d1746p-4,
                                0x1.3b13b13b13b14p-4, 0x1.1111111111111p-4, 0x1.e1e1e1e1e1e1ep-5,
                                0x1.af286bca1af28p-5, 0x1.8618618618618p-5};
    const unsigned long long bits = (unsigned long long)__double_as_longlong(x);
    long long e = (long long)((bits >> 52) & 0x7ffull) - 1023;
    double m = __longlong_as_double((long long)((bits & 0x000FFFFFFFFFFFFFull) | 0x3FF0000000000000ull));
    if (m > 0x1.6a09e667f3bcdp+0) {
        m = mul(m, 0.5);
        e += 1;
    }
    const double f = sub(m, 1.0);
    const double s = dvd(f, add(m, 1.0));
    const double z = mul(s, s);
    double acc = inv_odd[10];
#pragma unroll
    for (int i = 9; i >= 0; --i) acc = add(mul(acc, z), inv_odd[i]);
    const double ln_m = mul(add(s, s), acc);
    const double ed = __ll2double_rn(e);
    return add(mul(ed, 0x1.62e42fee00000p-1), add(mul(ed, 0x1.a39ef35793c76p-33), ln_m));
}

// exp: k = nearest integer to x / ln2 (halves away from zero),
// r = (x - k ln2_hi) - k ln2_lo, e^r by its degree-13 Taylor polynomial,
// times 2^k through the exponent field.  x is clamped to [-700, 700].
__device__ double det_exp(double x)
{
    const double inv_fact[14] = {0x1.0000000000000p+0, 0x1.0000000000000p+0, 0x1.0000000000000p-1,
                                 0x1.5555555555555p-3, 0x1.5555555555555p-5, 0x1.1111111111111p-7,
                                 0x1.6c16c16c16c17p-10, 0x1.a01a01a01a01ap-13, 0x1.a01a01a01a01ap-16,
                                 0x1.71de3a556c734p-19, 0x1.27e4fb7789f5cp-22, 0x1.ae64567f544e4p-26,
                                 0x1.1eed8eff8d898p-29, 0x1.6124613a86d09p-33};
    if (x > 700.0) x = 700.0;
    if (x < -700.0) x = -700.0;
    const double kf = mul(x, 0x1.71547652b82fep+0);
    const long long k = __double2ll_rz(kf >= 0.0 ? add(kf, 0.5) : sub(kf, 0.5));
    const double kd = __ll2double_rn(k);
    const double r = sub(sub(x, mul(kd, 0x1.62e42fee00000p-1)), mul(kd, 0x1.a39ef35793c76p-33));
    double acc = inv_fact[13];
#pragma unroll
    for (int i = 12; i >= 0; --i) acc = add(mul(acc, r), inv_fact[i]);
    return mul(acc, __longlong_as_double((long long)((unsigned long long)(k + 1023) << 52)));
}

// Wichura (1988), algorithm AS241 PPND16: rational approximations of degree 7
// in r = 0.180625 - q^2 (|q| <= 0.425, q = u - 1/2) or in
// r = sqrt(-ln min(u, 1 - u)) shifted by 1.6 (r <= 5) or by 5.
__device__ __forceinline__ double poly7(const double* c, double r)
{
    double acc = c[7];
#pragma unroll
    for (int i = 6; i >= 0; --i) acc = add(mul(acc, r), c[i]);
    return acc;
}

__device__ double det_ndtri(double u)
{
    const double a[8] = {0x1.b18d91e9eef75p+1, 0x1.0a4888b1a436ep+7, 0x1.ece5d2213c0ccp+10,
                         0x1.ad1d8cd4ee71dp+13, 0x1.66c3e869b752ap+15, 0x1.06c1c55b78f20p+16,
                         0x1.052d26b2e45e4p+15, 0x1.39a296f7d925ep+11};
    const double b[8] = {0x1.0000000000000p+0, 0x1.5281b386e1ab5p+5, 0x1.5797efdc8b3f7p+9,
                         0x1.512322e75c89fp+12, 0x1.4b772d5d65266p+14, 0x1.3317caa64f4bep+15,
                         0x1.c0e457cb1ae76p+14, 0x1.46a7eca984b69p+12};
    const double c[8] = {0x1.6c665fde9526ap+0, 0x1.2857748cab19bp+2, 0x1.713f71462256ap+2,
                         0x1.d2ecb1a3d02c4p+1, 0x1.453cc085375b2p+0, 0x1.ef2abb9b85c37p-3,
                         0x1.744eb6c45ec67p-6, 0x1.9615ac0b7ace9p-11};
    const double d[8] = {0x1.0000000000000p+0, 0x1.06cefbb46a449p+1, 0x1.ad278e6526633p+0,
                         0x1.61292f23385c9p-1, 0x1.2f5123394f040p-3, 0x1.f207a7eab17bfp-7,
                         0x1.1f18cbfdf2728p-11, 0x1.20d3f686439e4p-30};
    const double e[8] = {0x1.aa1b1c13ee526p+2, 0x1.5daea6e875003p+2, 0x1.c8ea6461fa445p+0,
                         0x1.2fad9315255cfp-2, 0x1.b2b41193b4ee7p-6, 0x1.45c1908425345p-10,
                         0x1.c6ec6cc59e02ap-16, 0x1.afb74d693bf93p-23};
    const double f[8] = {0x1.0000000000000p+0, 0x1.331d34fc7d77fp-1, 0x1.186eb183443fbp-3,
                         0x1.e76f93215462ap-7, 0x1.9c8bc979dc5d7p-11, 0x1.35c2c496374bfp-16,
                         0x1.31446f740b9e0p-23, 0x1.269bff1f8c190p-49};
    const double q = sub(u, 0.5);
    const double aq = q < 0.0 ? -q : q;
    if (aq <= 0x1.b333333333333p-2) {
        const double r = sub(0x1.71eb851eb851fp-3, mul(q, q));
        return dvd(mul(q, poly7(a, r)), poly7(b, r));
    }
    const double tail = q < 0.0 ? u : sub(1.0, u);
    double r = __dsqrt_rn(-det_log(tail));
    double v;
    if (r <= 5.0) {
        r = sub(r, 0x1.999999999999ap+0);
        v = dvd(poly7(c, r), poly7(d, r));
    } else {
        r = sub(r, 5.0);
        v = dvd(poly7(e, r), poly7(f, r));
    }
    return q < 0.0 ? -v : v;
}

// clip(floor(v + 1/2), lo, hi) for v >= 0 (NaN / inf / huge -> hi)
__device__ __forceinline__ int64_t round_clip(double v, int64_t lo, int64_t hi)
{
    const double y = add(v, 0.5);
    if (!(y < __ll2double_rn(hi))) return hi;
    const int64_t t = __double2ll_rz(y);
    return t < lo ? lo : t;
}

__device__ __forceinline__ int64_t dwell(const TraceParams& P, uint32_t k0, uint32_t k1, uint32_t sub_id,
                                         int64_t j)
{
    const U32x4 x = philox((uint32_t)j, sub_id, 1u, 0u, k0, k1);
    const double g = det_log(u01(x.v[0]));
    return __double2ll_rz(mul(-g, __ll2double_rn(P.dwell_mean_us)));
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
                const double zp = det_ndtri(u01(x.v[0]));
                p = round_clip(det_exp(add(P.prompt_mu, mul(P.prompt_sigma, zp))), P.prompt_min, P.prompt_max);
                const bool is_short = (uint64_t)x.v[1] < P.mix_short_thr;
                const double mu = is_short ? P.short_mu : P.long_mu;
                const double sg = is_short ? P.short_sigma : P.long_sigma;
                const double zo = det_ndtri(u01(x.v[2]));
                o = round_clip(det_exp(add(mu, mul(sg, zo))), P.out_min, P.out_max);
                const double zn = det_ndtri(u01(x.v[3]));
                oh = round_clip(mul(__ll2double_rn(o), det_exp(mul(P.noise_sigma, zn))), P.pred_min, P.pred_max);
                while (c < P.n_classes - 1 && (uint64_t)y.v[0] >= P.class_thr[c]) ++c;
                gap = __double2ll_rz(mul(-det_log(u01(y.v[1])), 1e9));
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
                t = lam / P.rate[0];
            } else {
                // walk the intervals until every live lane found the last j with A_j <= lam
                bool done = !live;
                for (;;) {
                    if (!done && lam < A_next) {
                        t = T + (lam - A) / P.rate[j & 1];
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
    const int warps_per_block = 8;
    int64_t blocks = (p.n_replicas + warps_per_block - 1) / warps_per_block;
    const int64_t cap = (int64_t)sms * 8;
    if (blocks > cap) blocks = cap;
    trace_kernel<<<(unsigned)blocks, warps_per_block * 32, 0, stream>>>(p);
    return cudaGetLastError();
}

}  // namespace ctr
