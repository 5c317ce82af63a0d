// ctr_internal.cuh -- declarations shared by the CUDA translation units of
// libctr.so (kernel parameter blocks and launchers).  Not part of the ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "../../include/ctr.h"

namespace ctr {

// Bounds-checked builds (libctr_checked.so) define CTR_BOUNDS_CHECK=1.
#ifndef CTR_BOUNDS_CHECK
#define CTR_BOUNDS_CHECK 0
#endif

constexpr int kWarp = 32;
constexpr int64_t kTimeLimit = int64_t(1) << 40;   // every simulated time stays below this
constexpr int64_t kArrivalLimit = int64_t(1) << 39;
constexpr int kKeyBits = 23;                        // request index bits in packed heap keys
constexpr uint64_t kKeyMask = (uint64_t(1) << kKeyBits) - 1;

// Checked accesses.  A build with CTR_BOUNDS_CHECK=1 compares every index with
// the length of its buffer first; an index outside skips the access (a load
// gives 0) and sets `bad`, and the kernel reports CTR_EBOUNDS for the row.
// Other builds compile the plain access (the length and the flag are dead code
// there).
#if CTR_BOUNDS_CHECK
__device__ __forceinline__ bool ck_out(int64_t i, int64_t len, bool& bad)
{
    const bool out = (uint64_t)i >= (uint64_t)len;
    bad = bad || out;
    return out;
}
#define CTR_CK_OUT(i, len, bad) ck_out((int64_t)(i), (len), (bad))
#else
#define CTR_CK_OUT(i, len, bad) false
#endif
// true when index i lies in [0, len) (always, in unchecked builds)
__device__ __forceinline__ bool ck_ok(int64_t i, int64_t len, bool& bad) { return !CTR_CK_OUT(i, len, bad); }
// (the index keeps the caller's type, so the unchecked address arithmetic is the plain one)
template <typename T, typename I>
__device__ __forceinline__ T ck_ld(const T* p, I i, int64_t len, bool& bad)
{
    if (CTR_CK_OUT(i, len, bad)) return T();
    return p[i];
}
template <typename T, typename I>
__device__ __forceinline__ T ck_ldg(const T* p, I i, int64_t len, bool& bad)  // read-only data
{
    if (CTR_CK_OUT(i, len, bad)) return T();
    return __ldg(p + i);
}
template <typename T, typename I>
__device__ __forceinline__ void ck_st(T* p, I i, int64_t len, T v, bool& bad)
{
    if (CTR_CK_OUT(i, len, bad)) return;
    p[i] = v;
}
// entries i and i + 1 as one 16-byte word (the checked build also checks its 16-byte alignment)
template <typename I>
__device__ __forceinline__ ulonglong2 ck_ld2(const uint64_t* p, I i, int64_t len, bool& bad)
{
    if (CTR_CK_OUT(i, len - 1, bad)) return make_ulonglong2(0, 0);
#if CTR_BOUNDS_CHECK
    if ((reinterpret_cast<uintptr_t>(p + i) & 15u) != 0) {
        bad = true;
        return make_ulonglong2(0, 0);
    }
#endif
    return *reinterpret_cast<const ulonglong2*>(p + i);
}

// Row checksum term mix(k, tag, v) = sm(sm((tag << 56) ^ k) ^ v), sm the
// splitmix64 output function (Steele, Lea and Flood, OOPSLA'14).
__device__ __forceinline__ uint64_t mix64(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}
__device__ __forceinline__ uint64_t hterm(int64_t k, uint64_t tag, uint64_t v)
{
    return mix64(mix64((tag << 56) ^ (uint64_t)k) ^ v);
}

// Philox4x32-10 (Salmon et al., SC'11): ten rounds of two 32x32 -> 64 products,
// the key bumped by the Weyl constants between rounds.
struct Philox4 {
    uint32_t v[4];
};
__device__ __forceinline__ Philox4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
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
    return Philox4{{c0, c1, c2, c3}};
}

// ---------------------------------------------------------------- trace
struct TraceParams {
    uint64_t seed;
    int64_t n_seeds;
    int32_t arrival_kind;
    int32_t n_classes;
    int64_t rate[2];
    uint64_t rate_recip[2];     // floor((2^64 - 1) / rate)
    int64_t dwell_mean_us;
    float dwell_mean_f;         // dwell_mean_us rounded once to fp32
    float prompt_mu, prompt_sigma, short_mu, short_sigma, long_mu, long_sigma, noise_sigma;
    int64_t prompt_min, prompt_max, out_min, out_max, pred_min, pred_max;
    uint64_t mix_short_thr;
    uint64_t class_thr[3];
    int64_t n_replicas, replica_offset, n_req;
    ctr_requests out;
};
cudaError_t launch_trace(const TraceParams& p, cudaStream_t stream);

// ---------------------------------------------------------------- simulator
struct ConstsDev {
    int64_t tau_pre0, tau_pre, tau_dec, w_q;
    int32_t w_b, w_s, rho, sigma[4];
    uint32_t ablate;
    uint32_t proxy;       // backlog from the priced in-flight ledger
    int64_t poll_us;      // > 0: occupancy polled on this period
    uint64_t poll_recip;  // floor((2^64 - 1) / poll_us)
};

// The host validates pre_tok, xfer_tok <= 2^20, dec_seq <= 2^16, kv_div <= 2^31
// and max_steps <= 2^31 - 2^21, so the kernel takes their products with
// 32-bit counts as single 32 x 32-bit multiplies of the low words.
struct SimParams {
    int32_t n_pre, n_dec;
    int64_t kv_cap;
    uint64_t kv_cap_recip;      // floor((2^64 - 1) / kv_cap)
    int64_t pre_base, pre_tok, xfer_tok;
    int64_t dec_base, dec_seq;
    int64_t kv_div;
    int64_t pre_batch;          // prefill batch token budget, 0 = serial prefill
    uint64_t kv_div_magic;      // ceil(2^64 / kv_div) (kv_div >= 2)
    int32_t n_classes, heur_thresh;
    int64_t max_steps;
    int32_t cap_pend, cap_wait, cap_act, cap_ring;
    int32_t cap_pend_store;     // pending heap entries: cap_pend + cap_wait + 1
    int32_t n_sets, n_pols;
    int32_t pols[8];
    int64_t n_req, n_rows;
    // per-slot workspace: three regions, each lane's entries contiguous within a region
    unsigned char* ws;
    uint32_t* next_row;
    int64_t slot_bytes;
    int64_t off_act, off_wait;  // byte offsets of the active heap and waiting ring inside a slot
    int32_t cap_pr;             // max(cap_pend_store, cap_ring): entries of the first region
    int32_t n_slots;
    ctr_requests trace;
    uint8_t* i_pre;
    uint8_t* i_dec;
    int64_t* t_first;
    int64_t* t_done;
    uint64_t* row_hash;
    int32_t* row_status;
    ConstsDev sets[CTR_MAX_CONST_SETS];
    int64_t trace_len;          // entries of each trace array (replicas x requests)
    int64_t out_len;            // entries of each per-request output (rows x requests)
};
int64_t sim_slot_bytes(const ctr_sim_cfg& cfg, int64_t* off_act, int64_t* off_wait, int32_t* cap_pr);
int sim_max_resident_warps(int* warps_per_block, int* blocks);
int sim_group_width(int n_instances);  // lanes per simulated row; 32 / width rows share a warp
cudaError_t launch_sim(const SimParams& p, int blocks, int warps_per_block, cudaStream_t stream);
// The first-token and completion checksum terms in a pass of their own (when no
// goodput pass adds them); kmix as for GoodputParams, or null.
cudaError_t launch_hash(const SimParams& p, const uint64_t* kmix, int blocks, cudaStream_t stream);
// The request-only halves of the checksum's first-token and completion terms:
// t[k] = mix64((2 << 56) ^ k) and t[n + k] = mix64((3 << 56) ^ k) for k < n,
// shared by every row of a call (the passes that sum the terms read them
// instead of mixing each row-request's index again).
cudaError_t launch_mix_table(uint64_t* t, int64_t n, cudaStream_t stream);

// ---------------------------------------------------------------- goodput
struct GoodputParams {
    ctr_requests trace;
    int64_t n_req, n_rows;
    int32_t rows_per_replica, n_classes;
    int64_t ttft[4], tpot[4];
    const int64_t* t_first;
    const int64_t* t_done;
    int64_t* met;
    int64_t* p99;
    // optional (both or neither): add each OK row's first-token and completion
    // checksum terms to row_hash in the same pass over the outputs
    uint64_t* row_hash;
    const int32_t* row_status;
    const uint64_t* kmix;  // optional with row_hash: the table of launch_mix_table for n_req
};
cudaError_t launch_goodput(const GoodputParams& p, cudaStream_t stream);
// Each row's nearest-rank P99 TPOT into p99_tpot[row] (-1 when no request has two tokens or more).
cudaError_t launch_tpot(const GoodputParams& p, int64_t* p99_tpot, cudaStream_t stream);

// ---------------------------------------------------------------- standalone scorer
struct ScoreParams {
    const float* p;
    const float* oh;
    const uint8_t* cls;
    int64_t n;
    const float* Q;
    const float* A;
    const float* kap;
    int32_t n_inst;
    float c[CTR_SCORE_N_CONST];
    int32_t* argmin;
    float* cost;
    int32_t* status;
};
cudaError_t launch_score(const ScoreParams& p, cudaStream_t stream);
cudaError_t launch_stream_probe(const ScoreParams& p, cudaStream_t stream);  // scorer's traffic only

}  // namespace ctr
