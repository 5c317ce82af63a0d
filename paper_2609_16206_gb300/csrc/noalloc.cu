// noalloc.cu -- ctr_simulate_noalloc: the simulator without a caller-provided
// workspace, for callers that cannot allocate device memory.
//
// Some callers of this library run where a device allocation is not allowed
// or not theirs to make: a scheduler plugin inside a serving process whose
// memory pool owns every byte of the GPU, code that runs between the capture
// calls of someone else's CUDA graph, or a real-time loop that must never hit
// the driver's allocator.  They still own their inputs and outputs; what they
// cannot provide is the simulator's scratch (the per-warp heaps, rings and the
// row counter).  This entry point takes that scratch from a fixed array that
// lives in this file for as long as the library stays loaded.
//
// The array is CTR_NOALLOC_SCRATCH_BYTES (64 MiB) of device memory per GPU that
// loads the library, held until the process exits.  The first call on a device
// looks the array's device address up (once per device, with that device
// current); make that first call before any stream capture.  Every call shares it: the row
// counter at its start is cleared by each call, the rest needs no clearing
// (every row resets the structures it uses).  Calls that overlap on the GPU
// -- on two streams, or from two host threads -- race on the array and give
// wrong results; serialise them.  A configuration whose per-warp slot does
// not fit the array is rejected with CTR_EINVAL; otherwise fewer warps run
// concurrently than with a full-size workspace, and the results are the same.
#include <mutex>

#include "ctr_internal.cuh"

namespace {

constexpr size_t kScratchBytes = CTR_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_scratch[kScratchBytes];

std::mutex g_setup_mutex;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device.  The host-side name is
// only a stand-in; the address has to come from the runtime, once per device,
// with that device current.
int scratch_address(void** out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return CTR_ECUDA;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || p == nullptr) return CTR_ECUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return CTR_OK;
}

}  // namespace

extern "C" {

int ctr_simulate_noalloc(const ctr_sim_cfg* cfg, const ctr_cost_consts* consts, int32_t n_const_sets,
                         const int32_t* policy_ids, int32_t n_policies, ctr_requests trace, int32_t n_replicas,
                         int64_t n_req, uint8_t* i_pre, uint8_t* i_dec, int64_t* t_first_us, int64_t* t_done_us,
                         uint64_t* row_hash, int32_t* row_status, void* stream)
{
    if (!cfg) return CTR_EINVAL;
    int64_t off_act = 0, off_wait = 0;
    int32_t cap_pr = 0;
    if (cfg->cap_pending >= 1 && cfg->cap_waiting >= 1 && cfg->cap_active >= 1 && cfg->cap_prefill_ring >= 1 &&
        cfg->cap_pending <= (1 << 20) && cfg->cap_waiting <= (1 << 20) && cfg->cap_active <= (1 << 20) &&
        cfg->cap_prefill_ring <= (1 << 20)) {
        const int64_t slot = ctr::sim_slot_bytes(*cfg, &off_act, &off_wait, &cap_pr);
        if (256 + slot > (int64_t)kScratchBytes) return CTR_EINVAL;  // one warp's structures do not fit
    }
    void* scratch = nullptr;
    const int rc = scratch_address(&scratch);
    if (rc != CTR_OK) return rc;
    return ctr_simulate(cfg, consts, n_const_sets, policy_ids, n_policies, trace, n_replicas, n_req, i_pre, i_dec,
                        t_first_us, t_done_us, row_hash, row_status, nullptr, nullptr, scratch, kScratchBytes,
                        stream);
}

}  // extern "C"
