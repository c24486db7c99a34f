// decode_no_alloc.cu -- parason_attn_decode_no_alloc: the decode step with its
// partial results in a fixed scratch array of the library's device image
// instead of a caller workspace, for callers that cannot hand over device
// memory at decode time.  Nothing here allocates: the array is reserved with
// the module, its address is looked up once per device, and the step itself
// is the one parason_attn_decode launches.
#include <cuda_runtime.h>

#include <mutex>

#include "internal.h"

// Partial results (unnormalised o, then the running max and sum of every
// row) of one decode step.  Never needs zeroing: the attention kernel writes
// every row the merge kernel of the same call reads.
static __device__ __align__(256) unsigned char g_partials_scratch[PARASON_NO_ALLOC_SCRATCH_BYTES];

namespace {

constexpr int kMaxDevices = 64;

std::mutex g_scratch_mutex;
void *g_scratch_addr[kMaxDevices] = {};

// Device address of g_partials_scratch on the current device; looked up on
// the first call for that device, with that device current.
parason_status scratch_on_current_device(void **addr) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) return PARASON_ECUDA;
    if (dev < 0 || dev >= kMaxDevices) return PARASON_EUNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_partials_scratch) != cudaSuccess || !p) {
            // leave no error pending for the next, unrelated runtime call
            cudaGetLastError();
            return PARASON_ECUDA;
        }
        g_scratch_addr[dev] = p;
    }
    *addr = g_scratch_addr[dev];
    return PARASON_OK;
}

}  // namespace

extern "C" parason_status parason_attn_decode_no_alloc(parason_plan plan, const void *q,
                                                       const void *k_pages, const void *v_pages,
                                                       const float *k_scale, const float *v_scale,
                                                       void *out, float *lse,
                                                       parason_stream_t stream) {
    if (!plan) return PARASON_EINVAL;
    if (parason_plan_workspace_bytes(plan) > sizeof(g_partials_scratch)) return PARASON_EUNSUPPORTED;
    // the plan's device must be current before the scratch is looked up:
    // the lookup loads the library's device image on the current device
    const int plan_dev = parason::plan_device(plan);
    if (plan_dev < 0) return PARASON_EINVAL;
    int cur = -1;
    if (cudaGetDevice(&cur) != cudaSuccess) {
        cudaGetLastError();
        return PARASON_ECUDA;
    }
    if (cur != plan_dev) return PARASON_EINVAL;
    void *scratch = nullptr;
    const parason_status st = scratch_on_current_device(&scratch);
    if (st != PARASON_OK) return st;
    return parason_attn_decode(plan, q, k_pages, v_pages, k_scale, v_scale, out, lse, scratch,
                               sizeof(g_partials_scratch), stream);
}
