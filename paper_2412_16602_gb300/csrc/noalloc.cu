// noalloc.cu - vmb_selective_scan_fwd_noalloc: the full selective scan for
// callers that cannot allocate device memory.
//
// vmb_selective_scan_fwd needs a caller-provided workspace for the state
// exchange between L-chunks.  Some callers cannot provide one: code hosted
// inside a framework whose memory pool owns the device and forbids
// allocations of its own, or a serving loop that must not allocate once it
// is running (cudaMalloc can synchronise the device and can fail when memory
// is fragmented).  This entry point takes the same inputs and outputs but
// keeps its scratch in a fixed-size array that is part of the library image
// itself: every GPU that loads libvmb holds kScratchBytes for it until the
// process exits, and the call itself allocates nothing.
#include <mutex>

#include "vmb_common.cuh"
#include "vmb_internal.h"

namespace vmb {
namespace {

constexpr size_t kScratchBytes = 16u << 20;  // 16 MiB per device

// The scratch array.  In host code this name is only a stand-in, not a
// device address: the address is looked up once per device with
// cudaGetSymbolAddress (see scratch_for_current_device) and passed on.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of g_scratch on the current device; looked up on the first
// call made with that device current and kept for the life of the process
// (the entry point must therefore not be used across a cudaDeviceReset of
// that device, after which the cached address no longer names the array).
vmb_status scratch_for_current_device(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return VMB_ERR_CUDA;
    if (dev < 0 || dev >= kMaxDevices) return VMB_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) return VMB_ERR_CUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return VMB_OK;
}

}  // namespace
}  // namespace vmb

using namespace vmb;

extern "C" vmb_status vmb_selective_scan_fwd_noalloc(const void* u, const void* delta, const float* A,
                                                     const void* Bs, const void* Cs, const float* Dskip,
                                                     const float* delta_bias, void* y, int B, int K, int D,
                                                     int N, int H, int W, unsigned flags, vmb_dtype dtype,
                                                     cudaStream_t stream) {
    if (H < 0 || W < 0) return VMB_ERR_INVALID_ARG;
    if ((long long)H * W > 0x7fffffffLL) return VMB_ERR_UNSUPPORTED;
    // Every argument check of vmb_selective_scan_fwd runs before anything is
    // queued on the GPU, so that a rejected call has no side effects.
    ScanArgs a{u, delta, A, Bs, Cs, Dskip, delta_bias, y, nullptr, B, K, D, N, H * W, flags, dtype, nullptr, 0};
    bool empty = false;
    vmb_status s = validate_scan(a, false, &empty);
    if (s != VMB_OK || empty) return s;
    ScanPlan plan{};
    s = plan_full(a, &plan);
    if (s != VMB_OK) return s;
    if (plan.ws_bytes > kScratchBytes) return VMB_ERR_WORKSPACE;  // more scratch than the built-in array
    void* scratch = nullptr;
    s = scratch_for_current_device(&scratch);
    if (s != VMB_OK) return s;
    a.ws = scratch;
    a.ws_bytes = kScratchBytes;
    // The array keeps whatever the previous call left in it.  The status
    // header and the chunk flags of this plan must start at zero; the
    // published states are only read after their flag is set, so they need
    // no clearing.
    const WsLayout w = ws_layout(plan);
    const size_t clear = plan.n_chunks > 1 ? w.aggP_off : 256;
    if (cudaMemsetAsync(scratch, 0, clear, stream) != cudaSuccess) return VMB_ERR_CUDA;
    return launch_full(a, plan, stream);
}
