// noalloc.cu -- rfq_linear_noalloc: the RFQ GEMM for callers that cannot
// allocate device memory.
//
// rfq_linear needs a small device workspace (its status word) from the
// caller.  Some callers cannot provide one: code that runs where
// cudaMalloc is not allowed or not wanted (a real-time serving loop that must
// not synchronize the device, a plug-in inside a host program that owns all
// device memory, a runtime without a device allocator of its own).  For them
// this entry point keeps the workspace in a fixed array in the library's own
// device memory instead.  It is a file-scope __device__ array, so every GPU
// that loads the library holds it until the process exits.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "internal.h"

namespace {

// Largest workspace the allocation-free entry point can stand in for.
constexpr size_t kNoallocScratchBytes = 256;

// The scratch array.  In host code this name is only a stand-in for the
// symbol, not a device address: its device address comes from
// cudaGetSymbolAddress, once per device.
static __device__ __align__(256) int32_t g_noalloc_scratch[kNoallocScratchBytes / sizeof(int32_t)];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array on the current device (looked up on
// the first call on that device, with that device current, and kept for the
// life of the process: a cudaDeviceReset, which reloads the library's device
// code, makes the kept address stale, so callers of this entry point do not
// reset the device).
rfq_status scratch_address(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return RFQ_ERR_DEVICE;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_scratch_addr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p)
            return RFQ_ERR_CUDA;
        g_scratch_addr[dev] = p;
    }
    *out = g_scratch_addr[dev];
    return RFQ_OK;
}

} // namespace

extern "C" rfq_status rfq_linear_noalloc(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi,
                                         int32_t phi_r_s, const rfq_qtensor *wq, void *y, int32_t out_dtype,
                                         void *stream)
{
    if (rfq_linear_workspace_bytes() > kNoallocScratchBytes)
        return RFQ_ERR_SHAPE;   // the GEMM needs more scratch than the fixed array holds
    // rfq_linear's own checks first: a call it would reject, or one with
    // nothing to compute, leaves the shared array untouched.
    bool launch = false;
    rfq_status s = rfq::linear_check(xq, xr, phi, phi_r_s, wq, y, out_dtype, nullptr, &launch, false);
    if (s != RFQ_OK || !launch)
        return s;
    void *scratch = nullptr;
    if ((s = scratch_address(&scratch)) != RFQ_OK)
        return s;
    // The array keeps whatever the previous call left; its status word must
    // start at zero or the GEMM returns without computing.
    if (cudaMemsetAsync(scratch, 0, kNoallocScratchBytes, static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return RFQ_ERR_CUDA;
    return rfq_linear(xq, xr, phi, phi_r_s, wq, y, out_dtype, scratch, stream);
}
