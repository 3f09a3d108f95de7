// host_path.cu -- rfq_linear_host: the RFQ linear layer (Algorithm 1, Eq. rfq)
// end to end from host memory.
//
// X arrives in host memory and Y goes back to it.  The call splits the rows
// into chunks; for each chunk it copies X to the device on a copy stream of
// the library's, runs the activation quantizer and the RFQ GEMM on the
// caller's stream, and copies Y back on a second copy stream, so that the
// copies of one chunk overlap the kernels and copies of its neighbours
// (the host link, not the kernels, bounds this path).  Everything on the
// device is the caller's memory; the library creates streams and events
// only.
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>
#include <vector>

#include "internal.h"

namespace {

constexpr int kMaxDevices = 64;
constexpr int64_t kDefaultChunkRows = 8192;

// The two copy streams of each device, created on first use and kept.
struct CopyStreams {
    cudaStream_t h2d = nullptr, d2h = nullptr;
};
std::mutex g_mu;
CopyStreams g_streams[kMaxDevices];

rfq_status copy_streams(CopyStreams *out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return RFQ_ERR_DEVICE;
    std::lock_guard<std::mutex> lock(g_mu);
    CopyStreams &c = g_streams[dev];
    if (!c.h2d && cudaStreamCreateWithFlags(&c.h2d, cudaStreamNonBlocking) != cudaSuccess)
        return RFQ_ERR_CUDA;
    if (!c.d2h && cudaStreamCreateWithFlags(&c.d2h, cudaStreamNonBlocking) != cudaSuccess)
        return RFQ_ERR_CUDA;
    *out = c;
    return RFQ_OK;
}

// Rows [r0, r0 + m) of an MXFP4 activation in the MMA scale layout (r0 a
// multiple of 128: its 128-row scale tiles are contiguous).
rfq_qtensor rows_of(const rfq_qtensor &q, int64_t r0, int64_t m)
{
    rfq_qtensor v = q;
    v.rows = m;
    v.codes = static_cast<uint8_t *>(q.codes) + r0 * (q.k / 2);
    v.scales = static_cast<uint8_t *>(q.scales) + r0 * (q.k / 32);
    return v;
}

// Events of one call, destroyed when the call returns (their pending
// records complete on their own).
struct Events {
    std::vector<cudaEvent_t> ev;
    cudaEvent_t make()
    {
        cudaEvent_t e = nullptr;
        if (cudaEventCreateWithFlags(&e, cudaEventDisableTiming) != cudaSuccess)
            return nullptr;
        ev.push_back(e);
        return e;
    }
    ~Events()
    {
        for (cudaEvent_t e : ev)
            cudaEventDestroy(e);
    }
};

} // namespace

extern "C" {

rfq_status rfq_linear_host(const void *x_host, int64_t M, int64_t K, const rfq_fallback *fb, const rfq_qtensor *wq,
                           void *y_host, int32_t out_dtype, int64_t chunk_rows, void *x_dev, rfq_qtensor *xq,
                           rfq_qtensor *xr, uint8_t *phi, void *y_dev, void *workspace, void *stream)
{
    using namespace rfq;
    if (!xq || !wq || !workspace || (M > 0 && (!x_host || !y_host || !x_dev || !y_dev)))
        return RFQ_ERR_INVALID_ARG;
    const int32_t mode = fb ? fb->mode : RFQ_FALLBACK_ALL;
    if (mode != RFQ_FALLBACK_NONE && mode != RFQ_FALLBACK_ALL && mode != RFQ_FALLBACK_AMAX)
        return RFQ_ERR_INVALID_ARG;
    if ((mode == RFQ_FALLBACK_NONE) != (xr == nullptr))
        return RFQ_ERR_INVALID_ARG;
    if (mode == RFQ_FALLBACK_AMAX && (!phi || fb->p_s != 128 || fb->r_s < 128 || fb->r_s % 128 != 0))
        return RFQ_ERR_INVALID_ARG;
    if (chunk_rows == 0)
        chunk_rows = kDefaultChunkRows;
    if (M < 0 || K <= 0 || chunk_rows < 0 || chunk_rows % 128 != 0)
        return RFQ_ERR_SHAPE;
    if (xq->rows != M || xq->k != K || (xr && (xr->rows != M || xr->k != K)))
        return RFQ_ERR_SHAPE;
    // MXFP4 pathways in the MMA scale layout (the layout the row chunks slice)
    if (xq->fmt != RFQ_FMT_MXFP4 || xq->scale_layout != RFQ_SCALE_MMA ||
        (xr && (xr->fmt != RFQ_FMT_MXFP4 || xr->scale_layout != RFQ_SCALE_MMA)) || wq->fmt != RFQ_FMT_MXFP4)
        return RFQ_ERR_UNSUPPORTED;
    if ((reinterpret_cast<uintptr_t>(x_dev) & 15u) != 0)
        return RFQ_ERR_ALIGNMENT;
    if (M == 0)
        return RFQ_OK;   // nothing to copy or compute
    const int32_t r_s = mode == RFQ_FALLBACK_AMAX ? fb->r_s : 256;
    // every host-side check of the GEMM, on the whole matrices
    bool launch = false;
    rfq_status s = linear_check(xq, xr, mode == RFQ_FALLBACK_AMAX ? phi : nullptr, r_s, wq, y_dev, out_dtype,
                                workspace, &launch, true);
    if (s != RFQ_OK || !launch)
        return s;
    CopyStreams cs;
    if ((s = copy_streams(&cs)) != RFQ_OK)
        return s;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int64_t N = wq->rows;
    const size_t ybytes = out_dtype == RFQ_OUT_BF16 ? 2 : 4;
    const int64_t phi_cols = (K + r_s - 1) / r_s;
    Events E;
    cudaEvent_t start = E.make(), done = E.make();
    if (!start || !done)
        return RFQ_ERR_CUDA;
    // the copies into x_dev start after the work already on `stream`
    if (cudaEventRecord(start, st) != cudaSuccess || cudaStreamWaitEvent(cs.h2d, start, 0) != cudaSuccess ||
        cudaStreamWaitEvent(cs.d2h, start, 0) != cudaSuccess)
        return RFQ_ERR_CUDA;
    for (int64_t r0 = 0; r0 < M; r0 += chunk_rows) {
        const int64_t m = M - r0 < chunk_rows ? M - r0 : chunk_rows;
        cudaEvent_t x_ready = E.make(), y_ready = E.make();
        if (!x_ready || !y_ready)
            return RFQ_ERR_CUDA;
        const size_t xoff = (size_t)r0 * (size_t)K * 2, xlen = (size_t)m * (size_t)K * 2;
        if (cudaMemcpyAsync(static_cast<uint8_t *>(x_dev) + xoff, static_cast<const uint8_t *>(x_host) + xoff, xlen,
                            cudaMemcpyHostToDevice, cs.h2d) != cudaSuccess ||
            cudaEventRecord(x_ready, cs.h2d) != cudaSuccess || cudaStreamWaitEvent(st, x_ready, 0) != cudaSuccess)
            return RFQ_ERR_CUDA;
        rfq_qtensor q = rows_of(*xq, r0, m), r = xr ? rows_of(*xr, r0, m) : rfq_qtensor{};
        uint8_t *ph = mode == RFQ_FALLBACK_AMAX ? phi + (r0 / 128) * phi_cols : nullptr;
        void *yd = static_cast<uint8_t *>(y_dev) + (size_t)r0 * (size_t)N * ybytes;
        if ((s = rfq_quantize_act(static_cast<uint8_t *>(x_dev) + xoff, m, K, fb, &q, xr ? &r : nullptr, ph,
                                  stream)) != RFQ_OK)
            return s;
        if ((s = rfq_linear(&q, xr ? &r : nullptr, ph, r_s, wq, yd, out_dtype, workspace, stream)) != RFQ_OK)
            return s;
        const size_t yoff = (size_t)r0 * (size_t)N * ybytes, ylen = (size_t)m * (size_t)N * ybytes;
        if (cudaEventRecord(y_ready, st) != cudaSuccess || cudaStreamWaitEvent(cs.d2h, y_ready, 0) != cudaSuccess ||
            cudaMemcpyAsync(static_cast<uint8_t *>(y_host) + yoff, static_cast<const uint8_t *>(y_dev) + yoff, ylen,
                            cudaMemcpyDeviceToHost, cs.d2h) != cudaSuccess)
            return RFQ_ERR_CUDA;
    }
    // `stream` passes this point once Y is in host memory (and the copy
    // streams have no work left that touches x_dev or y_dev)
    if (cudaEventRecord(done, cs.d2h) != cudaSuccess || cudaStreamWaitEvent(st, done, 0) != cudaSuccess)
        return RFQ_ERR_CUDA;
    cudaEvent_t h_done = E.make();
    if (!h_done || cudaEventRecord(h_done, cs.h2d) != cudaSuccess || cudaStreamWaitEvent(st, h_done, 0) != cudaSuccess)
        return RFQ_ERR_CUDA;
    return RFQ_OK;
}

} // extern "C"
