// api.cu -- the C ABI declared in include/rfq.h: argument validation,
// tensor-map encoding and kernel dispatch.  No entry point allocates device
// memory; every buffer belongs to the caller.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdlib>
#include <mutex>

#include "internal.h"

namespace rfq {
namespace {

typedef CUresult (*PFN_encodeTiled)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                    const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                    CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                    CUtensorMapFloatOOBfill);

PFN_encodeTiled get_encode()
{
    static PFN_encodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_encodeTiled>(p);
    });
    return fn;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

rfq_status check_device()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return RFQ_ERR_DEVICE;
    static int cache[64];   // 0 unknown, 1 ok, 2 not sm_103
    if (dev < 0 || dev >= 64)
        return RFQ_ERR_DEVICE;
    if (cache[dev] == 0) {
        int major = 0, minor = 0;
        if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess)
            return RFQ_ERR_DEVICE;
        cache[dev] = (major == 10 && minor == 3) ? 1 : 2;
    }
    return cache[dev] == 1 ? RFQ_OK : RFQ_ERR_DEVICE;
}

rfq_status from_cuda(cudaError_t e) { return e == cudaSuccess ? RFQ_OK : RFQ_ERR_CUDA; }

// The environment variable RFQ_DEBUG_SYNC (any value but "0") makes every
// GEMM entry point synchronize its stream after the launch and return the
// device status its workspace holds (RFQ_ERR_TIMEOUT, ...) instead of RFQ_OK.
bool debug_sync()
{
    static const int on = [] {
        const char *v = getenv("RFQ_DEBUG_SYNC");
        return v && v[0] && !(v[0] == '0' && v[1] == 0) ? 1 : 0;
    }();
    return on != 0;
}

bool fmt_ok(int32_t f)
{
    return f == RFQ_FMT_MXFP4 || f == RFQ_FMT_HIF4 || f == RFQ_FMT_BF16 || f == RFQ_FMT_MXFP8;
}
bool layout_ok(int32_t l) { return l == RFQ_SCALE_ROWMAJOR || l == RFQ_SCALE_MMA; }

// Granule of the k axis for a format / scale layout.
int64_t k_granule(int32_t fmt, int32_t layout)
{
    if (fmt == RFQ_FMT_HIF4)
        return 64;
    if (fmt == RFQ_FMT_BF16)
        return 8;
    return layout == RFQ_SCALE_MMA ? 128 : 32;
}

rfq_status check_qtensor(const rfq_qtensor *q, int64_t rows, int64_t k)
{
    if (!q || !fmt_ok(q->fmt) || !layout_ok(q->scale_layout))
        return RFQ_ERR_INVALID_ARG;
    if (q->rows != rows || q->k != k || rows < 0 || k <= 0 || k % k_granule(q->fmt, q->scale_layout) != 0)
        return RFQ_ERR_SHAPE;
    const bool need_scales = q->fmt != RFQ_FMT_BF16;
    if (rows > 0 && (!q->codes || (need_scales && !q->scales)))
        return RFQ_ERR_INVALID_ARG;
    if (!aligned16(q->codes) || (need_scales && !aligned16(q->scales)))
        return RFQ_ERR_ALIGNMENT;
    return RFQ_OK;
}

} // namespace

int num_sms()
{
    static int cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64)
        return 148;
    if (cache[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        cache[dev] = n;
    }
    return cache[dev];
}

int resident_blocks_per_sm(const void *kern, int threads, size_t smem)
{
    // (one entry per kernel: a handful of quantizers, looked up once each)
    struct Entry {
        const void *kern;
        int threads, blocks;
    };
    static Entry table[64];
    static int used = 0;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (int i = 0; i < used; ++i)
        if (table[i].kern == kern && table[i].threads == threads)
            return table[i].blocks;
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kern, threads, smem) != cudaSuccess || n < 1)
        n = 1;
    if (used < 64)
        table[used++] = {kern, threads, n};
    return n;
}

bool encode_tmap_2d_u8(CUtensorMap *map, const void *base, uint64_t inner_bytes, uint64_t rows,
                       uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows, int swizzle)
{
    PFN_encodeTiled enc = get_encode();
    if (!enc)
        return false;
    cuuint64_t dims[2] = {inner_bytes, rows};
    cuuint64_t strides[1] = {row_stride_bytes};
    cuuint32_t box[2] = {box_inner, box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void *>(base), dims, strides, box, estr,
                     CU_TENSOR_MAP_INTERLEAVE_NONE,
                     swizzle == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                     : swizzle == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                     : CU_TENSOR_MAP_SWIZZLE_NONE,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool encode_tmap_2d_e2m1_padded(CUtensorMap *map, const void *base, uint64_t k, uint64_t rows,
                                uint32_t box_rows)
{
    PFN_encodeTiled enc = get_encode();
    if (!enc || (reinterpret_cast<uintptr_t>(base) & 31u) != 0 || k % 128 != 0)
        return false;
    cuuint64_t dims[2] = {k, rows};         // in 4-bit codes
    cuuint64_t strides[1] = {k / 2};        // bytes
    cuuint32_t box[2] = {128, box_rows};    // 128 codes: 64 bytes read, 128 written
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_16U4_ALIGN16B, 2, const_cast<void *>(base), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

} // namespace rfq

using namespace rfq;

namespace rfq {
namespace {
// The status of a GEMM launch (see debug_sync).
rfq_status gemm_done(cudaError_t e, void *workspace, cudaStream_t st)
{
    if (e != cudaSuccess)
        return RFQ_ERR_CUDA;
    if (!debug_sync())
        return RFQ_OK;
    return rfq_workspace_status(workspace, 0, st);
}
} // namespace
} // namespace rfq

extern "C" {

const char *rfq_status_string(rfq_status s)
{
    switch (s) {
    case RFQ_OK: return "RFQ_OK";
    case RFQ_ERR_INVALID_ARG: return "RFQ_ERR_INVALID_ARG: null pointer or enum out of range";
    case RFQ_ERR_SHAPE: return "RFQ_ERR_SHAPE: sizes violate the call's constraints";
    case RFQ_ERR_ALIGNMENT: return "RFQ_ERR_ALIGNMENT: device pointer not 16-byte aligned";
    case RFQ_ERR_UNSUPPORTED: return "RFQ_ERR_UNSUPPORTED: combination not implemented";
    case RFQ_ERR_CUDA: return "RFQ_ERR_CUDA: CUDA runtime call or launch failed";
    case RFQ_ERR_TIMEOUT: return "RFQ_ERR_TIMEOUT: a kernel's bounded wait expired";
    case RFQ_ERR_DEVICE: return "RFQ_ERR_DEVICE: current device is not an sm_103 GPU";
    case RFQ_ERR_NONFINITE: return "RFQ_ERR_NONFINITE: the checked input holds an Inf or NaN";
    }
    return "RFQ_ERR_UNKNOWN";
}

rfq_status rfq_qtensor_bytes(int32_t fmt, int32_t scale_layout, int64_t rows, int64_t k, size_t *codes_bytes,
                             size_t *scale_bytes)
{
    if (!codes_bytes || !scale_bytes || !fmt_ok(fmt) || !layout_ok(scale_layout))
        return RFQ_ERR_INVALID_ARG;
    if (rows < 0 || k <= 0 || k % k_granule(fmt, scale_layout) != 0)
        return RFQ_ERR_SHAPE;
    *codes_bytes = (size_t)rows * (size_t)(fmt == RFQ_FMT_MXFP8 ? k : k / 2);
    if (fmt == RFQ_FMT_BF16) {
        *codes_bytes = (size_t)rows * (size_t)k * 2;
        *scale_bytes = 0;
    } else if (fmt == RFQ_FMT_HIF4 && scale_layout == RFQ_SCALE_MMA)
        *scale_bytes = (size_t)((rows + 127) / 128) * 128 * (size_t)(k / 64) * 4;
    else if (fmt == RFQ_FMT_HIF4)
        *scale_bytes = (size_t)rows * (size_t)(k / 64) * 4;
    else if (scale_layout == RFQ_SCALE_MMA)
        *scale_bytes = (size_t)((rows + 127) / 128) * 128 * (size_t)(k / 32);
    else
        *scale_bytes = (size_t)rows * (size_t)(k / 32);
    return RFQ_OK;
}

rfq_status rfq_quantize_weight(const void *w_bf16, int64_t K, int64_t N, rfq_qtensor *out, void *stream)
{
    if (!w_bf16 || !out)
        return RFQ_ERR_INVALID_ARG;
    if (K <= 0 || N < 0)
        return RFQ_ERR_SHAPE;
    rfq_status s = check_qtensor(out, N, K);
    if (s != RFQ_OK)
        return s;
    if (!aligned16(w_bf16))
        return RFQ_ERR_ALIGNMENT;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (N == 0)
        return RFQ_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (out->fmt == RFQ_FMT_MXFP4)
        return from_cuda(launch_weight_quant_mxfp4(w_bf16, K, N, out->codes, out->scales, out->scale_layout, st));
    if (out->fmt == RFQ_FMT_HIF4)
        return from_cuda(launch_weight_quant_hif4(w_bf16, K, N, out->codes, out->scales, out->scale_layout, st));
    if (out->fmt == RFQ_FMT_MXFP8)
        return from_cuda(launch_weight_quant_mxfp8(w_bf16, K, N, out->codes, out->scales, out->scale_layout, st));
    return RFQ_ERR_INVALID_ARG;
}

namespace {
// m16, r16: the GEMM operand forms written in the same pass (HiF4: the bf16
// values of X~ and X^; MXFP4 main with an MXFP8 residual: the MXFP8 codes and
// scales of X~); null for none
rfq_status quantize_act(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb, rfq_qtensor *xq,
                        rfq_qtensor *xr, uint8_t *phi, void *stream, void *m16, void *r16);
} // namespace

rfq_status rfq_quantize_act(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb, rfq_qtensor *xq,
                            rfq_qtensor *xr, uint8_t *phi, void *stream)
{
    return quantize_act(x_bf16, M, K, fb, xq, xr, phi, stream, nullptr, nullptr);
}

rfq_status rfq_quantize_act_expand(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb,
                                   rfq_qtensor *xq, rfq_qtensor *xr, uint8_t *phi, rfq_qtensor *xq_op,
                                   rfq_qtensor *xr_op, void *stream)
{
    const rfq_fallback_mode mode = fb ? (rfq_fallback_mode)fb->mode : RFQ_FALLBACK_ALL;
    if (!xq || !xq_op)
        return RFQ_ERR_INVALID_ARG;
    rfq_status s;
    if (xq->fmt == RFQ_FMT_MXFP4 && xr && xr->fmt == RFQ_FMT_MXFP8) {
        // the FP4-to-FP8 residual: X~ re-encoded as MXFP8 for the E4M3 GEMM;
        // the residual is already MXFP8, so there is no second operand
        if (mode == RFQ_FALLBACK_NONE || xr_op)
            return RFQ_ERR_INVALID_ARG;
        if ((s = check_qtensor(xq_op, M, K)) != RFQ_OK)
            return s;
        if (xq_op->fmt != RFQ_FMT_MXFP8 || xq_op->scale_layout != xq->scale_layout)
            return RFQ_ERR_INVALID_ARG;
        return quantize_act(x_bf16, M, K, fb, xq, xr, phi, stream, xq_op->codes, xq_op->scales);
    }
    if ((mode != RFQ_FALLBACK_NONE && !xr_op) || (mode == RFQ_FALLBACK_NONE && xr_op))
        return RFQ_ERR_INVALID_ARG;
    if (xq->fmt != RFQ_FMT_HIF4)
        return RFQ_ERR_UNSUPPORTED;   // the bf16 operands serve the HiF4 GEMM
    if ((s = check_qtensor(xq_op, M, K)) != RFQ_OK)
        return s;
    if (xq_op->fmt != RFQ_FMT_BF16 || (xr_op && xr_op->fmt != RFQ_FMT_BF16))
        return RFQ_ERR_INVALID_ARG;
    if (xr_op && (s = check_qtensor(xr_op, M, K)) != RFQ_OK)
        return s;
    return quantize_act(x_bf16, M, K, fb, xq, xr, phi, stream, xq_op->codes, xr_op ? xr_op->codes : nullptr);
}

namespace {
rfq_status quantize_act(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb, rfq_qtensor *xq,
                        rfq_qtensor *xr, uint8_t *phi, void *stream, void *m16, void *r16)
{
    rfq_fallback def = {RFQ_FALLBACK_ALL, 0.f, 128, 256};
    const rfq_fallback &f = fb ? *fb : def;
    if (!x_bf16 || !xq)
        return RFQ_ERR_INVALID_ARG;
    if (f.mode < RFQ_FALLBACK_NONE || f.mode > RFQ_FALLBACK_AMAX)
        return RFQ_ERR_INVALID_ARG;
    if (M < 0 || K <= 0)
        return RFQ_ERR_SHAPE;
    rfq_status s = check_qtensor(xq, M, K);
    if (s != RFQ_OK)
        return s;
    const bool res = f.mode != RFQ_FALLBACK_NONE;
    if (res) {
        if (!xr)
            return RFQ_ERR_INVALID_ARG;
        if ((s = check_qtensor(xr, M, K)) != RFQ_OK)
            return s;
        // the residual takes the main pathway's format, or MXFP8 under an
        // MXFP4 main pathway (the FP4-to-FP8 residual of Sec. 4.2)
        const bool fp8_res = xq->fmt == RFQ_FMT_MXFP4 && xr->fmt == RFQ_FMT_MXFP8;
        if ((xr->fmt != xq->fmt && !fp8_res) || xr->scale_layout != xq->scale_layout)
            return RFQ_ERR_INVALID_ARG;
        if (xq->fmt == RFQ_FMT_MXFP8)
            return RFQ_ERR_UNSUPPORTED;   // an MXFP8 main pathway has no residual here
    }
    if (f.p_s < 1 || f.r_s < 32 || f.r_s % 32 != 0 || (xq->fmt == RFQ_FMT_HIF4 && f.r_s % 64 != 0))
        return RFQ_ERR_SHAPE;
    if (xq->fmt == RFQ_FMT_BF16)
        return RFQ_ERR_INVALID_ARG;
    if (f.mode == RFQ_FALLBACK_AMAX && !phi)
        return RFQ_ERR_INVALID_ARG;
    if (!aligned16(x_bf16))
        return RFQ_ERR_ALIGNMENT;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (M == 0)
        return RFQ_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (xq->fmt == RFQ_FMT_MXFP8) {
        if (phi)
            if (cudaError_t e = launch_phi_fill(phi, (M + f.p_s - 1) / f.p_s * ((K + f.r_s - 1) / f.r_s), 0, st))
                return from_cuda(e);
        return from_cuda(launch_act_quant_mxfp8(x_bf16, M, K, xq->codes, xq->scales, xq->scale_layout, st));
    }
    if (res && xr->fmt == RFQ_FMT_MXFP8)
        return from_cuda(launch_act_quant_rfq8(x_bf16, M, K, f.mode, f.tau, f.p_s, f.r_s, xq->codes, xq->scales,
                                               xr->codes, xr->scales, phi, xq->scale_layout, st, m16, r16));
    if (xq->fmt == RFQ_FMT_MXFP4)
        return from_cuda(launch_act_quant_mxfp4(x_bf16, M, K, f.mode, f.tau, f.p_s, f.r_s, xq->codes, xq->scales,
                                                res ? xr->codes : nullptr, res ? xr->scales : nullptr, phi,
                                                xq->scale_layout, st));
    if (xq->fmt == RFQ_FMT_HIF4)
        return from_cuda(launch_act_quant_hif4(x_bf16, M, K, f.mode, f.tau, f.p_s, f.r_s, xq->codes, xq->scales,
                                               res ? xr->codes : nullptr, res ? xr->scales : nullptr, phi,
                                               xq->scale_layout, st, m16, r16));
    return RFQ_ERR_INVALID_ARG;
}
} // namespace

size_t rfq_linear_workspace_bytes(void) { return 256; }

} // extern "C"

namespace rfq {
// The host-side checks of rfq_linear, in its order; *launch is set when the
// call would launch a GEMM (false for M == 0 or N == 0).
rfq_status linear_check(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi, int32_t phi_r_s,
                        const rfq_qtensor *wq, void *y, int32_t out_dtype, void *workspace, bool *launch,
                        bool check_ws)
{
    *launch = false;
    if (!xq || !wq || !y || (check_ws && !workspace))
        return RFQ_ERR_INVALID_ARG;
    if (out_dtype != RFQ_OUT_F32 && out_dtype != RFQ_OUT_BF16)
        return RFQ_ERR_INVALID_ARG;
    const int64_t M = xq->rows, K = xq->k, N = wq->rows;
    if (M < 0 || N < 0 || K <= 0 || wq->k != K)
        return RFQ_ERR_SHAPE;
    rfq_status s = check_qtensor(xq, M, K);
    if (s != RFQ_OK)
        return s;
    if ((s = check_qtensor(wq, N, K)) != RFQ_OK)
        return s;
    if (xr) {
        if ((s = check_qtensor(xr, M, K)) != RFQ_OK)
            return s;
        if (xr->fmt != xq->fmt || xr->scale_layout != xq->scale_layout)
            return RFQ_ERR_INVALID_ARG;
    }
    // operand formats: MXFP4 x MXFP4; MXFP8 x MXFP8 (E4M3, also holding exact
    // re-encodings of MXFP4 tensors); MXFP8 x MXFP4 (W~ multiplied as E2M1,
    // K % 128 == 0, its codes 32-byte aligned); or HiF4 (codes, or their
    // exact bf16 expansion) x the bf16 expansion of W~
    const bool bf16_act = xq->fmt == RFQ_FMT_BF16;
    const bool hif4 = xq->fmt == RFQ_FMT_HIF4 || bf16_act;
    const bool f8 = xq->fmt == RFQ_FMT_MXFP8;
    const bool w4 = f8 && wq->fmt == RFQ_FMT_MXFP4;
    if (hif4 ? wq->fmt != RFQ_FMT_BF16 : (wq->fmt != (f8 ? RFQ_FMT_MXFP8 : RFQ_FMT_MXFP4) && !w4))
        return RFQ_ERR_INVALID_ARG;
    if (w4 && K % 128 != 0)
        return RFQ_ERR_SHAPE;
    if (bf16_act && K % 64 != 0)
        return RFQ_ERR_SHAPE;
    if (N % 16 != 0)
        return RFQ_ERR_SHAPE;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX || K > (int64_t)INT32_MAX)
        return RFQ_ERR_SHAPE;
    if (phi && xr && (hif4 ? (phi_r_s < 64 || phi_r_s % 64 != 0) : (phi_r_s < 128 || phi_r_s % 128 != 0)))
        return RFQ_ERR_SHAPE;
    if (!aligned16(y) || (check_ws && !aligned16(workspace)) ||
        (w4 && (reinterpret_cast<uintptr_t>(wq->codes) & 31u) != 0))
        return RFQ_ERR_ALIGNMENT;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (M == 0 || N == 0)
        return RFQ_OK;
    if (!bf16_act && xq->scale_layout != RFQ_SCALE_MMA)
        return RFQ_ERR_UNSUPPORTED;
    if (!hif4 && wq->scale_layout != RFQ_SCALE_MMA)
        return RFQ_ERR_UNSUPPORTED;
    *launch = true;
    return RFQ_OK;
}
} // namespace rfq

extern "C" {

rfq_status rfq_linear(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi, int32_t phi_r_s,
                      const rfq_qtensor *wq, void *y, int32_t out_dtype, void *workspace, void *stream)
{
    bool launch = false;
    const rfq_status s = linear_check(xq, xr, phi, phi_r_s, wq, y, out_dtype, workspace, &launch, true);
    if (s != RFQ_OK || !launch)
        return s;
    const int64_t M = xq->rows, K = xq->k, N = wq->rows;
    const bool bf16_act = xq->fmt == RFQ_FMT_BF16;
    const bool hif4 = xq->fmt == RFQ_FMT_HIF4 || bf16_act;
    const bool f8 = xq->fmt == RFQ_FMT_MXFP8;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (hif4) {
        GemmHif4Args a;
        a.a_bf16 = bf16_act;
        a.a_codes = xq->codes;
        a.a_meta = xq->scales;
        a.r_codes = xr ? xr->codes : nullptr;
        a.r_meta = xr ? xr->scales : nullptr;
        a.b_bf16 = wq->codes;
        a.phi = xr ? phi : nullptr;
        a.phi_r_s = phi_r_s;
        a.y = y;
        a.out_bf16 = out_dtype == RFQ_OUT_BF16;
        a.M = M;
        a.N = N;
        a.K = K;
        a.status = static_cast<int32_t *>(workspace);
        return gemm_done(launch_gemm_hif4(a, st), workspace, st);
    }
    GemmMxf4Args a;
    a.a_codes = xq->codes;
    a.a_sf = xq->scales;
    a.r_codes = xr ? xr->codes : nullptr;
    a.r_sf = xr ? xr->scales : nullptr;
    a.b_codes = wq->codes;
    a.b_sf = wq->scales;
    a.phi = xr ? phi : nullptr;
    a.phi_r_s = phi_r_s;
    a.y = y;
    a.out_bf16 = out_dtype == RFQ_OUT_BF16;
    a.M = M;
    a.N = N;
    a.K = K;
    a.status = static_cast<int32_t *>(workspace);
    a.f8 = f8;
    a.w4 = f8 && wq->fmt == RFQ_FMT_MXFP4;
    return gemm_done(launch_gemm_mxf4(a, st), workspace, st);
}

} // extern "C"

namespace {
// Workspace of rfq_linear_fused.  M <= 128 (the single-CTA fused kernel):
// the 256-byte GEMM workspace.  M > 128 (the CTA-pair kernel with its
// quantizer): the GEMM workspace, the counters (2 + T + T S + P words for T
// 128-row tiles, S 256-element k-stages and P 256-row blocks), then, each
// 1024-byte aligned, the scratch ring of R = min(kFusedRingPairs, P) slots
// of 256 rows: codes of X~ [256 R][K/2], of X^ [256 R][K/2] (with a
// residual), and their MMA-layout scales [256 R][K/32].
struct FusedLayout {
    size_t ctr, mcodes, rcodes, msf, rsf, total;
    int ring;
};

FusedLayout fused_layout(int64_t M, int64_t K, bool res)
{
    auto up = [](size_t v) { return (v + 1023) & ~size_t(1023); };
    FusedLayout L = {};
    const size_t base = rfq_linear_workspace_bytes();
    if (M <= 128) {
        L.total = base;
        return L;
    }
    const size_t tiles = (size_t)((M + 127) / 128), stages = (size_t)((K / 128 + 1) / 2);
    const size_t pairs = (size_t)((M + 255) / 256);
    L.ring = (int)(pairs < (size_t)kFusedRingPairs ? pairs : (size_t)kFusedRingPairs);
    const size_t rows = (size_t)L.ring * 256;
    const size_t codes = rows * (size_t)(K / 2), sf = rows * (size_t)(K / 32);
    L.ctr = base;
    L.mcodes = up(L.ctr + 4 * (2 + tiles + tiles * stages + pairs));
    L.rcodes = up(L.mcodes + codes);
    L.msf = up(L.rcodes + (res ? codes : 0));
    L.rsf = up(L.msf + sf);
    L.total = up(L.rsf + (res ? sf : 0));
    return L;
}
} // namespace

extern "C" {

size_t rfq_linear_fused_workspace_bytes(int64_t M, int64_t K, const rfq_fallback *fb)
{
    if (M < 0 || K <= 0 || K % 128 != 0)
        return 0;
    return fused_layout(M, K, !fb || fb->mode != RFQ_FALLBACK_NONE).total;
}

rfq_status rfq_linear_fused(const void *x_bf16, int64_t M, int64_t K, const rfq_qtensor *wq,
                            const rfq_fallback *fb, void *y, int32_t out_dtype, void *workspace, void *stream)
{
    if (!x_bf16 || !wq || !y || !workspace)
        return RFQ_ERR_INVALID_ARG;
    if (out_dtype != RFQ_OUT_F32 && out_dtype != RFQ_OUT_BF16)
        return RFQ_ERR_INVALID_ARG;
    const int32_t mode = fb ? fb->mode : RFQ_FALLBACK_ALL;
    if (mode != RFQ_FALLBACK_ALL && mode != RFQ_FALLBACK_NONE && mode != RFQ_FALLBACK_AMAX)
        return RFQ_ERR_INVALID_ARG;
    const int64_t N = wq->rows;
    if (M < 0 || N < 0 || K <= 0 || wq->k != K)
        return RFQ_ERR_SHAPE;
    rfq_status s = check_qtensor(wq, N, K);
    if (s != RFQ_OK)
        return s;
    if (wq->fmt != RFQ_FMT_MXFP4)
        return RFQ_ERR_INVALID_ARG;
    if (K % 128 != 0 || N % 16 != 0)
        return RFQ_ERR_SHAPE;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX || K > (int64_t)INT32_MAX)
        return RFQ_ERR_SHAPE;
    if (!aligned16(x_bf16) || !aligned16(y) || !aligned16(workspace))
        return RFQ_ERR_ALIGNMENT;
    if (mode == RFQ_FALLBACK_AMAX || wq->scale_layout != RFQ_SCALE_MMA)
        return RFQ_ERR_UNSUPPORTED;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (M == 0 || N == 0)
        return RFQ_OK;
    if (M > 128) {
        // CTA pairs, X quantized once into the workspace's scratch by the GEMM's own warps
        const bool res = mode == RFQ_FALLBACK_ALL;
        const FusedLayout L = fused_layout(M, K, res);
        uint8_t *w = static_cast<uint8_t *>(workspace);
        GemmMxf4Args a;
        a.a_codes = w + L.mcodes;
        a.a_sf = w + L.msf;
        a.r_codes = res ? w + L.rcodes : nullptr;
        a.r_sf = res ? w + L.rsf : nullptr;
        a.b_codes = wq->codes;
        a.b_sf = wq->scales;
        a.phi = nullptr;
        a.phi_r_s = 0;
        a.y = y;
        a.out_bf16 = out_dtype == RFQ_OUT_BF16;
        a.M = M;
        a.N = N;
        a.K = K;
        a.status = static_cast<int32_t *>(workspace);
        a.fq_x = x_bf16;
        a.fq_ctr = reinterpret_cast<int32_t *>(w + L.ctr);
        a.fq_ring = L.ring;
        return gemm_done(launch_gemm_mxf4_pair(a, static_cast<cudaStream_t>(stream)), workspace,
                         static_cast<cudaStream_t>(stream));
    }
    GemmFusedArgs a;
    a.x = x_bf16;
    a.b_codes = wq->codes;
    a.b_sf = wq->scales;
    a.y = y;
    a.out_bf16 = out_dtype == RFQ_OUT_BF16;
    a.residual = mode == RFQ_FALLBACK_ALL;
    a.M = M;
    a.N = N;
    a.K = K;
    a.status = static_cast<int32_t *>(workspace);
    return gemm_done(launch_gemm_mxf4_fused(a, static_cast<cudaStream_t>(stream)), workspace,
                         static_cast<cudaStream_t>(stream));
}

rfq_status rfq_linear_mixed(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi, int32_t phi_r_s,
                            const rfq_qtensor *wq, void *y, int32_t out_dtype, void *workspace, void *stream)
{
    if (!xq || !xr || !wq || !y || !workspace)
        return RFQ_ERR_INVALID_ARG;
    if (out_dtype != RFQ_OUT_F32 && out_dtype != RFQ_OUT_BF16)
        return RFQ_ERR_INVALID_ARG;
    if (xq->fmt != RFQ_FMT_MXFP4 || wq->fmt != RFQ_FMT_MXFP4 || xr->fmt != RFQ_FMT_MXFP8)
        return RFQ_ERR_INVALID_ARG;
    const int64_t M = xq->rows, K = xq->k, N = wq->rows;
    if (M < 0 || N < 0 || K <= 0 || wq->k != K)
        return RFQ_ERR_SHAPE;
    rfq_status s;
    if ((s = check_qtensor(xq, M, K)) != RFQ_OK || (s = check_qtensor(xr, M, K)) != RFQ_OK ||
        (s = check_qtensor(wq, N, K)) != RFQ_OK)
        return s;
    if (xq->scale_layout != RFQ_SCALE_MMA || xr->scale_layout != RFQ_SCALE_MMA || wq->scale_layout != RFQ_SCALE_MMA)
        return RFQ_ERR_UNSUPPORTED;
    if (K % 128 != 0 || N % 16 != 0)
        return RFQ_ERR_SHAPE;
    if (M > (int64_t)INT32_MAX || N > (int64_t)INT32_MAX || K > (int64_t)INT32_MAX)
        return RFQ_ERR_SHAPE;
    if (phi && (phi_r_s < 128 || phi_r_s % 128 != 0))
        return RFQ_ERR_SHAPE;
    if (!aligned16(y) || !aligned16(workspace))
        return RFQ_ERR_ALIGNMENT;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (M == 0 || N == 0)
        return RFQ_OK;
    GemmMxf4Args a;
    a.a_codes = xq->codes;
    a.a_sf = xq->scales;
    a.r_codes = xr->codes;
    a.r_sf = xr->scales;
    a.b_codes = wq->codes;
    a.b_sf = wq->scales;
    a.b4_codes = wq->codes;
    a.phi = phi;
    a.phi_r_s = phi_r_s;
    a.y = y;
    a.out_bf16 = out_dtype == RFQ_OUT_BF16;
    a.M = M;
    a.N = N;
    a.K = K;
    a.status = static_cast<int32_t *>(workspace);
    a.f8 = 1;
    return gemm_done(launch_gemm_mxf4_pair(a, static_cast<cudaStream_t>(stream)), workspace,
                     static_cast<cudaStream_t>(stream));
}

rfq_status rfq_linear_profile(const rfq_qtensor *xq, const rfq_qtensor *xr, const rfq_qtensor *wq, void *y,
                              int32_t out_dtype, void *workspace, void *stream)
{
    bool launch = false;
    rfq_status s = linear_check(xq, xr, nullptr, 0, wq, y, out_dtype, workspace, &launch, true);
    if (s != RFQ_OK || !launch)
        return s;
    if (!xr || xq->fmt != RFQ_FMT_MXFP4 || xq->rows <= 128)
        return RFQ_ERR_UNSUPPORTED;
    GemmMxf4Args a;
    a.a_codes = xq->codes;
    a.a_sf = xq->scales;
    a.r_codes = xr->codes;
    a.r_sf = xr->scales;
    a.b_codes = wq->codes;
    a.b_sf = wq->scales;
    a.phi = nullptr;
    a.phi_r_s = 0;
    a.y = y;
    a.out_bf16 = out_dtype == RFQ_OUT_BF16;
    a.M = xq->rows;
    a.N = wq->rows;
    a.K = xq->k;
    a.status = static_cast<int32_t *>(workspace);
    a.prof = 1;
    return gemm_done(launch_gemm_mxf4_pair(a, static_cast<cudaStream_t>(stream)), workspace,
                         static_cast<cudaStream_t>(stream));
}

rfq_status rfq_fp4_mma_peak(int32_t cta_pair, int64_t iters, void *workspace, double *flop_per_launch,
                            void *stream)
{
    if (!workspace || !flop_per_launch || (cta_pair != 0 && cta_pair != 1))
        return RFQ_ERR_INVALID_ARG;
    if (iters < 1 || iters > ((int64_t)1 << 24))
        return RFQ_ERR_SHAPE;
    if (!aligned16(workspace))
        return RFQ_ERR_ALIGNMENT;
    rfq_status s = check_device();
    if (s != RFQ_OK)
        return s;
    return from_cuda(launch_fp4_mma_peak(cta_pair, iters, static_cast<int32_t *>(workspace), flop_per_launch,
                                         static_cast<cudaStream_t>(stream)));
}

rfq_status rfq_debug_bounds(int32_t *line, int32_t clear)
{
#ifdef RFQ_DEBUG_BOUNDS
    if (!line)
        return RFQ_ERR_INVALID_ARG;
    if (cudaDeviceSynchronize() != cudaSuccess)
        return RFQ_ERR_CUDA;
    const int words[2] = {debug_word_quant_mxfp4(clear), debug_word_gemm_mxf4_pair(clear)};
    *line = 0;
    for (int w : words) {
        if (w < 0)
            return RFQ_ERR_CUDA;
        if (w > 0 && *line == 0)
            *line = w;
    }
    return *line ? RFQ_ERR_SHAPE : RFQ_OK;
#else
    (void)clear;
    if (line)
        *line = 0;
    return RFQ_ERR_UNSUPPORTED;
#endif
}

rfq_status rfq_workspace_status(void *workspace, int32_t clear, void *stream)
{
    if (!workspace)
        return RFQ_ERR_INVALID_ARG;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int32_t v = 0;
    if (cudaMemcpyAsync(&v, workspace, sizeof v, cudaMemcpyDeviceToHost, st) != cudaSuccess)
        return RFQ_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess)
        return RFQ_ERR_CUDA;
    if (clear && v != kDevOk) {
        if (cudaMemsetAsync(workspace, 0, sizeof(int32_t), st) != cudaSuccess)
            return RFQ_ERR_CUDA;
    }
    return v == kDevOk ? RFQ_OK
           : v == kDevBadGroups ? RFQ_ERR_SHAPE
           : v == kDevNonFinite ? RFQ_ERR_NONFINITE
                                : RFQ_ERR_TIMEOUT;
}

rfq_status rfq_dequant(const rfq_qtensor *q, void *out, int32_t out_dtype, void *stream)
{
    if (!q || !out || (out_dtype != RFQ_OUT_F32 && out_dtype != RFQ_OUT_BF16))
        return RFQ_ERR_INVALID_ARG;
    rfq_status s = check_qtensor(q, q->rows, q->k);
    if (s != RFQ_OK)
        return s;
    if (q->fmt == RFQ_FMT_BF16)
        return RFQ_ERR_INVALID_ARG;
    if (!aligned16(out))
        return RFQ_ERR_ALIGNMENT;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (q->rows == 0)
        return RFQ_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const bool bf16 = out_dtype == RFQ_OUT_BF16;
    if (q->fmt == RFQ_FMT_HIF4)
        return from_cuda(launch_dequant_hif4(q->codes, q->scales, q->rows, q->k, q->scale_layout, out, bf16, st));
    if (q->fmt == RFQ_FMT_MXFP8)
        return from_cuda(launch_dequant_mxfp8(q->codes, q->scales, q->rows, q->k, q->scale_layout, out, bf16, st));
    if (bf16)
        return from_cuda(launch_dequant_mxfp4_bf16(q->codes, q->scales, q->rows, q->k, q->scale_layout, out, st));
    return from_cuda(
        launch_dequant_mxfp4(q->codes, q->scales, q->rows, q->k, q->scale_layout, static_cast<float *>(out), st));
}

rfq_status rfq_check_finite(const void *x_bf16, int64_t rows, int64_t k, void *workspace, void *stream)
{
    if (!x_bf16 || !workspace)
        return RFQ_ERR_INVALID_ARG;
    if (rows < 0 || k <= 0 || k % 8 != 0)
        return RFQ_ERR_SHAPE;
    if (!aligned16(x_bf16) || !aligned16(workspace))
        return RFQ_ERR_ALIGNMENT;
    rfq_status s = check_device();
    if (s != RFQ_OK)
        return s;
    if (rows == 0)
        return RFQ_OK;
    return from_cuda(launch_check_finite(x_bf16, rows * (k / 8), static_cast<int32_t *>(workspace),
                                         static_cast<cudaStream_t>(stream)));
}

rfq_status rfq_convert(const rfq_qtensor *src, rfq_qtensor *dst, void *stream)
{
    if (!src || !dst)
        return RFQ_ERR_INVALID_ARG;
    rfq_status s = check_qtensor(src, src->rows, src->k);
    if (s != RFQ_OK)
        return s;
    if ((s = check_qtensor(dst, src->rows, src->k)) != RFQ_OK)
        return s;
    if (src->fmt != RFQ_FMT_MXFP4 || dst->fmt != RFQ_FMT_MXFP8 || src->scale_layout != dst->scale_layout)
        return RFQ_ERR_UNSUPPORTED;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (src->rows == 0)
        return RFQ_OK;
    size_t cb = 0, sb = 0;
    if ((s = rfq_qtensor_bytes(src->fmt, src->scale_layout, src->rows, src->k, &cb, &sb)) != RFQ_OK)
        return s;
    return from_cuda(launch_convert_mxfp4_mxfp8(src->codes, src->scales, src->rows, src->k, sb, dst->codes,
                                                dst->scales, static_cast<cudaStream_t>(stream)));
}

rfq_status rfq_linear_grouped(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi, int32_t phi_r_s,
                              const int32_t *group_off, int32_t groups, const rfq_qtensor *wq, int64_t N, void *y,
                              int32_t out_dtype, void *workspace, void *stream)
{
    if (!xq || !wq || !y || !workspace || !group_off)
        return RFQ_ERR_INVALID_ARG;
    if (out_dtype != RFQ_OUT_F32 && out_dtype != RFQ_OUT_BF16)
        return RFQ_ERR_INVALID_ARG;
    if (groups < 1 || groups > 128)
        return RFQ_ERR_SHAPE;
    const int64_t M = xq->rows, K = xq->k;
    if (M < 0 || N <= 0 || K <= 0 || wq->k != K || wq->rows != N * groups)
        return RFQ_ERR_SHAPE;
    rfq_status s = check_qtensor(xq, M, K);
    if (s != RFQ_OK)
        return s;
    if ((s = check_qtensor(wq, wq->rows, K)) != RFQ_OK)
        return s;
    if (xr) {
        if ((s = check_qtensor(xr, M, K)) != RFQ_OK)
            return s;
        if (xr->fmt != xq->fmt || xr->scale_layout != xq->scale_layout)
            return RFQ_ERR_INVALID_ARG;
    }
    const bool f8 = xq->fmt == RFQ_FMT_MXFP8;
    const bool w4 = f8 && wq->fmt == RFQ_FMT_MXFP4;   // W~ multiplied as E2M1
    if ((xq->fmt != RFQ_FMT_MXFP4 && !f8) || (wq->fmt != xq->fmt && !w4))
        return RFQ_ERR_UNSUPPORTED;
    // every group's W~ rows start on a 128-row scale atom and a 16-column Y boundary
    if (N % 128 != 0 || K % 128 != 0)
        return RFQ_ERR_SHAPE;
    if (M > (int64_t)INT32_MAX || N * groups > (int64_t)INT32_MAX || K > (int64_t)INT32_MAX)
        return RFQ_ERR_SHAPE;
    if (phi && xr && (phi_r_s < 128 || phi_r_s % 128 != 0))
        return RFQ_ERR_SHAPE;
    if (!aligned16(y) || !aligned16(workspace) || !aligned16(group_off) ||
        (w4 && (reinterpret_cast<uintptr_t>(wq->codes) & 31u) != 0))
        return RFQ_ERR_ALIGNMENT;
    if (xq->scale_layout != RFQ_SCALE_MMA || wq->scale_layout != RFQ_SCALE_MMA)
        return RFQ_ERR_UNSUPPORTED;
    if ((s = check_device()) != RFQ_OK)
        return s;
    if (M == 0)
        return RFQ_OK;
    GemmMxf4Args a;
    a.a_codes = xq->codes;
    a.a_sf = xq->scales;
    a.r_codes = xr ? xr->codes : nullptr;
    a.r_sf = xr ? xr->scales : nullptr;
    a.b_codes = wq->codes;
    a.b_sf = wq->scales;
    a.phi = xr ? phi : nullptr;
    a.phi_r_s = phi_r_s;
    a.y = y;
    a.out_bf16 = out_dtype == RFQ_OUT_BF16;
    a.M = M;
    a.N = N;
    a.K = K;
    a.status = static_cast<int32_t *>(workspace);
    a.f8 = f8;
    a.w4 = w4;
    a.group_off = group_off;
    a.groups = groups;
    return gemm_done(launch_gemm_mxf4(a, static_cast<cudaStream_t>(stream)), workspace,
                     static_cast<cudaStream_t>(stream));
}

} // extern "C"
