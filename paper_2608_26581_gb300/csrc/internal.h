// internal.h -- launchers shared between the C-ABI layer and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "../../include/rfq.h"

namespace rfq {

// ---- the debug build (compiled with -DRFQ_DEBUG_BOUNDS, librfq_debug.so):
// every direct global store of the kernels that carry these checks tests
// its index against its buffer's extent; an out-of-range store is skipped
// and the source line of the first one is kept in the translation unit's
// debug word (RFQ_DEBUG_WORD_DECL), which rfq_debug_bounds reads.  In the
// normal build the checks compile to nothing.
__device__ __forceinline__ bool debug_in_bounds(int64_t i, int64_t n, int line, int *word)
{
    if (i >= 0 && i < n)
        return true;
    atomicCAS(word, 0, line);
    return false;
}
#ifdef RFQ_DEBUG_BOUNDS
#define RFQ_DEBUG_WORD_DECL static __device__ int g_rfq_debug_word = 0;
#define RFQ_IN_BOUNDS(i, n) ::rfq::debug_in_bounds((int64_t)(i), (int64_t)(n), __LINE__, &g_rfq_debug_word)
#define RFQ_DEBUG_WORD_ACCESSOR(fn)                                                                               \
    int fn(int clear)                                                                                             \
    {                                                                                                             \
        int v = 0;                                                                                                \
        if (cudaMemcpyFromSymbol(&v, g_rfq_debug_word, sizeof v) != cudaSuccess)                                  \
            return -1;                                                                                            \
        if (clear) {                                                                                              \
            const int z = 0;                                                                                      \
            if (cudaMemcpyToSymbol(g_rfq_debug_word, &z, sizeof z) != cudaSuccess)                                \
                return -1;                                                                                        \
        }                                                                                                         \
        return v;                                                                                                 \
    }
#else
#define RFQ_DEBUG_WORD_DECL
#define RFQ_IN_BOUNDS(i, n) true
#define RFQ_DEBUG_WORD_ACCESSOR(fn)                                                                               \
    int fn(int) { return 0; }
#endif
// Each translation unit with bounds checks: its debug word (the source line
// of the first out-of-range store, 0 if none; -1 if it cannot be read).
int debug_word_quant_mxfp4(int clear);
int debug_word_gemm_mxf4_pair(int clear);

// Device status word values written into a workspace by kernels.
constexpr int32_t kDevOk = 0;
constexpr int32_t kDevTimeout = 1;
constexpr int32_t kDevBadGroups = 2;   // grouped GEMM: device-side row offsets break the contract
constexpr int32_t kDevNonFinite = 3;   // rfq_check_finite found an Inf or NaN

// Bounded waits in the GEMM give up after this many nanoseconds.
constexpr uint64_t kWaitLimitNs = 2000000000ull;

// Words (int32) of a GEMM call's workspace, zeroed by the caller:
//   [kWsStatus] device status (kDevOk, kDevTimeout, ...), sticky;
//   [kWsWaitUs] limit of this call's bounded waits in microseconds
//               (0: kWaitLimitNs);
//   [kWsHold]   held start: when non-zero, each TMA producer waits (bounded)
//               for word [kWsOpen] to become non-zero before its first copy,
//               so a caller can make a wait run out with no copy or MMA in
//               flight and check the kernel's timeout path.
constexpr int kWsStatus = 0, kWsWaitUs = 1, kWsHold = 2, kWsOpen = 3;

// The wait limit a workspace asks for.
__device__ __forceinline__ uint64_t ws_wait_limit_ns(const int32_t *ws)
{
    const int32_t us = reinterpret_cast<const volatile int32_t *>(ws)[kWsWaitUs];
    return us > 0 ? (uint64_t)us * 1000ull : kWaitLimitNs;
}

// Byte offset of E8M0 scale (row m, 32-element block b) in the MMA layout
// (512-byte atoms of 128 rows x 4 blocks; kc = K / 128 atoms per row band).
__host__ __device__ inline int64_t sf_mma_offset(int64_t m, int64_t b, int64_t kc)
{
    return (((m >> 7) * kc + (b >> 2)) << 9) + ((m & 31) << 4) + (((m >> 5) & 3) << 2) + (b & 3);
}

// ---- MXFP8 (E4M3) quantization and the FP4-to-FP8 residual (quant_mxfp8.cu)
cudaError_t launch_act_quant_mxfp8(const void *x, int64_t M, int64_t K, void *codes, void *scales, int layout,
                                   cudaStream_t st);
// m8codes / m8scales (may be null): X~ re-encoded as MXFP8 in the same pass
cudaError_t launch_act_quant_rfq8(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                  void *mcodes, void *mscales, void *rcodes, void *rscales, uint8_t *phi, int layout,
                                  cudaStream_t st, void *m8codes = nullptr, void *m8scales = nullptr);
cudaError_t launch_weight_quant_mxfp8(const void *w, int64_t K, int64_t N, void *codes, void *scales, int layout,
                                      cudaStream_t st);
cudaError_t launch_convert_mxfp4_mxfp8(const void *src_codes, const void *src_scales, int64_t rows, int64_t k,
                                       size_t scale_bytes, void *dst_codes, void *dst_scales, cudaStream_t st);
cudaError_t launch_dequant_mxfp8(const void *codes, const void *scales, int64_t rows, int64_t k, int layout, void *out,
                                 bool bf16, cudaStream_t st);

// ---- input check (quant_mxfp4.cu): records kDevNonFinite if x holds an Inf / NaN
cudaError_t launch_check_finite(const void *x, int64_t n8, int32_t *status, cudaStream_t st);

// ---- MXFP4 quantization (quant_mxfp4.cu)
// Activation: main (+ residual) codes and scales in one pass over X.
cudaError_t launch_act_quant_mxfp4(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                   void *mcodes, void *mscales, void *rcodes, void *rscales, uint8_t *phi,
                                   int layout, cudaStream_t st);
// phi(p, r) tiles: amax > tau, or a constant (0 / 1)
cudaError_t launch_phi_amax(const void *x, int64_t M, int64_t K, int p_s, int r_s, float tau, uint8_t *phi,
                            cudaStream_t st);
cudaError_t launch_phi_fill(uint8_t *phi, int64_t n, int value, cudaStream_t st);
cudaError_t launch_weight_quant_mxfp4(const void *w, int64_t K, int64_t N, void *codes, void *scales, int layout,
                                      cudaStream_t st);
cudaError_t launch_dequant_mxfp4(const void *codes, const void *scales, int64_t rows, int64_t k, int layout,
                                 float *out, cudaStream_t st);

// ---- MXFP4 RFQ GEMM (gemm_mxf4.cu)
struct GemmMxf4Args {
    const void *a_codes, *r_codes, *b_codes;   // [M][K/2], [M][K/2] or null, [N][K/2] (f8: [..][K] E4M3)
    const void *a_sf, *r_sf, *b_sf;            // MMA-layout scales
    const uint8_t *phi;                        // [ceil(M/128)][K/phi_r_s] or null
    int phi_r_s;
    void *y;
    int out_bf16;
    int64_t M, N, K;
    int32_t *status;
    int f8 = 0;                                // every operand MXFP8 (E4M3): kind::mxf8f6f4, CTA pairs
    int w4 = 0;                                // with f8: W~ MXFP4 [N][K/2] (32-byte aligned), multiplied
                                               // as E2M1 (E4M3 x E2M1 MMAs) from the padded 4-bit form
    const int32_t *group_off = nullptr;        // grouped GEMM: device row offsets [groups + 1]
    int groups = 0;                            // grouped GEMM: N is per group, W~ has groups * N rows
    // fused quantizer (CTA-pair kernel): bf16 X [M][K]; the kernel quantizes
    // it into a_codes / a_sf (and r_codes / r_sf) itself, a ring of fq_ring
    // slots of 256 rows, and counts finished units in fq_ctr (zero on entry,
    // left zero on exit)
    const void *fq_x = nullptr;
    int32_t *fq_ctr = nullptr;
    int fq_ring = 0;                           // fused quantizer: 256-row slots of the scratch ring
    int prof = 0;                              // CTA-pair kernel: the MMA thread's counters (rfq_linear_profile)
    // mixed-rate FP4-to-FP8 residual (CTA-pair kernel): W~ packed [N][K/2]
    // (32-byte aligned); a_codes / a_sf are then X~ packed, r_codes / r_sf
    // X^ as E4M3, b_sf W~'s scales (b_codes unused)
    const void *b4_codes = nullptr;
};

// Slots of 256 rows in the fused quantizer's scratch ring (rfq_linear_fused).
constexpr int kFusedRingPairs = 12;
cudaError_t launch_gemm_mxf4(const GemmMxf4Args &a, cudaStream_t st);
// CTA-pair kernel (gemm_mxf4_pair.cu), used by launch_gemm_mxf4 when M > 128.
cudaError_t launch_gemm_mxf4_pair(const GemmMxf4Args &a, cudaStream_t st);

// ---- RFQ linear with the quantizer fused into the GEMM (gemm_mxf4_fused.cu)
struct GemmFusedArgs {
    const void *x;                 // bf16 [M][K]
    const void *b_codes, *b_sf;    // MXFP4 weight, MMA-layout scales
    void *y;
    int out_bf16;
    int residual;                  // 1: phi = 1 everywhere, 0: plain W4A4
    int64_t M, N, K;
    int32_t *status;
};
cudaError_t launch_gemm_mxf4_fused(const GemmFusedArgs &a, cudaStream_t st);

// ---- HiF4 quantization (quant_hif4.cu); metadata layout RFQ_SCALE_MMA is
// block-major [K/64][rows rounded up to 128]
// phi: computed (AMAX) or filled (other modes) here when given; m16 / r16
// (may be null): bf16 [M][K] receiving the exact values of X~ / X^
cudaError_t launch_act_quant_hif4(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                  void *mcodes, void *mmeta, void *rcodes, void *rmeta, uint8_t *phi, int layout,
                                  cudaStream_t st, void *m16 = nullptr, void *r16 = nullptr);
cudaError_t launch_weight_quant_hif4(const void *w, int64_t K, int64_t N, void *codes, void *meta, int layout,
                                     cudaStream_t st);
cudaError_t launch_dequant_hif4(const void *codes, const void *meta, int64_t rows, int64_t k, int layout,
                                void *out, bool bf16, cudaStream_t st);
cudaError_t launch_dequant_mxfp4_bf16(const void *codes, const void *scales, int64_t rows, int64_t k, int layout,
                                      void *out, cudaStream_t st);

// ---- HiF4 RFQ GEMM (gemm_hif4.cu)
struct GemmHif4Args {
    bool a_bf16;                     // activations given as exact bf16 expansions [M][K]
    const void *a_codes, *r_codes;   // [M][K/2] HiF4 codes (or bf16 [M][K]); r_codes may be null
    const void *a_meta, *r_meta;     // block-major [K/64][Mpad] metadata words
    const void *b_bf16;              // exact bf16 expansion of W~, [N][K]
    const uint8_t *phi;
    int phi_r_s;
    void *y;
    int out_bf16;
    int64_t M, N, K;
    int32_t *status;
};
cudaError_t launch_gemm_hif4(const GemmHif4Args &a, cudaStream_t st);

// ---- tensor maps (api.cu)
// swizzle: 0 none, 64 or 128 (bytes)
bool encode_tmap_2d_u8(CUtensorMap *map, const void *base, uint64_t inner_bytes, uint64_t rows,
                       uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows, int swizzle);
// Packed E2M1 codes [rows x k] (k % 128 == 0, base 32-byte aligned) loaded
// in 128-code boxes as the padded 4-bit form that kind::mxf8f6f4 reads (16
// codes in 8 bytes, then 8 bytes of gap: 128-byte rows), 128-byte swizzle.
// A box's copy counts the 64 bytes per row it reads toward complete_tx.
bool encode_tmap_2d_e2m1_padded(CUtensorMap *map, const void *base, uint64_t k, uint64_t rows,
                                uint32_t box_rows);

// ---- the dense FP4 MMA rate alone (mma_peak.cu): `iters` MMAs per SM (pair
// = 0, 128 x 256 x 64) or per CTA pair (pair = 1, 256 x 256 x 64); *flop =
// the launch's MMA work
cudaError_t launch_fp4_mma_peak(int pair, int64_t iters, int32_t *status, double *flop, cudaStream_t st);

// rfq_linear's host-side checks (api.cu): RFQ_OK with *launch set when the
// call would launch a GEMM, else the status rfq_linear returns; check_ws =
// false leaves the workspace pointer out of the checks.
rfq_status linear_check(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi, int32_t phi_r_s,
                        const rfq_qtensor *wq, void *y, int32_t out_dtype, void *workspace, bool *launch,
                        bool check_ws);

// Blocks of `threads` threads (and `smem` dynamic shared bytes) of `kern`
// resident on one SM at once (cached per kernel): grid-stride kernels launch
// at most that many per SM, so no partial second wave trails the first.
int resident_blocks_per_sm(const void *kern, int threads, size_t smem);

// Number of SMs of the current device (cached).
int num_sms();

} // namespace rfq
