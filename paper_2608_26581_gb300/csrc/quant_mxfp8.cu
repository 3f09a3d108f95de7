// quant_mxfp8.cu -- MXFP8 (E4M3) quantizers (Sec. 3.2.1 with the block rule
// of Sec. 3.2 Eqs. 3-4) and the FP4-to-FP8 residual pathway (Sec. 4.2,
// Sec. 4.3):
//   act_quant_mxfp8      X -> E4M3 codes + E8M0 scales (W4A8 / W8A8 activations)
//   act_quant_rfq8       X~ = Q_MXFP4(X) and X^ = Q_MXFP8(X - X~) in one pass,
//                        optionally with X~ re-encoded as MXFP8
//   weight_quant_mxfp8   W [K x N] -> K-major E4M3 codes + scales
//   convert_mxfp4_mxfp8  MXFP4 codes -> E4M3 codes of the same values (exact:
//                        every E2M1 value is an E4M3 value), scales unchanged
//   dequant_mxfp8        codes x scales -> fp32 or bf16
// The E8M0 byte of an E4M3 block is the fp32 exponent field of its amax
// minus 8 (floor(log2 amax) - 8, clamped at 0); x 2^-e is exact, and
// cvt.rn.satfinite.e4m3x2 rounds to nearest even and saturates at +-448.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cstdint>

#include "internal.h"
#include "mxfp4_math.cuh"

namespace rfq {
namespace {

template <int LAYOUT>
__device__ __forceinline__ int64_t scale_index8(int64_t m, int64_t b, int64_t kblocks)
{
    if (LAYOUT == RFQ_SCALE_MMA)
        return sf_mma_offset(m, b, kblocks >> 2);
    return m * kblocks + b;
}

// E8M0 byte of an E4M3 block from the fp32 bits of its amax.
__device__ __forceinline__ int scale8_byte_from_f32_bits(uint32_t amax_bits)
{
    return max((int)((amax_bits >> 23) & 0xFF) - 8, 0);
}

// Eight fp32 values -> eight E4M3 codes (element i in byte i).
__device__ __forceinline__ uint2 e4m3x8(const float (&y)[8])
{
    uint32_t lo, hi;
    asm("{\n\t.reg .b16 h0, h1, h2, h3;\n\t"
        "cvt.rn.satfinite.e4m3x2.f32 h0, %3, %2;\n\t"
        "cvt.rn.satfinite.e4m3x2.f32 h1, %5, %4;\n\t"
        "cvt.rn.satfinite.e4m3x2.f32 h2, %7, %6;\n\t"
        "cvt.rn.satfinite.e4m3x2.f32 h3, %9, %8;\n\t"
        "mov.b32 %0, {h0, h1};\n\t"
        "mov.b32 %1, {h2, h3};\n\t}"
        : "=r"(lo), "=r"(hi)
        : "f"(y[0]), "f"(y[1]), "f"(y[2]), "f"(y[3]), "f"(y[4]), "f"(y[5]), "f"(y[6]), "f"(y[7]));
    return make_uint2(lo, hi);
}

// Two E4M3 codes (a 16-bit pair) -> two floats (exact through f16).
__device__ __forceinline__ void e4m3x2_decode(uint32_t pair, float &a, float &b)
{
    uint32_t h;
    asm("{\n\t.reg .b16 p;\n\tcvt.u16.u32 p, %1;\n\tcvt.rn.f16x2.e4m3x2 %0, p;\n\t}" : "=r"(h) : "r"(pair));
    const __half2 v = *reinterpret_cast<const __half2 *>(&h);
    a = __low2float(v);
    b = __high2float(v);
}

// Block-max of this lane's eight values over the four lanes of its block.
__device__ __forceinline__ float block_amax(const float (&v)[8])
{
    float am = absmax8(v);
    am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 1));
    return fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 2));
}

// E4M3 codes and E8M0 byte of this lane's eight values (its block spans
// four lanes; all 32 lanes take part).
__device__ __forceinline__ uint2 mxfp8_quant8(const float (&xf)[8], int &sb)
{
    sb = scale8_byte_from_f32_bits(__float_as_uint(block_amax(xf)));
    const float inv = pow2_neg_e(sb);
    float y[8];
#pragma unroll
    for (int i = 0; i < 8; ++i)
        y[i] = xf[i] * inv;
    return e4m3x8(y);
}

constexpr int kSeg = 1024;   // elements per (row, segment) item of a warp
constexpr int kU = kSeg / 256;

// One warp per (row, 1024-element segment); four lanes per 32-element block.
// RFQ8 = false: X -> MXFP8.  RFQ8 = true: X -> MXFP4 main codes and the
// MXFP8 residual X - X~ (zero on phi = 0 tiles when PHI); with OP also X~
// re-encoded as MXFP8 (the E4M3 code of each E2M1 value, which is exact,
// under the same scale byte), the operand the E4M3 GEMM multiplies.
template <bool RFQ8, bool PHI, int LAYOUT, bool OP = false>
__global__ void __launch_bounds__(256) act_quant8_kernel(const uint4 *__restrict__ x, int64_t M, int64_t K,
                                                        uint8_t *__restrict__ mcodes, uint8_t *__restrict__ mscales,
                                                        uint8_t *__restrict__ rcodes, uint8_t *__restrict__ rscales,
                                                        const uint8_t *__restrict__ phi, int p_s, int r_s,
                                                        int64_t pad_rows, uint8_t *__restrict__ m8codes = nullptr,
                                                        uint8_t *__restrict__ m8scales = nullptr)
{
    const int lane = threadIdx.x & 31;
    const int kchunks = (int)(K >> 3);
    const int kblocks = (int)(K >> 5);
    const int segs = (kchunks + kSeg / 8 - 1) / (kSeg / 8);
    const int64_t items = M * segs;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

    if (LAYOUT == RFQ_SCALE_MMA && pad_rows > 0) {
        const int64_t n = pad_rows * kblocks;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
            const int64_t off = scale_index8<LAYOUT>(M + i / kblocks, i % kblocks, kblocks);
            mscales[off] = 0;
            if (RFQ8)
                rscales[off] = 0;
            if (OP)
                m8scales[off] = 0;
        }
    }

    for (int64_t it = gwarp; it < items; it += nwarps) {
        const int64_t m = it / segs;
        const int c0 = (int)(it - m * segs) * (kSeg / 8);
        const uint4 *xr = x + m * kchunks;
        uint4 v[kU];
#pragma unroll
        for (int j = 0; j < kU; ++j) {
            const int c = c0 + j * 32 + lane;
            v[j] = c < kchunks ? __ldcs(xr + c) : make_uint4(0, 0, 0, 0);
        }
        const uint8_t *prow = PHI ? phi + (m / p_s) * ((K + r_s - 1) / r_s) : nullptr;
#pragma unroll
        for (int j = 0; j < kU; ++j) {
            const int c = c0 + j * 32 + lane;
            const bool ok = c < kchunks; // uniform over each group of 4 lanes
            const int64_t soff = scale_index8<LAYOUT>(m, c >> 2, kblocks);
            float xf[8];
            bf16x8_to_f32(v[j], xf);
            if (!RFQ8) {
                int sb;
                const uint2 q = mxfp8_quant8(xf, sb);
                if (ok) {
                    *reinterpret_cast<uint2 *>(mcodes + m * K + (int64_t)c * 8) = q;
                    if ((lane & 3) == 0)
                        mscales[soff] = (uint8_t)sb;
                }
            } else {
                const Mx8 q4 = mxfp4_quant8<false>(xf);
                // the residual x - x~, exact in fp32
                float q[8], r[8];
                e2m1x8_decode(q4.code, q);
                const float sc = pow2_e(q4.sb);
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    r[i] = fmaf(-q[i], sc, xf[i]);
                int rb;
                const uint2 rq = mxfp8_quant8(r, rb);
                const bool on = !PHI || (ok && prow[(c * 8) / r_s] != 0);
                if (ok) {
                    reinterpret_cast<uint32_t *>(mcodes + m * (K >> 1))[c] = q4.code;
                    *reinterpret_cast<uint2 *>(rcodes + m * K + (int64_t)c * 8) = on ? rq : make_uint2(0, 0);
                    if (OP)
                        *reinterpret_cast<uint2 *>(m8codes + m * K + (int64_t)c * 8) = e4m3x8(q);
                    if ((lane & 3) == 0) {
                        mscales[soff] = (uint8_t)q4.sb;
                        rscales[soff] = on ? (uint8_t)rb : 0;
                        if (OP)
                            m8scales[soff] = (uint8_t)q4.sb;
                    }
                }
            }
        }
    }
}

// The FP4-to-FP8 quantizer (no phi, or phi given) with one lane per
// 32-element block, as act_quant_mxfp4_kernel: X~ = Q_MXFP4(X)
// (mxfp4_quant32), the residual x - x~ exactly (one FMA per element) and
// X^ = Q_MXFP8 of it.  A lane reads its block's 64 bytes in two 32-byte
// loads and writes 16 bytes of X~ codes and 32 of X^; no shuffles.
template <bool PHI, int LAYOUT>
__global__ void __launch_bounds__(256) act_quant_rfq8_kernel(const uint4 *__restrict__ x, int64_t M, int64_t K,
                                                            uint8_t *__restrict__ mcodes,
                                                            uint8_t *__restrict__ mscales,
                                                            uint8_t *__restrict__ rcodes,
                                                            uint8_t *__restrict__ rscales,
                                                            const uint8_t *__restrict__ phi, int p_s, int r_s,
                                                            int64_t pad_rows)
{
    const int lane = threadIdx.x & 31;
    const int kblocks = (int)(K >> 5);
    const int segs = (kblocks + 31) / 32;
    const int64_t items = M * segs;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

    if (LAYOUT == RFQ_SCALE_MMA && pad_rows > 0) {
        const int64_t n = pad_rows * kblocks;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
            const int64_t off = scale_index8<LAYOUT>(M + i / kblocks, i % kblocks, kblocks);
            mscales[off] = 0;
            rscales[off] = 0;
        }
    }

    uint4 *mc4 = reinterpret_cast<uint4 *>(mcodes);
    uint4 *rc4 = reinterpret_cast<uint4 *>(rcodes);
    const int phi_cols = PHI ? (int)((K + r_s - 1) / r_s) : 0;
    for (int64_t it = gwarp; it < items; it += nwarps) {
        const int64_t m = it / segs;
        const int b = (int)(it - m * segs) * 32 + lane;   // this lane's block
        const bool ok = b < kblocks;
        uint32_t w[16];
        if (ok) {
            const uint4 *p = x + m * (K >> 3) + (int64_t)b * 4;
            uint32_t t0[8], t1[8];
            ldg256_stream(p, t0);
            ldg256_stream(p + 2, t1);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                w[i] = t0[i];
                w[8 + i] = t1[i];
            }
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                w[i] = 0;
        }
        float xf[32];
        bf16x32_to_f32(w, xf);
        const Mx32 q4 = mxfp4_quant32<false>(xf);
        const float sc = pow2_e(q4.sb);
        const uint32_t cw[4] = {q4.code.x, q4.code.y, q4.code.z, q4.code.w};
        float r[32];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            float qg[8];
            e2m1x8_decode(cw[g], qg);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                r[8 * g + i] = fmaf(-qg[i], sc, xf[8 * g + i]); // x - x~, exact
        }
        const int rb = scale8_byte_from_f32_bits(__float_as_uint(absmax32(r)));
        const float inv = pow2_neg_e(rb);
        uint2 rq[4];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            float y[8];
#pragma unroll
            for (int i = 0; i < 8; ++i)
                y[i] = r[8 * g + i] * inv;
            rq[g] = e4m3x8(y);
        }
        if (!ok)
            continue;
        const bool on = !PHI || phi[(m / p_s) * phi_cols + (b * 32) / r_s] != 0;
        const int64_t soff = scale_index8<LAYOUT>(m, b, kblocks);
        const int64_t blk = m * kblocks + b;
        mc4[blk] = q4.code;
        mscales[soff] = (uint8_t)q4.sb;
        rc4[2 * blk] = on ? make_uint4(rq[0].x, rq[0].y, rq[1].x, rq[1].y) : make_uint4(0, 0, 0, 0);
        rc4[2 * blk + 1] = on ? make_uint4(rq[2].x, rq[2].y, rq[3].x, rq[3].y) : make_uint4(0, 0, 0, 0);
        rscales[soff] = on ? (uint8_t)rb : 0;
    }
}

// The FP4-to-FP8 quantizer with AMAX phi on 128 x 256 tiles (Sec. 4.3),
// fused as act_quant_mxfp4_amax_kernel: one 256-thread block per tile
// stages its 64 KB in shared memory with cp.async (warp w rows 16w .. 16w +
// 15, lane l the l-th 16-byte chunk of each), reduces max |x| (packed
// bf16x2 max, NaN dropped, as phi_amax_kernel), writes phi, then writes X~
// (MXFP4; with OP also as MXFP8) and, on a phi = 1 tile, the MXFP8
// residual (zeros otherwise, without computing it).  X is read once.
__device__ __forceinline__ void cp_async16_zfill(uint32_t saddr, const void *g, uint32_t src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(saddr), "l"(g), "r"(src_bytes) : "memory");
}

__device__ __forceinline__ uint4 lds128(uint32_t saddr)
{
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(saddr)
                 : "memory");
    return v;
}

template <int LAYOUT, bool OP>
__global__ void __launch_bounds__(256, 3) act_quant_rfq8_amax_kernel(const uint4 *__restrict__ x, int64_t M,
                                                                    int64_t K, uint8_t *__restrict__ mcodes,
                                                                    uint8_t *__restrict__ mscales,
                                                                    uint8_t *__restrict__ rcodes,
                                                                    uint8_t *__restrict__ rscales,
                                                                    uint8_t *__restrict__ phi, float tau,
                                                                    uint8_t *__restrict__ m8codes,
                                                                    uint8_t *__restrict__ m8scales)
{
    constexpr int R = 16, NW = 8;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t kchunks = K >> 3;
    const int kblocks = (int)(K >> 5);
    const int nr = (int)(K >> 8);
    const int64_t tile = blockIdx.x;
    const int64_t p = tile / nr;
    const int r = (int)(tile - p * nr);
    const int64_t m0 = p * 128 + warp * R;
    const int c = r * 32 + lane;
    extern __shared__ __align__(16) uint8_t tile_smem[];
    // this thread's row i sits at sbase + 512 i; no other thread reads it
    const uint32_t sbase = (uint32_t)__cvta_generic_to_shared(tile_smem) + (uint32_t)(((warp * R) * 32 + lane) * 16);
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const bool ok = m0 + i < M; // rows past M are zero-filled, not read
        cp_async16_zfill(sbase + 512 * i, ok ? x + (m0 + i) * kchunks + c : x, ok ? 16u : 0u);
    }
    asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
    uint32_t acc = 0;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const uint4 vi = lds128(sbase + 512 * i);
        const uint32_t q[4] = {vi.x, vi.y, vi.z, vi.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
            asm("max.bf16x2 %0, %1, %2;" : "=r"(acc) : "r"(acc), "r"(q[j] & 0x7fff7fffu));
    }
    const float am = fmaxf(__uint_as_float(acc << 16), __uint_as_float(acc & 0xffff0000u));
    __shared__ uint32_t red[NW];
    const uint32_t wmax = __reduce_max_sync(0xFFFFFFFFu, __float_as_uint(am)); // am >= 0: integer order
    if (lane == 0)
        red[warp] = wmax;
    __syncthreads();
    uint32_t tmax = red[0];
#pragma unroll
    for (int i = 1; i < NW; ++i)
        tmax = max(tmax, red[i]);
    const bool on = __uint_as_float(tmax) > tau;
    if (threadIdx.x == 0)
        phi[tile] = on ? 1 : 0;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const int64_t m = m0 + i; // uniform over the warp
        const int64_t soff = scale_index8<LAYOUT>(m, c >> 2, kblocks);
        if (m >= M) {
            if (LAYOUT == RFQ_SCALE_MMA && (lane & 3) == 0) {
                // rows M .. of the last tile are the layout's padding rows
                mscales[soff] = 0;
                rscales[soff] = 0;
                if (OP)
                    m8scales[soff] = 0;
            }
            continue;
        }
        float xf[8];
        bf16x8_to_f32(lds128(sbase + 512 * i), xf);
        const Mx8 q4 = mxfp4_quant8<false>(xf);
        float q[8];
        e2m1x8_decode(q4.code, q);
        reinterpret_cast<uint32_t *>(mcodes + m * (K >> 1))[c] = q4.code;
        if (OP)
            *reinterpret_cast<uint2 *>(m8codes + m * K + (int64_t)c * 8) = e4m3x8(q);
        uint2 rq = make_uint2(0, 0);
        int rb = 0;
        if (on) {
            // the residual x - x~, exact in fp32
            const float sc = pow2_e(q4.sb);
            float rr[8];
#pragma unroll
            for (int k = 0; k < 8; ++k)
                rr[k] = fmaf(-q[k], sc, xf[k]);
            rq = mxfp8_quant8(rr, rb);
        }
        *reinterpret_cast<uint2 *>(rcodes + m * K + (int64_t)c * 8) = rq;
        if ((lane & 3) == 0) {
            mscales[soff] = (uint8_t)q4.sb;
            rscales[soff] = (uint8_t)rb;
            if (OP)
                m8scales[soff] = (uint8_t)q4.sb;
        }
    }
}

// One thread per (column n, 32-block b) of W [K x N].
template <int LAYOUT>
__global__ void __launch_bounds__(256) weight_quant_mxfp8_kernel(const __nv_bfloat16 *__restrict__ w, int64_t K,
                                                                int64_t N, int64_t Npad, uint8_t *__restrict__ codes,
                                                                uint8_t *__restrict__ scales)
{
    const int64_t kblocks = K >> 5;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t n = t % Npad, b = t / Npad;
    if (b >= kblocks)
        return;
    if (n >= N) {
        if (LAYOUT == RFQ_SCALE_MMA)
            scales[scale_index8<LAYOUT>(n, b, kblocks)] = 0;
        return;
    }
    float xf[32];
    uint32_t am = 0;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        const uint16_t bits = __bfloat16_as_ushort(w[(b * 32 + i) * N + n]);
        am = max(am, (uint32_t)(bits & 0x7FFF));
        xf[i] = __uint_as_float((uint32_t)bits << 16);
    }
    const int sb = scale8_byte_from_f32_bits(am << 16);
    const float inv = pow2_neg_e(sb);
    uint4 *dst = reinterpret_cast<uint4 *>(codes + n * K + b * 32);
#pragma unroll
    for (int g = 0; g < 2; ++g) {
        float y0[8], y1[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            y0[i] = xf[g * 16 + i] * inv;
            y1[i] = xf[g * 16 + 8 + i] * inv;
        }
        const uint2 a = e4m3x8(y0), c = e4m3x8(y1);
        dst[g] = make_uint4(a.x, a.y, c.x, c.y);
    }
    scales[scale_index8<LAYOUT>(n, b, kblocks)] = (uint8_t)sb;
}

// E2M1 code -> E4M3 code of the same value: sign moves to bit 7; the
// magnitudes 0, 0.5, 1, 1.5, 2, 3, 4, 6 are 0x00, 0x30, 0x38, 0x3C, 0x40,
// 0x44, 0x48, 0x4C (exponent field e + 7, mantissa m / 8).
__device__ __forceinline__ uint32_t e2m1_to_e4m3(uint32_t c)
{
    const uint32_t mag = c & 7u;
    uint32_t code = 0;
    if (mag == 1)
        code = 6u << 3;                                            // 0.5 = 2^-1
    else if (mag >= 2)
        code = (((mag >> 1) + 6u) << 3) | ((mag & 1u) << 2);      // 2^(k-1) (1 + m/2), k = mag / 2
    return ((c & 8u) << 4) | code;
}

// One thread per 8 elements: 4 bytes of MXFP4 codes -> 8 bytes of E4M3.
__global__ void convert_mxfp4_mxfp8_kernel(const uint32_t *__restrict__ src, uint2 *__restrict__ dst, int64_t n8)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8; i += (int64_t)gridDim.x * blockDim.x) {
        const uint32_t w = src[i];
        uint32_t lo = 0, hi = 0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            lo |= e2m1_to_e4m3((w >> (4 * j)) & 0xFu) << (8 * j);
            hi |= e2m1_to_e4m3((w >> (16 + 4 * j)) & 0xFu) << (8 * j);
        }
        dst[i] = make_uint2(lo, hi);
    }
}

template <int LAYOUT, bool BF16>
__global__ void dequant_mxfp8_kernel(const uint2 *__restrict__ codes, const uint8_t *__restrict__ scales, int64_t rows,
                                     int64_t k, void *__restrict__ out)
{
    const int64_t kchunks = k >> 3;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < rows * kchunks;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = c / kchunks, cc = c % kchunks;
        const float s = pow2_e(scales[scale_index8<LAYOUT>(m, cc >> 2, k >> 5)]);
        const uint2 w = codes[c];
        float q[8];
        e4m3x2_decode(w.x & 0xFFFFu, q[0], q[1]);
        e4m3x2_decode(w.x >> 16, q[2], q[3]);
        e4m3x2_decode(w.y & 0xFFFFu, q[4], q[5]);
        e4m3x2_decode(w.y >> 16, q[6], q[7]);
        if (BF16) {
            uint32_t p[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                // exact unless below bf16's normal range (round-to-nearest-even there)
                __nv_bfloat162 b = __floats2bfloat162_rn(q[2 * i] * s, q[2 * i + 1] * s);
                p[i] = *reinterpret_cast<uint32_t *>(&b);
            }
            static_cast<uint4 *>(out)[c] = make_uint4(p[0], p[1], p[2], p[3]);
        } else {
            float4 *o = reinterpret_cast<float4 *>(static_cast<float *>(out) + c * 8);
            o[0] = make_float4(q[0] * s, q[1] * s, q[2] * s, q[3] * s);
            o[1] = make_float4(q[4] * s, q[5] * s, q[6] * s, q[7] * s);
        }
    }
}

int grid8(int64_t work, int threads, int max_blocks)
{
    int64_t b = (work + threads - 1) / threads;
    if (b > max_blocks)
        b = max_blocks;
    return (int)(b < 1 ? 1 : b);
}

} // namespace

cudaError_t launch_act_quant_mxfp8(const void *x, int64_t M, int64_t K, void *codes, void *scales, int layout,
                                   cudaStream_t st)
{
    const int64_t pad = layout == RFQ_SCALE_MMA ? ((M + 127) / 128) * 128 - M : 0;
    const int64_t warps = M * ((K + kSeg - 1) / kSeg);
    const int blocks = grid8(warps * 32 > pad * (K / 32) ? warps * 32 : pad * (K / 32), 256, 152 * 24);
    auto *xi = static_cast<const uint4 *>(x);
    auto *c = static_cast<uint8_t *>(codes);
    auto *s = static_cast<uint8_t *>(scales);
    if (layout == RFQ_SCALE_MMA)
        act_quant8_kernel<false, false, RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>(xi, M, K, c, s, nullptr, nullptr,
                                                                             nullptr, 1, 32, pad);
    else
        act_quant8_kernel<false, false, RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>(xi, M, K, c, s, nullptr, nullptr,
                                                                                  nullptr, 1, 32, pad);
    return cudaGetLastError();
}

cudaError_t launch_act_quant_rfq8(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                  void *mcodes, void *mscales, void *rcodes, void *rscales, uint8_t *phi, int layout,
                                  cudaStream_t st, void *m8codes, void *m8scales)
{
    if (mode == RFQ_FALLBACK_AMAX && p_s == 128 && r_s == 256 && K % 256 == 0) {
        // the GEMMs' phi granularity: phi computed in the quantizer's pass
        const unsigned tiles = (unsigned)(((M + 127) / 128) * (K / 256));
        auto *xi = static_cast<const uint4 *>(x);
        auto *mc = static_cast<uint8_t *>(mcodes);
        auto *ms = static_cast<uint8_t *>(mscales);
        auto *rc = static_cast<uint8_t *>(rcodes);
        auto *rs = static_cast<uint8_t *>(rscales);
        auto *oc = static_cast<uint8_t *>(m8codes);
        auto *os = static_cast<uint8_t *>(m8scales);
        constexpr int smem = 128 * 256 * 2;   // the tile, staged in shared memory
        auto k = layout == RFQ_SCALE_MMA ? (oc ? act_quant_rfq8_amax_kernel<RFQ_SCALE_MMA, true>
                                               : act_quant_rfq8_amax_kernel<RFQ_SCALE_MMA, false>)
                                         : (oc ? act_quant_rfq8_amax_kernel<RFQ_SCALE_ROWMAJOR, true>
                                               : act_quant_rfq8_amax_kernel<RFQ_SCALE_ROWMAJOR, false>);
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess)
            return e;
        k<<<tiles, 256, smem, st>>>(xi, M, K, mc, ms, rc, rs, phi, tau, oc, os);
        return cudaGetLastError();
    }
    if (mode == RFQ_FALLBACK_AMAX) {
        cudaError_t e = launch_phi_amax(x, M, K, p_s, r_s, tau, phi, st);
        if (e != cudaSuccess)
            return e;
    } else if (phi) {
        cudaError_t e = launch_phi_fill(phi, (M + p_s - 1) / p_s * ((K + r_s - 1) / r_s), 1, st);
        if (e != cudaSuccess)
            return e;
    }
    const int64_t pad = layout == RFQ_SCALE_MMA ? ((M + 127) / 128) * 128 - M : 0;
    const int64_t warps = M * ((K + kSeg - 1) / kSeg);
    const int blocks = grid8(warps * 32 > pad * (K / 32) ? warps * 32 : pad * (K / 32), 256, 152 * 24);
    auto *xi = static_cast<const uint4 *>(x);
    auto *mc = static_cast<uint8_t *>(mcodes);
    auto *ms = static_cast<uint8_t *>(mscales);
    auto *rc = static_cast<uint8_t *>(rcodes);
    auto *rs = static_cast<uint8_t *>(rscales);
    const bool sel = mode == RFQ_FALLBACK_AMAX;
    auto *oc = static_cast<uint8_t *>(m8codes);
    auto *os = static_cast<uint8_t *>(m8scales);
    // Without the E4M3 X~: one lane per 32-element block, as many 256-thread
    // blocks as are resident at once, each warp looping over (row,
    // 1024-element) items (Wan FFN: 0.100 against 0.115 ms for four lanes per
    // block).  With it the four-lane kernel stays faster (0.146 against 0.164
    // ms: the lane form then holds X~'s values for the second conversion).
    const int64_t lane_work = M * ((K / 32 + 31) / 32) * 32;
    const int64_t work = lane_work > pad * (K / 32) ? lane_work : pad * (K / 32);
    auto grid = [&](auto kern) {
        return grid8(work, 256, num_sms() * resident_blocks_per_sm((const void *)kern, 256, 0));
    };
#define RFQ_AQ8(PHI, LAY)                                                                                         \
    do {                                                                                                          \
        if (oc)                                                                                                   \
            act_quant8_kernel<true, PHI, LAY, true><<<blocks, 256, 0, st>>>(xi, M, K, mc, ms, rc, rs, phi, p_s,    \
                                                                           r_s, pad, oc, os);                     \
        else                                                                                                      \
            act_quant_rfq8_kernel<PHI, LAY><<<grid(act_quant_rfq8_kernel<PHI, LAY>), 256, 0, st>>>(                \
                xi, M, K, mc, ms, rc, rs, phi, p_s, r_s, pad);                                                    \
    } while (0)
    if (layout == RFQ_SCALE_MMA) {
        if (sel) RFQ_AQ8(true, RFQ_SCALE_MMA);
        else RFQ_AQ8(false, RFQ_SCALE_MMA);
    } else {
        if (sel) RFQ_AQ8(true, RFQ_SCALE_ROWMAJOR);
        else RFQ_AQ8(false, RFQ_SCALE_ROWMAJOR);
    }
#undef RFQ_AQ8
    return cudaGetLastError();
}

cudaError_t launch_weight_quant_mxfp8(const void *w, int64_t K, int64_t N, void *codes, void *scales, int layout,
                                      cudaStream_t st)
{
    const int64_t Npad = layout == RFQ_SCALE_MMA ? ((N + 127) / 128) * 128 : N;
    const int64_t work = Npad * (K / 32);
    const int blocks = (int)((work + 255) / 256);
    auto *wi = static_cast<const __nv_bfloat16 *>(w);
    if (layout == RFQ_SCALE_MMA)
        weight_quant_mxfp8_kernel<RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>(wi, K, N, Npad, static_cast<uint8_t *>(codes),
                                                                        static_cast<uint8_t *>(scales));
    else
        weight_quant_mxfp8_kernel<RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>(
            wi, K, N, Npad, static_cast<uint8_t *>(codes), static_cast<uint8_t *>(scales));
    return cudaGetLastError();
}

cudaError_t launch_convert_mxfp4_mxfp8(const void *src_codes, const void *src_scales, int64_t rows, int64_t k,
                                       size_t scale_bytes, void *dst_codes, void *dst_scales, cudaStream_t st)
{
    const int64_t n8 = rows * (k / 8);
    convert_mxfp4_mxfp8_kernel<<<grid8(n8, 256, 152 * 16), 256, 0, st>>>(static_cast<const uint32_t *>(src_codes),
                                                                         static_cast<uint2 *>(dst_codes), n8);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return e;
    return cudaMemcpyAsync(dst_scales, src_scales, scale_bytes, cudaMemcpyDeviceToDevice, st);
}

cudaError_t launch_dequant_mxfp8(const void *codes, const void *scales, int64_t rows, int64_t k, int layout, void *out,
                                 bool bf16, cudaStream_t st)
{
    const int64_t n = rows * (k / 8);
    const int blocks = grid8(n, 256, 152 * 16);
    auto *c = static_cast<const uint2 *>(codes);
    auto *s = static_cast<const uint8_t *>(scales);
    if (layout == RFQ_SCALE_MMA) {
        if (bf16) dequant_mxfp8_kernel<RFQ_SCALE_MMA, true><<<blocks, 256, 0, st>>>(c, s, rows, k, out);
        else dequant_mxfp8_kernel<RFQ_SCALE_MMA, false><<<blocks, 256, 0, st>>>(c, s, rows, k, out);
    } else {
        if (bf16) dequant_mxfp8_kernel<RFQ_SCALE_ROWMAJOR, true><<<blocks, 256, 0, st>>>(c, s, rows, k, out);
        else dequant_mxfp8_kernel<RFQ_SCALE_ROWMAJOR, false><<<blocks, 256, 0, st>>>(c, s, rows, k, out);
    }
    return cudaGetLastError();
}

} // namespace rfq
