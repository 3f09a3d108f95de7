// quant_hif4.cu -- HiF4 quantization kernels for sm_103a (Sec. 3.3).
//
// A HiF4 block is 64 elements along K with one 32-bit metadata word:
//   bits [7:0]   UE6M2 macro scale S = 2^(E-48) (1 + M/4)   (E in [7:2], M in [1:0])
//   bits [15:8]  E1_8:  one exponent bit per group of 8 elements
//   bits [31:16] E1_16: one exponent bit per sub-group of 4 elements
// and 4-bit S1P2 codes (sign, magnitude k/4 with k = 0..7):
//   V_i = S 2^(E1_8[i/8] + E1_16[i/4]) (k_i / 4).
// The encoder is this library's reading of the paper, which gives only the
// decoder: S is the smallest UE6M2 value with 7 S >= amax; a sub-group takes
// the smallest exponent t in {0,1,2} with amax_sub <= 1.75 2^t S; E1_8 is set
// when a sub-group of its group needs t = 2 and E1_16 = max(t - E1_8, 0);
// elements round to the nearest k/4 step, ties to even k, saturating at 7.
// Every comparison is exact in fp32 (all products carry a few significant
// bits), so the kernels reproduce the fp64 definition bit for bit.
//
//   act_quant_hif4     main (+ residual, Sec. 4.3) codes and metadata of X,
//                      optionally with their exact bf16 values
//   weight_quant_hif4  W [K x N] -> K-major HiF4
//   dequant_hif4       -> fp32 or bf16 values
//
// Metadata layouts: row-major [rows][K/64] words, or block-major
// [K/64][rows] words (RFQ_SCALE_MMA: one k-block of every row contiguous, as
// the HiF4 GEMM stages it).
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"

namespace rfq {
namespace {

__device__ __forceinline__ float fmax3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

__device__ __forceinline__ float ue6m2_value(int E, int M) // 2^(E-48) (1 + M/4), E in [0, 63]
{
    return __uint_as_float(((uint32_t)(E - 48 + 127) << 23) | ((uint32_t)M << 21));
}

// Smallest UE6M2 byte with 7 * value >= amax (amax > 0), clamped to [0, 255].
// With amax = sig 2^ea (sig in [1, 2)), the candidates 7 (1 + M/4) 2^(E-48)
// in increasing order are, for E - 48 = ea - 3, sig x {0.875, 1.09375,
// 1.3125, 1.53125} and then, for E - 48 = ea - 2, {1.75, 2.1875, ...}; so
// the answer follows from the significand bits of amax alone (thresholds
// 0.09375, 0.3125, 0.53125 and 0.75 of the fraction: 0x0C0000, 0x280000,
// 0x440000, 0x600000 in the 23-bit field), then the E range [0, 63].
__device__ __forceinline__ int hif4_scale_byte(float amax)
{
    const uint32_t b = __float_as_uint(amax);
    if (b < 0x00800000u)   // a subnormal amax is below every 7 S: byte 0
        return 0;
    const uint32_t f = b & 0x7FFFFFu;
    const int e0 = (int)(b >> 23) - 127 - 3 + 48;   // E of the first candidate row
    int E, M;
    if (f <= 0x600000u && e0 >= 0) {
        // first row, M = 1..3, or (E0 + 1, 0)
        M = 1 + (f > 0x0C0000u) + (f > 0x280000u) + (f > 0x440000u);
        E = e0;
        if (M == 4) {
            M = 0;
            E = e0 + 1;
        }
    } else if (e0 >= -1) {
        // second row: (E0 + 1, 0) if sig <= 1.75, else (E0 + 1, 1); with
        // E0 = -1 the first row is out of range and this is the smallest
        E = e0 + 1;
        M = f > 0x600000u ? 1 : 0;
    } else {
        return 0;          // below the smallest macro scale: 2^-48 covers it
    }
    if (E > 63)
        return 255;        // above the largest macro scale: saturate
    return (E << 2) | M;
}

// Quantizes the eight elements x[0..7] of group g (sub-groups 2g, 2g+1) of a
// 64-element block whose macro scale byte sb = (E << 2) | M is given.
// Returns the codes (element i in nibble i) and this group's E1_8 / E1_16
// bits (placed at their final metadata positions); `deq` receives the
// dequantized values.
//
// A sub-group with exponent ex has the step 0.25 S 2^ex = 2^(E - 50 + ex)
// (1 + M/4), formed from its bits, and its reciprocal is 2^(50 - E - ex)
// 4 / (4 + M): rounded to fp32 that is the power of two times RN(4 / (4 + M))
// (scaling by a power of two commutes with rounding in the normal range,
// which every E in [0, 63] and ex in [0, 2] stays in), i.e. exactly the
// correctly rounded reciprocal of the step, from one of four constants.
__device__ __forceinline__ uint32_t hif4_group(const float (&x)[8], int sb, int g, uint32_t &meta_bits,
                                               float (&deq)[8])
{
    const int E = sb >> 2, M = sb & 3;
    const float S = ue6m2_value(E, M);
    const float recip_m = M == 0 ? 1.0f : M == 1 ? 0.8f : M == 2 ? 0.6666666865348816f : 0.5714285969734192f;
    int t[2];
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const float a = fmax3(fmaxf(fabsf(x[4 * h]), fabsf(x[4 * h + 1])), fabsf(x[4 * h + 2]), fabsf(x[4 * h + 3]));
        t[h] = a <= 1.75f * S ? 0 : (a <= 3.5f * S ? 1 : 2);
    }
    const int e18 = (t[0] == 2 || t[1] == 2) ? 1 : 0;
    const int e116_0 = max(t[0] - e18, 0), e116_1 = max(t[1] - e18, 0);
    meta_bits = ((uint32_t)e18 << (8 + g)) | ((uint32_t)e116_0 << (16 + 2 * g)) | ((uint32_t)e116_1 << (17 + 2 * g));
    float kf[8];   // the magnitudes k as floats (exact small integers)
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int ex = e18 + (h ? e116_1 : e116_0);
        const float step = __uint_as_float(((uint32_t)(E + ex + 77) << 23) | ((uint32_t)M << 21));
        const float inv = __uint_as_float((uint32_t)(177 - E - ex) << 23) * recip_m;   // RN(1 / step)
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float v = x[4 * h + i];
            const float a = fabsf(v);
            // nearest k, ties to even, from the correctly rounded quotient
            // a / step: a * inv is within one ulp of it (inv is the correctly
            // rounded reciprocal), the remainder a - q step is exact (fma),
            // and one correction q + r inv rounds to the correctly rounded
            // quotient (Markstein's division refinement, P. Markstein, IA-64
            // and Elementary Functions, 2000).  A true tie (a half-integer
            // quotient) is then exact, and adding 2^23 rounds it to the even
            // integer; any other quotient lies at least 2^-9 / 7 from every
            // half-integer (a has 8 significant bits, step = D 2^s with D in
            // {4,5,6,7}/4), far beyond the rounding error.  fminf saturates
            // (NaN -> 7) before the rounding.
            float q = a * inv;
            q = fmaf(fmaf(-q, step, a), inv, q);
            const float k = (fminf(q, 7.0f) + 8388608.0f) - 8388608.0f;
            kf[4 * h + i] = k;
            deq[4 * h + i] = copysignf(k * step, v);
        }
    }
    // the eight 3-bit magnitudes into nibbles: two sums of k 16^i (exact
    // below 2^16), their integer bits by adding 2^23, the low halves joined;
    // then the sign bits (bit 3 of each nibble) from the inputs' sign bits
    const float lo = fmaf(kf[3], 4096.0f, fmaf(kf[2], 256.0f, fmaf(kf[1], 16.0f, kf[0])));
    const float hi = fmaf(kf[7], 4096.0f, fmaf(kf[6], 256.0f, fmaf(kf[5], 16.0f, kf[4])));
    uint32_t codes = __byte_perm(__float_as_uint(lo + 8388608.0f), __float_as_uint(hi + 8388608.0f), 0x5410);
#pragma unroll
    for (int i = 0; i < 8; ++i)
        codes |= (__float_as_uint(x[i]) >> (28 - 4 * i)) & (8u << (4 * i));
    return codes;
}

// rows: the matrix's row count; the block-major layout pads it to 128.
template <int LAYOUT>
__device__ __forceinline__ int64_t meta_index(int64_t m, int64_t blk, int64_t rows, int64_t kblocks)
{
    return LAYOUT == RFQ_SCALE_MMA ? blk * (((rows + 127) >> 7) << 7) + m : m * kblocks + blk;
}

// act_quant_hif4_kernel: 8 / kHNG consecutive lanes hold one 64-element
// block (lane l: kHNG consecutive groups, hif4_chunk_n); the fused
// AMAX kernel below keeps eight lanes per block (lane l: group l % 8,
// hif4_chunk).  Quantizes x (main), and with RES its residual x - x~
// (Sec. 4.3).  Items are (row, 1024-element segment): a warp loads its four
// 16-byte chunks per lane up front, and the row and block indices come from
// the item without a 64-bit division per chunk.  With EXP the kernel also writes the exact bf16
// values of X~ (and X^; zeros where phi = 0) as [M][K] row-major, the
// operands of the bf16 tensor-core GEMM: every HiF4 value has at most six
// significant bits and an exponent inside bf16's range.
constexpr int kHSeg = 1024;
constexpr int kHU = kHSeg / 256;

__device__ __forceinline__ uint4 bf16x8_pack(const float (&v)[8]) // exact for the values above
{
    uint32_t p[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        __nv_bfloat162 b = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
        p[i] = *reinterpret_cast<uint32_t *>(&b);
    }
    return make_uint4(p[0], p[1], p[2], p[3]);
}

// One lane's eight elements xf (group g of its 64-element block; the block's
// eight lanes take part together) at chunk c of the [M][K / 8] chunk grid:
// the main codes and metadata, with RES the residual's (zeros when !on),
// with EXP the exact bf16 values of both.  ok: the chunk is inside the row
// (uniform over the block's lanes); stores happen only then.
template <bool RES, bool EXP, int LAYOUT>
__device__ __forceinline__ void hif4_chunk(const float (&xf)[8], int g, bool ok, bool on, int64_t c, int64_t moff,
                                           uint32_t *__restrict__ mcodes, uint32_t *__restrict__ mmeta,
                                           uint32_t *__restrict__ rcodes, uint32_t *__restrict__ rmeta,
                                           uint4 *__restrict__ m16, uint4 *__restrict__ r16)
{
    float am = fmax3(fmax3(fabsf(xf[0]), fabsf(xf[1]), fabsf(xf[2])),
                     fmax3(fabsf(xf[3]), fabsf(xf[4]), fabsf(xf[5])), fmaxf(fabsf(xf[6]), fabsf(xf[7])));
#pragma unroll
    for (int o = 1; o < 8; o <<= 1)
        am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, o));
    const int sb = am > 0.f ? hif4_scale_byte(am) : 0;
    uint32_t bits;
    float deq[8];
    uint32_t code = hif4_group(xf, sb, g, bits, deq);
    if (am == 0.f) {
        bits = 0;   // all-zero block: metadata 0, codes keep the sign of zero
    }
#pragma unroll
    for (int o = 1; o < 8; o <<= 1)
        bits |= __shfl_xor_sync(0xFFFFFFFFu, bits, o);
    if (ok) {
        mcodes[c] = code;
        if (g == 0)
            mmeta[moff] = am == 0.f ? 0u : (bits | (uint32_t)sb);
        if (EXP)
            m16[c] = bf16x8_pack(deq);
    }
    if (RES) {
        float r[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            r[i] = xf[i] - deq[i]; // exact
        float ra = fmax3(fmax3(fabsf(r[0]), fabsf(r[1]), fabsf(r[2])),
                         fmax3(fabsf(r[3]), fabsf(r[4]), fabsf(r[5])), fmaxf(fabsf(r[6]), fabsf(r[7])));
#pragma unroll
        for (int o = 1; o < 8; o <<= 1)
            ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, o));
        const int rsb = ra > 0.f ? hif4_scale_byte(ra) : 0;
        uint32_t rbits;
        float rdeq[8];
        const uint32_t rcode = hif4_group(r, rsb, g, rbits, rdeq);
#pragma unroll
        for (int o = 1; o < 8; o <<= 1)
            rbits |= __shfl_xor_sync(0xFFFFFFFFu, rbits, o);
        if (ok) {
            rcodes[c] = on ? rcode : 0u;
            if (g == 0)
                rmeta[moff] = (on && ra > 0.f) ? (rbits | (uint32_t)rsb) : 0u;
            if (EXP)
                r16[c] = on ? bf16x8_pack(rdeq) : make_uint4(0, 0, 0, 0);
        }
    }
}

// The same for one lane's 8 NG elements xf (groups NG gq .. NG gq + NG - 1
// of its 64-element block, 8 / NG lanes per block) at chunks c .. c + NG - 1:
// the block's amax, macro scale and metadata reduce over 8 / NG lanes, so
// each lane does that per-block work for NG times the elements of
// hif4_chunk.
template <int NG>
struct CodeVec;
template <>
struct CodeVec<2> {
    using T = uint2;
    static __device__ __forceinline__ T make(const uint32_t (&c)[2]) { return make_uint2(c[0], c[1]); }
};
template <>
struct CodeVec<4> {
    using T = uint4;
    static __device__ __forceinline__ T make(const uint32_t (&c)[4]) { return make_uint4(c[0], c[1], c[2], c[3]); }
};

template <bool RES, bool EXP, int NG>
__device__ __forceinline__ void hif4_chunk_n(const float (&xf)[8 * NG], int gq, bool ok, bool on, int64_t c,
                                             int64_t moff, uint32_t *__restrict__ mcodes,
                                             uint32_t *__restrict__ mmeta, uint32_t *__restrict__ rcodes,
                                             uint32_t *__restrict__ rmeta, uint4 *__restrict__ m16,
                                             uint4 *__restrict__ r16)
{
    using CV = CodeVec<NG>;
    float am = 0.f;
#pragma unroll
    for (int i = 0; i < 8 * NG; i += 4)
        am = fmax3(am, fmaxf(fabsf(xf[i]), fabsf(xf[i + 1])), fmaxf(fabsf(xf[i + 2]), fabsf(xf[i + 3])));
#pragma unroll
    for (int o = 1; o < 8 / NG; o <<= 1)
        am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, o));
    const int sb = am > 0.f ? hif4_scale_byte(am) : 0;
    float xg[NG][8], d[NG][8];
    uint32_t code[NG], bits = 0;
#pragma unroll
    for (int j = 0; j < NG; ++j) {
#pragma unroll
        for (int i = 0; i < 8; ++i)
            xg[j][i] = xf[8 * j + i];
        uint32_t b;
        code[j] = hif4_group(xg[j], sb, NG * gq + j, b, d[j]);
        bits |= b;
    }
    if (am == 0.f)
        bits = 0;   // all-zero block: metadata 0, codes keep the sign of zero
#pragma unroll
    for (int o = 1; o < 8 / NG; o <<= 1)
        bits |= __shfl_xor_sync(0xFFFFFFFFu, bits, o);
    if (ok) {
        *reinterpret_cast<typename CV::T *>(mcodes + c) = CV::make(code);
        if (gq == 0)
            mmeta[moff] = am == 0.f ? 0u : (bits | (uint32_t)sb);
        if (EXP) {
#pragma unroll
            for (int j = 0; j < NG; ++j)
                m16[c + j] = bf16x8_pack(d[j]);
        }
    }
    if (RES) {
        float r[NG][8];
        float ra = 0.f;
#pragma unroll
        for (int j = 0; j < NG; ++j) {
#pragma unroll
            for (int i = 0; i < 8; ++i)
                r[j][i] = xg[j][i] - d[j][i]; // exact
#pragma unroll
            for (int i = 0; i < 8; i += 4)
                ra = fmax3(ra, fmaxf(fabsf(r[j][i]), fabsf(r[j][i + 1])), fmaxf(fabsf(r[j][i + 2]), fabsf(r[j][i + 3])));
        }
#pragma unroll
        for (int o = 1; o < 8 / NG; o <<= 1)
            ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, o));
        const int rsb = ra > 0.f ? hif4_scale_byte(ra) : 0;
        uint32_t rcode[NG], rbits = 0;
        float e[NG][8];
#pragma unroll
        for (int j = 0; j < NG; ++j) {
            uint32_t b;
            rcode[j] = hif4_group(r[j], rsb, NG * gq + j, b, e[j]);
            rbits |= b;
        }
#pragma unroll
        for (int o = 1; o < 8 / NG; o <<= 1)
            rbits |= __shfl_xor_sync(0xFFFFFFFFu, rbits, o);
        if (ok) {
            if (!on) {
#pragma unroll
                for (int j = 0; j < NG; ++j)
                    rcode[j] = 0u;
            }
            *reinterpret_cast<typename CV::T *>(rcodes + c) = CV::make(rcode);
            if (gq == 0)
                rmeta[moff] = (on && ra > 0.f) ? (rbits | (uint32_t)rsb) : 0u;
            if (EXP) {
#pragma unroll
                for (int j = 0; j < NG; ++j)
                    r16[c + j] = on ? bf16x8_pack(e[j]) : make_uint4(0, 0, 0, 0);
            }
        }
    }
}

// Groups per lane in act_quant_hif4_kernel: 2 (0.092 ms on the Qwen3-VL
// down projection) against 1 (0.100 ms, eight lanes per block) and 4
// (0.102 ms: 115 registers, two blocks per SM).
constexpr int kHNG = 2;

template <bool RES, bool PHI, int LAYOUT, bool EXP>
__global__ void __launch_bounds__(256) act_quant_hif4_kernel(const uint4 *__restrict__ x, int64_t M, int64_t K,
                                                            uint32_t *__restrict__ mcodes,
                                                            uint32_t *__restrict__ mmeta,
                                                            uint32_t *__restrict__ rcodes,
                                                            uint32_t *__restrict__ rmeta,
                                                            const uint8_t *__restrict__ phi, int p_s, int r_s,
                                                            uint4 *__restrict__ m16, uint4 *__restrict__ r16)
{
    const int lane = threadIdx.x & 31;
    constexpr int NG = kHNG, LPB = 8 / NG;         // groups per lane, lanes per block
    const int gq = lane & (LPB - 1);               // the lane's place in its block
    const int kchunks = (int)(K >> 3);
    const int64_t kblocks = K >> 6;
    const int segs = (kchunks + kHSeg / 8 - 1) / (kHSeg / 8);
    const int64_t items = M * segs;
    const int phi_cols = PHI ? (int)((K + r_s - 1) / r_s) : 0;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    for (int64_t item = gwarp; item < items; item += nwarps) {
        const int64_t m = item / segs;
        const int c0 = (int)(item - m * segs) * (kHSeg / 8);
        const uint4 *xr = x + m * kchunks;
        // steps of 256 NG elements; lane l takes chunks NG l .. NG l + NG - 1
        // of each (K is a multiple of 64, so a block is wholly inside the row
        // or past it)
        uint4 vv[kHU];
#pragma unroll
        for (int j = 0; j < kHU; ++j) {
            const int c = c0 + (j / NG) * 32 * NG + NG * lane + (j % NG);
            vv[j] = c < kchunks ? __ldcs(xr + c) : make_uint4(0, 0, 0, 0);
        }
        const uint8_t *prow = PHI ? phi + (m / p_s) * phi_cols : nullptr;
#pragma unroll
        for (int s = 0; s < kHU / NG; ++s) {
            const int cr = c0 + s * 32 * NG + NG * lane;   // first of the lane's NG chunks
            const bool ok = cr < kchunks;                  // uniform over each block's lanes
            float xf[8 * NG];
#pragma unroll
            for (int u = 0; u < NG; ++u) {
                const uint32_t w[4] = {vv[NG * s + u].x, vv[NG * s + u].y, vv[NG * s + u].z, vv[NG * s + u].w};
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    xf[8 * u + 2 * i] = __uint_as_float(w[i] << 16);
                    xf[8 * u + 2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
                }
            }
            // r_s is a multiple of 64: the block lies in one phi column
            const bool on = !PHI || (ok && prow[(cr * 8) / r_s] != 0);
            hif4_chunk_n<RES, EXP, NG>(xf, gq, ok, on, m * kchunks + cr,
                                       meta_index<LAYOUT>(m, cr >> 3, M, kblocks), mcodes, mmeta, rcodes, rmeta,
                                       m16, r16);
        }
    }
}

// AMAX fallback (Sec. 4.3) for phi tiles of 128 rows x 256 columns, fused
// into the quantizer (as act_quant_mxfp4_amax_kernel): one 512-thread block
// per tile keeps its 64 KB in registers (warp w rows 8w .. 8w + 7, lane l
// the l-th 16-byte chunk of each; lanes 8b .. 8b + 7 hold 64-element block
// b), reduces max |x| (packed bf16x2 max, NaN dropped, as phi_amax_kernel),
// writes phi, then quantizes; the residual of a phi = 0 tile is written as
// zeros without being computed.  X is read once.
constexpr int kHAmaxRows = 8;

template <int LAYOUT, bool EXP>
__global__ void __launch_bounds__(512, 1) act_quant_hif4_amax_kernel(const uint4 *__restrict__ x, int64_t M,
                                                                    int64_t K, uint32_t *__restrict__ mcodes,
                                                                    uint32_t *__restrict__ mmeta,
                                                                    uint32_t *__restrict__ rcodes,
                                                                    uint32_t *__restrict__ rmeta,
                                                                    uint8_t *__restrict__ phi, float tau,
                                                                    uint4 *__restrict__ m16, uint4 *__restrict__ r16)
{
    constexpr int R = kHAmaxRows, NW = 16;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t kchunks = K >> 3;
    const int64_t kblocks = K >> 6;
    const int nr = (int)(K >> 8);
    const int64_t tile = blockIdx.x;
    const int64_t p = tile / nr;
    const int r = (int)(tile - p * nr);
    const int64_t m0 = p * 128 + warp * R;
    const int cr = r * 32 + lane;
    uint4 v[R];
#pragma unroll
    for (int i = 0; i < R; ++i)
        v[i] = m0 + i < M ? __ldcs(x + (m0 + i) * kchunks + cr) : make_uint4(0, 0, 0, 0);
    uint32_t acc = 0;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const uint32_t q[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
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
    const int g = lane & 7;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const int64_t m = m0 + i; // uniform over the warp
        if (m >= M)
            break;
        float xf[8];
        const uint32_t w[4] = {v[i].x, v[i].y, v[i].z, v[i].w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            xf[2 * k] = __uint_as_float(w[k] << 16);
            xf[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        }
        const int64_t c = m * kchunks + cr;
        const int64_t moff = meta_index<LAYOUT>(m, cr >> 3, M, kblocks);
        if (on) {
            hif4_chunk<true, EXP, LAYOUT>(xf, g, true, true, c, moff, mcodes, mmeta, rcodes, rmeta, m16, r16);
        } else {
            hif4_chunk<false, EXP, LAYOUT>(xf, g, true, true, c, moff, mcodes, mmeta, rcodes, rmeta, m16, r16);
            rcodes[c] = 0u;
            if (g == 0)
                rmeta[moff] = 0u;
            if (EXP)
                r16[c] = make_uint4(0, 0, 0, 0);
        }
    }
}

// One thread per (column n, 64-block) of W [K x N]: a warp reads 32
// consecutive columns of one K row at a time.
template <int LAYOUT>
__global__ void __launch_bounds__(256) weight_quant_hif4_kernel(const __nv_bfloat16 *__restrict__ w, int64_t K,
                                                               int64_t N, uint8_t *__restrict__ codes,
                                                               uint32_t *__restrict__ meta)
{
    const int64_t kblocks = K >> 6;
    const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    const int64_t n = t % N, blk = t / N;
    if (blk >= kblocks)
        return;
    float am = 0.f;
    for (int i = 0; i < 64; ++i)
        am = fmaxf(am, fabsf(__bfloat162float(w[(blk * 64 + i) * N + n])));
    const int sb = am > 0.f ? hif4_scale_byte(am) : 0;
    uint32_t bits = 0, out[8];
    for (int g = 0; g < 8; ++g) {
        float xf[8], deq[8];
        for (int i = 0; i < 8; ++i)
            xf[i] = __bfloat162float(w[(blk * 64 + 8 * g + i) * N + n]);
        uint32_t gb;
        out[g] = hif4_group(xf, sb, g, gb, deq);
        bits |= gb;
    }
    uint4 *dst = reinterpret_cast<uint4 *>(codes + n * (K >> 1) + blk * 32);
    dst[0] = make_uint4(out[0], out[1], out[2], out[3]);
    dst[1] = make_uint4(out[4], out[5], out[6], out[7]);
    meta[meta_index<LAYOUT>(n, blk, N, kblocks)] = am == 0.f ? 0u : (bits | (uint32_t)sb);
}

// x = S 2^(E1_8 + E1_16) k / 4 with the code's sign; 8 elements per thread.
template <int LAYOUT, bool BF16>
__global__ void dequant_hif4_kernel(const uint32_t *__restrict__ codes, const uint32_t *__restrict__ meta,
                                    int64_t rows, int64_t k, void *__restrict__ out)
{
    const int64_t kchunks = k >> 3;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < rows * kchunks;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = c / kchunks, cc = c % kchunks;
        const int64_t blk = cc >> 3;
        const int g = (int)(cc & 7);
        const uint32_t md = meta[meta_index<LAYOUT>(m, blk, rows, k >> 6)];
        const float S = ue6m2_value((int)((md >> 2) & 63), (int)(md & 3));
        const uint32_t cw = codes[c];
        float v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            const int j = 2 * g + (i >> 2); // sub-group
            const int ex = (int)((md >> (8 + g)) & 1) + (int)((md >> (16 + j)) & 1);
            const uint32_t code = (cw >> (4 * i)) & 0xF;
            const float q = (float)(code & 7) * 0.25f * S * (float)(1 << ex);
            v[i] = (code & 8) ? -q : q;
        }
        if (BF16) {
            uint32_t p[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                __nv_bfloat162 b = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]); // exact
                p[i] = *reinterpret_cast<uint32_t *>(&b);
            }
            reinterpret_cast<uint4 *>(out)[c] = make_uint4(p[0], p[1], p[2], p[3]);
        } else {
            float4 *o = reinterpret_cast<float4 *>(static_cast<float *>(out) + c * 8);
            o[0] = make_float4(v[0], v[1], v[2], v[3]);
            o[1] = make_float4(v[4], v[5], v[6], v[7]);
        }
    }
}

int grid_for(int64_t work, int threads, int max_blocks)
{
    int64_t b = (work + threads - 1) / threads;
    if (b > max_blocks)
        b = max_blocks;
    return (int)(b < 1 ? 1 : b);
}

} // namespace

cudaError_t launch_act_quant_hif4(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                  void *mcodes, void *mmeta, void *rcodes, void *rmeta, uint8_t *phi, int layout,
                                  cudaStream_t st, void *m16, void *r16)
{
    const int64_t np = (M + p_s - 1) / p_s, nr = (K + r_s - 1) / r_s;
    if (mode == RFQ_FALLBACK_AMAX && p_s == 128 && r_s == 256 && K % 256 == 0) {
        // the GEMMs' phi granularity: phi computed in the quantizer's pass
        auto *xi = static_cast<const uint4 *>(x);
        auto *mc = static_cast<uint32_t *>(mcodes);
        auto *mm = static_cast<uint32_t *>(mmeta);
        auto *rc = static_cast<uint32_t *>(rcodes);
        auto *rm = static_cast<uint32_t *>(rmeta);
        auto *e0 = static_cast<uint4 *>(m16);
        auto *e1 = static_cast<uint4 *>(r16);
        const unsigned tiles = (unsigned)(np * nr);
#define RFQ_HA(LAY, EXP) \
    act_quant_hif4_amax_kernel<LAY, EXP><<<tiles, 512, 0, st>>>(xi, M, K, mc, mm, rc, rm, phi, tau, e0, e1)
        if (layout == RFQ_SCALE_MMA) {
            if (e0) RFQ_HA(RFQ_SCALE_MMA, true);
            else RFQ_HA(RFQ_SCALE_MMA, false);
        } else {
            if (e0) RFQ_HA(RFQ_SCALE_ROWMAJOR, true);
            else RFQ_HA(RFQ_SCALE_ROWMAJOR, false);
        }
#undef RFQ_HA
        return cudaGetLastError();
    }
    if (mode == RFQ_FALLBACK_AMAX) {
        cudaError_t e = launch_phi_amax(x, M, K, p_s, r_s, tau, phi, st);
        if (e != cudaSuccess)
            return e;
    } else if (phi) {
        cudaError_t e = launch_phi_fill(phi, np * nr, mode == RFQ_FALLBACK_ALL ? 1 : 0, st);
        if (e != cudaSuccess)
            return e;
    }
    const int64_t items = M * ((K / 8 + kHSeg / 8 - 1) / (kHSeg / 8));
    const int blocks = grid_for(items * 32, 256, 152 * 24);
    auto *xi = static_cast<const uint4 *>(x);
    auto *mc = static_cast<uint32_t *>(mcodes);
    auto *mm = static_cast<uint32_t *>(mmeta);
    auto *rc = static_cast<uint32_t *>(rcodes);
    auto *rm = static_cast<uint32_t *>(rmeta);
    auto *e0 = static_cast<uint4 *>(m16);
    auto *e1 = static_cast<uint4 *>(r16);
#define RFQ_HQ(RES, PHI, LAY, EXP)                                                                                \
    act_quant_hif4_kernel<RES, PHI, LAY, EXP><<<blocks, 256, 0, st>>>(xi, M, K, mc, mm, rc, rm, phi, p_s, r_s, e0, e1)
#define RFQ_HQ_E(RES, PHI, LAY)                                                                                   \
    do {                                                                                                          \
        if (e0) RFQ_HQ(RES, PHI, LAY, true);                                                                      \
        else RFQ_HQ(RES, PHI, LAY, false);                                                                        \
    } while (0)
    if (mode == RFQ_FALLBACK_NONE) {
        if (layout == RFQ_SCALE_MMA) RFQ_HQ_E(false, false, RFQ_SCALE_MMA);
        else RFQ_HQ_E(false, false, RFQ_SCALE_ROWMAJOR);
    } else if (mode == RFQ_FALLBACK_ALL) {
        if (layout == RFQ_SCALE_MMA) RFQ_HQ_E(true, false, RFQ_SCALE_MMA);
        else RFQ_HQ_E(true, false, RFQ_SCALE_ROWMAJOR);
    } else {
        if (layout == RFQ_SCALE_MMA) RFQ_HQ_E(true, true, RFQ_SCALE_MMA);
        else RFQ_HQ_E(true, true, RFQ_SCALE_ROWMAJOR);
    }
#undef RFQ_HQ_E
#undef RFQ_HQ
    return cudaGetLastError();
}

cudaError_t launch_weight_quant_hif4(const void *w, int64_t K, int64_t N, void *codes, void *meta, int layout,
                                     cudaStream_t st)
{
    const int64_t work = N * (K / 64);
    const unsigned blocks = (unsigned)((work + 255) / 256);
    if (layout == RFQ_SCALE_MMA)
        weight_quant_hif4_kernel<RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>((const __nv_bfloat16 *)w, K, N,
                                                                         (uint8_t *)codes, (uint32_t *)meta);
    else
        weight_quant_hif4_kernel<RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>((const __nv_bfloat16 *)w, K, N,
                                                                              (uint8_t *)codes, (uint32_t *)meta);
    return cudaGetLastError();
}

cudaError_t launch_dequant_hif4(const void *codes, const void *meta, int64_t rows, int64_t k, int layout,
                                void *out, bool bf16, cudaStream_t st)
{
    const int blocks = grid_for(rows * (k / 8), 256, 152 * 32);
    auto *c = static_cast<const uint32_t *>(codes);
    auto *m = static_cast<const uint32_t *>(meta);
    if (layout == RFQ_SCALE_MMA) {
        if (bf16) dequant_hif4_kernel<RFQ_SCALE_MMA, true><<<blocks, 256, 0, st>>>(c, m, rows, k, out);
        else dequant_hif4_kernel<RFQ_SCALE_MMA, false><<<blocks, 256, 0, st>>>(c, m, rows, k, out);
    } else {
        if (bf16) dequant_hif4_kernel<RFQ_SCALE_ROWMAJOR, true><<<blocks, 256, 0, st>>>(c, m, rows, k, out);
        else dequant_hif4_kernel<RFQ_SCALE_ROWMAJOR, false><<<blocks, 256, 0, st>>>(c, m, rows, k, out);
    }
    return cudaGetLastError();
}

} // namespace rfq
