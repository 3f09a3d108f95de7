// mxfp4_math.cuh -- per-lane MXFP4 quantization arithmetic (Sec. 3.2 Eq. 3-4,
// Sec. 4.3), shared by the activation quantizers and the GEMMs that quantize
// X themselves.
//
// Two arrangements: four consecutive lanes hold one 32-element block, eight
// elements each (mxfp4_quant8), or one lane holds a whole block
// (mxfp4_quant32: no shuffles, the block's scale computed once).
// The E8M0 byte is the fp32 exponent field of the block's amax minus 2 (OCP
// rule floor(log2 amax) - 2, clamped at 0), every scaling is by a power of
// two, the E2M1 conversion rounds to nearest even and saturates, and the
// residual x - q 2^e is exact in fp32 (at most 11 significant bits), so the
// result is the fp64 definition bit for bit.
#pragma once

#include <cuda_fp16.h>
#include <cstdint>

namespace rfq {

// Four E2M1 conversions (round-to-nearest-even, saturating): eight fp32
// values -> eight codes, element 2i in the low nibble of byte i.
__device__ __forceinline__ uint32_t e2m1x8(const float (&y)[8])
{
    uint32_t out;
    asm("{\n\t.reg .b8 b0, b1, b2, b3;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b0, %2, %1;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b1, %4, %3;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b2, %6, %5;\n\t"
        "cvt.rn.satfinite.e2m1x2.f32 b3, %8, %7;\n\t"
        "mov.b32 %0, {b0, b1, b2, b3};\n\t}"
        : "=r"(out)
        : "f"(y[0]), "f"(y[1]), "f"(y[2]), "f"(y[3]), "f"(y[4]), "f"(y[5]), "f"(y[6]), "f"(y[7]));
    return out;
}

// Eight E2M1 codes -> their values (exact), via the e2m1x2 -> f16x2 decode.
__device__ __forceinline__ void e2m1x8_decode(uint32_t codes, float (&q)[8])
{
    uint32_t h[4];
    asm("{\n\t.reg .b8 b0, b1, b2, b3;\n\t"
        "mov.b32 {b0, b1, b2, b3}, %4;\n\t"
        "cvt.rn.f16x2.e2m1x2 %0, b0;\n\t"
        "cvt.rn.f16x2.e2m1x2 %1, b1;\n\t"
        "cvt.rn.f16x2.e2m1x2 %2, b2;\n\t"
        "cvt.rn.f16x2.e2m1x2 %3, b3;\n\t}"
        : "=r"(h[0]), "=r"(h[1]), "=r"(h[2]), "=r"(h[3])
        : "r"(codes));
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        __half2 v = *reinterpret_cast<__half2 *>(&h[i]);
        q[2 * i] = __low2float(v);
        q[2 * i + 1] = __high2float(v);
    }
}

// E8M0 byte of a block from the fp32 exponent field of its amax:
// floor(log2 amax) - 2 + 127 = field - 2, clamped at 0 (2^-127; also amax = 0).
__device__ __forceinline__ int scale_byte_from_f32_bits(uint32_t amax_bits)
{
    return max((int)((amax_bits >> 23) & 0xFF) - 2, 0);
}

__device__ __forceinline__ float pow2_neg_e(int byte) // 2^-(byte-127), normal for byte <= 252
{
    return __uint_as_float((uint32_t)(254 - byte) << 23);
}

__device__ __forceinline__ float pow2_e(int byte) // 2^(byte-127); byte 0 -> subnormal 2^-127
{
    return byte ? __uint_as_float((uint32_t)byte << 23) : __uint_as_float(0x00400000u);
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4 &v, float (&x)[8])
{
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

// Packed fp32 pairs (Blackwell f32x2 arithmetic): one instruction for two
// multiplies or fused multiply-adds, both rounded to nearest even.
__device__ __forceinline__ uint64_t f2pack(float a, float b)
{
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}

__device__ __forceinline__ void f2unpack(uint64_t v, float &a, float &b)
{
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}

__device__ __forceinline__ uint64_t fmul2(uint64_t a, uint64_t b)
{
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

__device__ __forceinline__ uint64_t ffma2(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}

__device__ __forceinline__ float fmax3(float a, float b, float c)
{
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// max |v_i| over eight values
__device__ __forceinline__ float absmax8(const float (&v)[8])
{
    const float m0 = fmax3(fabsf(v[0]), fabsf(v[1]), fabsf(v[2]));
    const float m1 = fmax3(fabsf(v[3]), fabsf(v[4]), fabsf(v[5]));
    return fmax3(m0, m1, fmaxf(fabsf(v[6]), fabsf(v[7])));
}

// The residual X - X~ of this lane's eight elements (its 32-element block
// spread over four consecutive lanes, all 32 lanes take part), given their
// E2M1 codes and E8M0 byte: the residual's E2M1 codes and E8M0 byte.
__device__ __forceinline__ void mxfp4_resid8(const float (&xf)[8], uint32_t code, int sb, uint32_t &rcode, int &rb)
{
    float q[8], r[8];
    e2m1x8_decode(code, q);
    const float nsc = -pow2_e(sb);
    const uint64_t nsc2 = f2pack(nsc, nsc);
#pragma unroll
    for (int i = 0; i < 4; ++i) // x - x~ (exact)
        f2unpack(ffma2(f2pack(q[2 * i], q[2 * i + 1]), nsc2, f2pack(xf[2 * i], xf[2 * i + 1])), r[2 * i],
                 r[2 * i + 1]);
    float ra = absmax8(r);
    ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, 1));
    ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, 2));
    rb = scale_byte_from_f32_bits(__float_as_uint(ra));
    const float rinv = pow2_neg_e(rb);
    const uint64_t rinv2 = f2pack(rinv, rinv);
#pragma unroll
    for (int i = 0; i < 4; ++i)
        f2unpack(fmul2(f2pack(r[2 * i], r[2 * i + 1]), rinv2), r[2 * i], r[2 * i + 1]);
    rcode = e2m1x8(r);
}

// Quantizes this lane's eight elements (its 32-element block is spread over
// four consecutive lanes, all 32 lanes take part): the E2M1 codes (element
// 2i in the low nibble of byte i) and E8M0 byte of X~, the block's max |x|
// (NaN elements dropped), and with RES the codes and byte of the residual
// X - X~.
struct Mx8 {
    uint32_t code, rcode;
    int sb, rb;
    float am;
};

template <bool RES>
__device__ __forceinline__ Mx8 mxfp4_quant8(const float (&xf)[8])
{
    Mx8 o;
    float am = absmax8(xf);
    am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 1));
    am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 2));
    o.am = am;
    o.sb = scale_byte_from_f32_bits(__float_as_uint(am));
    const float inv = pow2_neg_e(o.sb);
    const uint64_t inv2 = f2pack(inv, inv);
    float y[8];
#pragma unroll
    for (int i = 0; i < 4; ++i)
        f2unpack(fmul2(f2pack(xf[2 * i], xf[2 * i + 1]), inv2), y[2 * i], y[2 * i + 1]);
    o.code = e2m1x8(y);
    o.rcode = 0;
    o.rb = 0;
    if (RES)
        mxfp4_resid8(xf, o.code, o.sb, o.rcode, o.rb);
    return o;
}

// ---- one lane per 32-element block

// 256-bit load of global memory that is read once (not kept in L1).
__device__ __forceinline__ void ldg256_stream(const void *p, uint32_t (&r)[8])
{
    asm volatile("ld.global.nc.L1::no_allocate.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "l"(p));
}

// max |v_i| over 32 values (NaN elements dropped)
__device__ __forceinline__ float absmax32(const float (&v)[32])
{
    float m[11];
#pragma unroll
    for (int i = 0; i < 10; ++i)
        m[i] = fmax3(fabsf(v[3 * i]), fabsf(v[3 * i + 1]), fabsf(v[3 * i + 2]));
    m[10] = fmaxf(fabsf(v[30]), fabsf(v[31]));
    const float a = fmax3(m[0], m[1], m[2]), b = fmax3(m[3], m[4], m[5]), c = fmax3(m[6], m[7], m[8]);
    return fmax3(fmax3(a, b, c), m[9], m[10]);
}

// 32 fp32 values (exact bf16 inputs) -> 32 E2M1 codes (element 2i in the
// low nibble of byte i) scaled by 2^-(byte - 127)
__device__ __forceinline__ uint4 e2m1x32_scaled(const float (&v)[32], int byte)
{
    const float inv = pow2_neg_e(byte);
    const uint64_t inv2 = f2pack(inv, inv);
    uint32_t c[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        float y[8];
#pragma unroll
        for (int i = 0; i < 4; ++i)
            f2unpack(fmul2(f2pack(v[8 * g + 2 * i], v[8 * g + 2 * i + 1]), inv2), y[2 * i], y[2 * i + 1]);
        c[g] = e2m1x8(y);
    }
    return make_uint4(c[0], c[1], c[2], c[3]);
}

// One 32-element MXFP4 block held by one lane (Sec. 3.2 Eq. 3-4; with RES
// the residual block of Sec. 4.3): the codes and E8M0 byte of X~, and of
// X^ = Q(X - X~).  The same arithmetic as mxfp4_quant8 on four lanes, with
// the block maximum, the scale and the residual computed once per block.
struct Mx32 {
    uint4 code, rcode;
    int sb, rb;
};

template <bool RES>
__device__ __forceinline__ Mx32 mxfp4_quant32(const float (&xf)[32])
{
    Mx32 o;
    o.sb = scale_byte_from_f32_bits(__float_as_uint(absmax32(xf)));
    o.code = e2m1x32_scaled(xf, o.sb);
    o.rcode = make_uint4(0, 0, 0, 0);
    o.rb = 0;
    if (RES) {
        const float nsc = -pow2_e(o.sb);
        const uint64_t nsc2 = f2pack(nsc, nsc);
        const uint32_t cw[4] = {o.code.x, o.code.y, o.code.z, o.code.w};
        float r[32];
#pragma unroll
        for (int g = 0; g < 4; ++g) {
            float q[8];
            e2m1x8_decode(cw[g], q);
#pragma unroll
            for (int i = 0; i < 4; ++i) // x - x~ (exact)
                f2unpack(ffma2(f2pack(q[2 * i], q[2 * i + 1]), nsc2, f2pack(xf[8 * g + 2 * i], xf[8 * g + 2 * i + 1])),
                         r[8 * g + 2 * i], r[8 * g + 2 * i + 1]);
        }
        o.rb = scale_byte_from_f32_bits(__float_as_uint(absmax32(r)));
        o.rcode = e2m1x32_scaled(r, o.rb);
    }
    return o;
}

// 16 words of bf16 pairs -> 32 fp32 values (exact)
__device__ __forceinline__ void bf16x32_to_f32(const uint32_t (&w)[16], float (&x)[32])
{
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        x[2 * i] = __uint_as_float(w[i] << 16);
        x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
}

} // namespace rfq
