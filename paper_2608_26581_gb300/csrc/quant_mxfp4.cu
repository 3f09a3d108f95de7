// quant_mxfp4.cu -- MXFP4 quantization kernels for sm_103a.
//
//   act_quant_mxfp4   one pass over bf16 X [M x K]: per 32-element block the
//                     shared E8M0 exponent (Sec. 3.2 Eq. 3, OCP rule
//                     floor(log2 amax) - 2), the E2M1 codes (Eq. 4,
//                     round-to-nearest-even, saturating), the residual
//                     dX = X - X~ and its own MXFP4 block (Sec. 4.3).
//   phi_amax          fallback indicator tiles (Sec. 4.3) for the amax mode.
//   weight_quant      W [K x N] -> K-major MXFP4 (Sec. 4.3, Algorithm 1).
//   dequant           x = code * 2^(byte - 127).
//
// Exactness: every scaling is by a power of two, the residual x - q 2^e is
// exactly representable in fp32 (at most 11 significant bits), and the
// scale byte is read from the exponent field, so the kernels reproduce the
// fp64 definition bit for bit.  Built without fast-math / flush-to-zero so
// bf16 subnormals survive.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"

namespace rfq {
namespace {

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

template <int LAYOUT>
__device__ __forceinline__ int64_t scale_index(int64_t m, int64_t b, int64_t kblocks)
{
    if (LAYOUT == RFQ_SCALE_MMA)
        return sf_mma_offset(m, b, kblocks >> 2);
    return m * kblocks + b;
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

// Items are (row, 1024-element segment); a warp handles one item with four
// 16-byte loads per lane in flight; four consecutive lanes form one
// 32-element block.
constexpr int kSeg = 1024;
constexpr int kU = kSeg / 256;

template <bool RES, bool PHI, int LAYOUT>
__global__ void __launch_bounds__(256) act_quant_mxfp4_kernel(const uint4 *__restrict__ x, int64_t M, int64_t K,
                                                             uint32_t *__restrict__ mcodes,
                                                             uint8_t *__restrict__ mscales,
                                                             uint32_t *__restrict__ rcodes,
                                                             uint8_t *__restrict__ rscales,
                                                             const uint8_t *__restrict__ phi, int p_s, int r_s,
                                                             int64_t pad_rows)
{
    const int lane = threadIdx.x & 31;
    const int kchunks = (int)(K >> 3); // 8-element chunks per row
    const int kblocks = (int)(K >> 5);
    const int segs = (kchunks + kSeg / 8 - 1) / (kSeg / 8);
    const int64_t items = M * segs;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

    // Scale bytes of the padding rows of the MMA layout are zero.
    if (LAYOUT == RFQ_SCALE_MMA && pad_rows > 0) {
        const int64_t n = pad_rows * kblocks;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
            const int64_t off = scale_index<LAYOUT>(M + i / kblocks, i % kblocks, kblocks);
            mscales[off] = 0;
            if (RES)
                rscales[off] = 0;
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
        uint32_t *mrow = mcodes + m * kchunks;
        uint32_t *rrow = RES ? rcodes + m * kchunks : nullptr;
        // scale byte offset of (m, block 0) and the per-block step
        int64_t srow;
        if (LAYOUT == RFQ_SCALE_MMA)
            srow = ((m >> 7) * (int64_t)(kblocks >> 2) << 9) + ((m & 31) << 4) + (((m >> 5) & 3) << 2);
        else
            srow = m * kblocks;
        const uint8_t *prow = PHI ? phi + (m / p_s) * ((K + r_s - 1) / r_s) : nullptr;
#pragma unroll
        for (int j = 0; j < kU; ++j) {
            const int c = c0 + j * 32 + lane;
            const bool ok = c < kchunks; // uniform over each group of 4 lanes
            const int b = c >> 2;
            const int64_t soff = LAYOUT == RFQ_SCALE_MMA ? srow + ((b >> 2) << 9) + (b & 3) : srow + b;
            float xf[8];
            bf16x8_to_f32(v[j], xf);
            // block amax -> E8M0 byte from the exponent field (Sec. 3.2 Eq. 3, OCP rule)
            float am = absmax8(xf);
            am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 1));
            am = fmaxf(am, __shfl_xor_sync(0xFFFFFFFFu, am, 2));
            const int sb = scale_byte_from_f32_bits(__float_as_uint(am));
            const float inv = pow2_neg_e(sb);
            const uint64_t inv2 = f2pack(inv, inv);
            float y[8];
#pragma unroll
            for (int i = 0; i < 4; ++i)
                f2unpack(fmul2(f2pack(xf[2 * i], xf[2 * i + 1]), inv2), y[2 * i], y[2 * i + 1]);
            const uint32_t qc = e2m1x8(y);
            if (ok) {
                mrow[c] = qc;
                if ((lane & 3) == 0)
                    mscales[soff] = (uint8_t)sb;
            }
            if (RES) {
                const bool on = !PHI || (ok && prow[(c * 8) / r_s] != 0);
                float q[8], r[8];
                e2m1x8_decode(qc, q);
                const float nsc = -pow2_e(sb);
                const uint64_t nsc2 = f2pack(nsc, nsc);
#pragma unroll
                for (int i = 0; i < 4; ++i) // x - x~ (exact)
                    f2unpack(ffma2(f2pack(q[2 * i], q[2 * i + 1]), nsc2, f2pack(xf[2 * i], xf[2 * i + 1])),
                             r[2 * i], r[2 * i + 1]);
                float ra = absmax8(r);
                ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, 1));
                ra = fmaxf(ra, __shfl_xor_sync(0xFFFFFFFFu, ra, 2));
                const int rb = scale_byte_from_f32_bits(__float_as_uint(ra));
                const float rinv = pow2_neg_e(rb);
                const uint64_t rinv2 = f2pack(rinv, rinv);
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    f2unpack(fmul2(f2pack(r[2 * i], r[2 * i + 1]), rinv2), r[2 * i], r[2 * i + 1]);
                const uint32_t rc = e2m1x8(r);
                if (ok) {
                    rrow[c] = on ? rc : 0u;
                    if ((lane & 3) == 0)
                        rscales[soff] = on ? (uint8_t)rb : 0;
                }
            }
        }
    }
}

// phi(p, r) = [max |x| over the p_s x r_s tile > tau]; one block per tile.
__global__ void __launch_bounds__(256) phi_amax_kernel(const __nv_bfloat16 *__restrict__ x, int64_t M, int64_t K,
                                                      int p_s, int r_s, float tau, uint8_t *__restrict__ phi)
{
    const int64_t nr = (K + r_s - 1) / r_s;
    const int64_t p = blockIdx.x / nr, r = blockIdx.x % nr;
    const int64_t m0 = p * p_s, k0 = r * r_s;
    const int64_t m1 = min(M, m0 + p_s), k1 = min(K, k0 + r_s);
    const int64_t w = k1 - k0;
    float a = 0.f;
    for (int64_t i = threadIdx.x; i < (m1 - m0) * w; i += blockDim.x)
        a = fmaxf(a, fabsf(__bfloat162float(x[(m0 + i / w) * K + k0 + i % w])));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1)
        a = fmaxf(a, __shfl_xor_sync(0xFFFFFFFFu, a, o));
    __shared__ float red[8];
    if ((threadIdx.x & 31) == 0)
        red[threadIdx.x >> 5] = a;
    __syncthreads();
    if (threadIdx.x == 0) {
        for (int i = 1; i < (int)(blockDim.x >> 5); ++i)
            a = fmaxf(a, red[i]);
        phi[blockIdx.x] = a > tau ? 1 : 0;
    }
}

__global__ void fill_u8_kernel(uint8_t *p, int64_t n, uint8_t v)
{
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        p[i] = v;
}

// One thread per (column n, 32-block b) of W [K x N]: a warp reads 32
// consecutive columns of one K row at a time (coalesced).
template <int LAYOUT>
__global__ void __launch_bounds__(256) weight_quant_mxfp4_kernel(const __nv_bfloat16 *__restrict__ w, int64_t K,
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
            scales[scale_index<LAYOUT>(n, b, kblocks)] = 0;
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
    const int sb = scale_byte_from_f32_bits(am << 16);
    const float inv = pow2_neg_e(sb);
    uint32_t out[4];
#pragma unroll
    for (int g = 0; g < 4; ++g) {
        float y[8];
#pragma unroll
        for (int i = 0; i < 8; ++i)
            y[i] = xf[g * 8 + i] * inv;
        out[g] = e2m1x8(y);
    }
    *reinterpret_cast<uint4 *>(codes + n * (K >> 1) + b * 16) = make_uint4(out[0], out[1], out[2], out[3]);
    scales[scale_index<LAYOUT>(n, b, kblocks)] = (uint8_t)sb;
}

template <int LAYOUT>
__global__ void dequant_mxfp4_kernel(const uint32_t *__restrict__ codes, const uint8_t *__restrict__ scales,
                                     int64_t rows, int64_t k, float *__restrict__ out)
{
    const int64_t kchunks = k >> 3;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < rows * kchunks;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = c / kchunks, cc = c % kchunks;
        const int sb = scales[scale_index<LAYOUT>(m, cc >> 2, k >> 5)];
        float q[8];
        e2m1x8_decode(codes[c], q);
        const float s = pow2_e(sb);
        float4 *o = reinterpret_cast<float4 *>(out + c * 8);
        o[0] = make_float4(q[0] * s, q[1] * s, q[2] * s, q[3] * s);
        o[1] = make_float4(q[4] * s, q[5] * s, q[6] * s, q[7] * s);
    }
}

template <int LAYOUT>
__global__ void dequant_mxfp4_bf16_kernel(const uint32_t *__restrict__ codes, const uint8_t *__restrict__ scales,
                                          int64_t rows, int64_t k, uint4 *__restrict__ out)
{
    const int64_t kchunks = k >> 3;
    for (int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; c < rows * kchunks;
         c += (int64_t)gridDim.x * blockDim.x) {
        const int64_t m = c / kchunks, cc = c % kchunks;
        const int sb = scales[scale_index<LAYOUT>(m, cc >> 2, k >> 5)];
        float q[8];
        e2m1x8_decode(codes[c], q);
        const float s = pow2_e(sb);
        uint32_t p[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            // code value times a power of two: exact in bf16 except below its
            // normal range, where round-to-nearest-even applies
            __nv_bfloat162 b = __floats2bfloat162_rn(q[2 * i] * s, q[2 * i + 1] * s);
            p[i] = *reinterpret_cast<uint32_t *>(&b);
        }
        out[c] = make_uint4(p[0], p[1], p[2], p[3]);
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

cudaError_t launch_phi_amax(const void *x, int64_t M, int64_t K, int p_s, int r_s, float tau, uint8_t *phi,
                            cudaStream_t st)
{
    const int64_t np = (M + p_s - 1) / p_s, nr = (K + r_s - 1) / r_s;
    phi_amax_kernel<<<(unsigned)(np * nr), 256, 0, st>>>((const __nv_bfloat16 *)x, M, K, p_s, r_s, tau, phi);
    return cudaGetLastError();
}

cudaError_t launch_phi_fill(uint8_t *phi, int64_t n, int value, cudaStream_t st)
{
    fill_u8_kernel<<<grid_for(n, 256, 1024), 256, 0, st>>>(phi, n, (uint8_t)value);
    return cudaGetLastError();
}

cudaError_t launch_act_quant_mxfp4(const void *x, int64_t M, int64_t K, int mode, float tau, int p_s, int r_s,
                                   void *mcodes, void *mscales, void *rcodes, void *rscales, uint8_t *phi,
                                   int layout, cudaStream_t st)
{
    const int64_t np = (M + p_s - 1) / p_s, nr = (K + r_s - 1) / r_s;
    if (mode == RFQ_FALLBACK_AMAX) {
        phi_amax_kernel<<<(unsigned)(np * nr), 256, 0, st>>>((const __nv_bfloat16 *)x, M, K, p_s, r_s, tau, phi);
    } else if (phi) {
        fill_u8_kernel<<<grid_for(np * nr, 256, 1024), 256, 0, st>>>(phi, np * nr, mode == RFQ_FALLBACK_ALL ? 1 : 0);
    }
    const int64_t pad = layout == RFQ_SCALE_MMA ? ((M + 127) / 128) * 128 - M : 0;
    const int64_t warps = M * ((K + kSeg - 1) / kSeg);
    const int blocks = grid_for(warps * 32 > pad * (K / 32) ? warps * 32 : pad * (K / 32), 256, 152 * 24);
    auto *xi = static_cast<const uint4 *>(x);
    auto *mc = static_cast<uint32_t *>(mcodes);
    auto *ms = static_cast<uint8_t *>(mscales);
    auto *rc = static_cast<uint32_t *>(rcodes);
    auto *rs = static_cast<uint8_t *>(rscales);
#define RFQ_AQ(RES, PHI, LAY)                                                                                     \
    act_quant_mxfp4_kernel<RES, PHI, LAY><<<blocks, 256, 0, st>>>(xi, M, K, mc, ms, rc, rs, phi, p_s, r_s, pad)
    if (mode == RFQ_FALLBACK_NONE) {
        if (layout == RFQ_SCALE_MMA) RFQ_AQ(false, false, RFQ_SCALE_MMA);
        else RFQ_AQ(false, false, RFQ_SCALE_ROWMAJOR);
    } else if (mode == RFQ_FALLBACK_ALL) {
        if (layout == RFQ_SCALE_MMA) RFQ_AQ(true, false, RFQ_SCALE_MMA);
        else RFQ_AQ(true, false, RFQ_SCALE_ROWMAJOR);
    } else {
        if (layout == RFQ_SCALE_MMA) RFQ_AQ(true, true, RFQ_SCALE_MMA);
        else RFQ_AQ(true, true, RFQ_SCALE_ROWMAJOR);
    }
#undef RFQ_AQ
    return cudaGetLastError();
}

cudaError_t launch_weight_quant_mxfp4(const void *w, int64_t K, int64_t N, void *codes, void *scales, int layout,
                                      cudaStream_t st)
{
    const int64_t Npad = layout == RFQ_SCALE_MMA ? ((N + 127) / 128) * 128 : N;
    const int64_t work = Npad * (K / 32);
    const unsigned blocks = (unsigned)((work + 255) / 256);
    if (layout == RFQ_SCALE_MMA)
        weight_quant_mxfp4_kernel<RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>(
            (const __nv_bfloat16 *)w, K, N, Npad, (uint8_t *)codes, (uint8_t *)scales);
    else
        weight_quant_mxfp4_kernel<RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>(
            (const __nv_bfloat16 *)w, K, N, Npad, (uint8_t *)codes, (uint8_t *)scales);
    return cudaGetLastError();
}

cudaError_t launch_dequant_mxfp4(const void *codes, const void *scales, int64_t rows, int64_t k, int layout,
                                 float *out, cudaStream_t st)
{
    const int blocks = grid_for(rows * (k / 8), 256, 152 * 32);
    if (layout == RFQ_SCALE_MMA)
        dequant_mxfp4_kernel<RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>((const uint32_t *)codes, (const uint8_t *)scales,
                                                                     rows, k, out);
    else
        dequant_mxfp4_kernel<RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>((const uint32_t *)codes,
                                                                          (const uint8_t *)scales, rows, k, out);
    return cudaGetLastError();
}

cudaError_t launch_dequant_mxfp4_bf16(const void *codes, const void *scales, int64_t rows, int64_t k, int layout,
                                      void *out, cudaStream_t st)
{
    const int blocks = grid_for(rows * (k / 8), 256, 152 * 32);
    if (layout == RFQ_SCALE_MMA)
        dequant_mxfp4_bf16_kernel<RFQ_SCALE_MMA><<<blocks, 256, 0, st>>>(
            (const uint32_t *)codes, (const uint8_t *)scales, rows, k, (uint4 *)out);
    else
        dequant_mxfp4_bf16_kernel<RFQ_SCALE_ROWMAJOR><<<blocks, 256, 0, st>>>(
            (const uint32_t *)codes, (const uint8_t *)scales, rows, k, (uint4 *)out);
    return cudaGetLastError();
}

} // namespace rfq
