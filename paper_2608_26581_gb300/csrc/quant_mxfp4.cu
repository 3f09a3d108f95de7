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
#include "mxfp4_math.cuh"

namespace rfq {
namespace {

RFQ_DEBUG_WORD_DECL

// Bytes of an MXFP4 scale array for `rows` rows of K (the MMA layout pads
// rows to 128): the extent of the debug build's bounds checks.
template <int LAYOUT>
__device__ __forceinline__ int64_t scale_bytes(int64_t rows, int64_t K)
{
    return (LAYOUT == RFQ_SCALE_MMA ? (rows + 127) / 128 * 128 : rows) * (K >> 5);
}

template <int LAYOUT>
__device__ __forceinline__ int64_t scale_index(int64_t m, int64_t b, int64_t kblocks)
{
    if (LAYOUT == RFQ_SCALE_MMA)
        return sf_mma_offset(m, b, kblocks >> 2);
    return m * kblocks + b;
}

// Items are (row, 1024-element segment): a warp handles one item, each lane
// one 32-element block (two 32-byte loads, the block's E8M0 scale, codes and
// residual computed in the lane, one 16-byte store of codes per pathway).
// (Four lanes per block with shuffles for the block maximum took 12% longer:
// the scale and the residual's scale were formed four times per block.)
constexpr int kSeg = 1024;

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
    const int kblocks = (int)(K >> 5);
    const int segs = (kblocks + 31) / 32;
    const int64_t items = M * segs;
    const int64_t gwarp = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;

    // Scale bytes of the padding rows of the MMA layout are zero.
    if (LAYOUT == RFQ_SCALE_MMA && pad_rows > 0) {
        const int64_t n = pad_rows * kblocks;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
            const int64_t off = scale_index<LAYOUT>(M + i / kblocks, i % kblocks, kblocks);
            if (!RFQ_IN_BOUNDS(off, scale_bytes<LAYOUT>(M, K)))
                continue;
            mscales[off] = 0;
            if (RES)
                rscales[off] = 0;
        }
    }

    uint4 *mc4 = reinterpret_cast<uint4 *>(mcodes);
    uint4 *rc4 = reinterpret_cast<uint4 *>(rcodes);
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
        const Mx32 qz = mxfp4_quant32<RES>(xf);
        if (!ok)
            continue;
        const int64_t soff = scale_index<LAYOUT>(m, b, kblocks);
        const int64_t coff = m * kblocks + b;               // 16-byte words of codes
        if (!RFQ_IN_BOUNDS(coff, M * kblocks) || !RFQ_IN_BOUNDS(soff, scale_bytes<LAYOUT>(M, K)))
            continue;
        mc4[coff] = qz.code;
        mscales[soff] = (uint8_t)qz.sb;
        if (RES) {
            const bool on = !PHI || phi[(m / p_s) * ((K + r_s - 1) / r_s) + ((int64_t)b * 32) / r_s] != 0;
            rc4[coff] = on ? qz.rcode : make_uint4(0, 0, 0, 0);
            rscales[soff] = on ? (uint8_t)qz.rb : 0;
        }
    }
}

// phi(p, r) = [max |x| over the p_s x r_s tile > tau]; one block per tile.
// |x| of a bf16 is the bf16 with its sign bit cleared, so the block takes a
// packed bf16x2 max over 16-byte loads (two bf16 per 32-bit lane; where one
// operand is NaN the max returns the other, so NaN is dropped as fmaxf
// would) and converts the winner to fp32 once.
// Rows are 16-byte aligned (K % 32 == 0); tiles whose column range is not a
// whole number of 8-element chunks take the scalar loop.
__global__ void __launch_bounds__(256) phi_amax_kernel(const __nv_bfloat16 *__restrict__ x, int64_t M, int64_t K,
                                                      int p_s, int r_s, float tau, uint8_t *__restrict__ phi)
{
    const int64_t nr = (K + r_s - 1) / r_s;
    const int64_t p = blockIdx.x / nr, r = blockIdx.x % nr;
    const int64_t m0 = p * p_s, k0 = r * r_s;
    const int rows = (int)(min(M, m0 + p_s) - m0), w = (int)(min(K, k0 + r_s) - k0);
    uint32_t acc = 0; // two packed 15-bit magnitudes
    if ((k0 & 7) == 0 && (w & 7) == 0) {
        const int cw = w >> 3, n = rows * cw;
        const __nv_bfloat16 *base = x + m0 * K + k0;
#pragma unroll 4
        for (int i = threadIdx.x; i < n; i += blockDim.x) {
            const int row = i / cw, c = i - row * cw;
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(base + (int64_t)row * K + 8 * c));
            const uint32_t q[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int j = 0; j < 4; ++j)
                asm("max.bf16x2 %0, %1, %2;" : "=r"(acc) : "r"(acc), "r"(q[j] & 0x7fff7fffu));
        }
    } else {
        for (int row = 0; row < rows; ++row)
            for (int c = threadIdx.x; c < w; c += blockDim.x) {
                const uint32_t mag = __bfloat16_as_ushort(x[(m0 + row) * K + k0 + c]) & 0x7fffu;
                asm("max.bf16x2 %0, %1, %2;" : "=r"(acc) : "r"(acc), "r"(mag));
            }
    }
    float a = fmaxf(__uint_as_float(acc << 16), __uint_as_float(acc & 0xffff0000u));
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

// AMAX fallback (Sec. 4.3) for phi tiles of 128 rows x 256 columns, fused
// into the quantizer: one block per tile stages the tile's 64 KB in shared
// memory with cp.async (warp w holds rows 16w .. 16w + 15, lane l the l-th
// 16-byte chunk of each; three blocks per SM), reduces max |x| over it (NaN
// dropped, as by phi_amax_kernel), writes phi, then quantizes the tile.  A
// phi = 0 tile's residual is written as zero codes and zero scales without
// being computed.  X is read from DRAM once, against twice for
// phi_amax_kernel followed by act_quant_mxfp4_kernel.  (Measured slower:
// the tile held in registers, two blocks per SM; splitting a tile over a
// cluster of 2 or 4 blocks that exchange their maxima through distributed
// shared memory; a persistent 512-thread form streaming the tiles through a
// cp.async ring.)
constexpr int kAmaxRows = 16; // rows per warp (8 warps = 128 rows)

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

template <int LAYOUT>
__global__ void __launch_bounds__(256, 3)
    act_quant_mxfp4_amax_kernel(const uint4 *__restrict__ x, int64_t M, int64_t K, uint32_t *__restrict__ mcodes,
                                uint8_t *__restrict__ mscales, uint32_t *__restrict__ rcodes,
                                uint8_t *__restrict__ rscales, uint8_t *__restrict__ phi, float tau)
{
    constexpr int R = kAmaxRows;
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
    auto row = [&](int i) { return lds128(sbase + 512 * i); };
    // max |x| as two packed bf16 magnitudes: sign bits cleared, then the
    // bf16x2 max, which returns the other operand where one is NaN (NaN
    // dropped, as in phi_amax_kernel); starts at +0
    uint32_t acc = 0;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const uint4 vi = row(i);
        const uint32_t q[4] = {vi.x, vi.y, vi.z, vi.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
            asm("max.bf16x2 %0, %1, %2;" : "=r"(acc) : "r"(acc), "r"(q[j] & 0x7fff7fffu));
    }
    const float am = fmaxf(__uint_as_float(acc << 16), __uint_as_float(acc & 0xffff0000u));
    __shared__ uint32_t red[8];
    const uint32_t wmax = __reduce_max_sync(0xFFFFFFFFu, __float_as_uint(am)); // am >= 0: integer order
    if (lane == 0)
        red[warp] = wmax;
    __syncthreads();
    uint32_t tmax = red[0];
#pragma unroll
    for (int i = 1; i < 8; ++i)
        tmax = max(tmax, red[i]);
    const bool on = __uint_as_float(tmax) > tau;
    if (threadIdx.x == 0)
        phi[tile] = on ? 1 : 0;

    const int b = c >> 2;
#pragma unroll
    for (int i = 0; i < R; ++i) {
        const int64_t m = m0 + i; // uniform over the warp
        const int64_t soff = scale_index<LAYOUT>(m, b, kblocks);
        // (the debug build's checks gate the stores only: the quantization
        // below takes all 32 lanes)
        const bool inb = RFQ_IN_BOUNDS(soff, scale_bytes<LAYOUT>(M, K)) &&
                         (m >= M || RFQ_IN_BOUNDS(m * kchunks + c, M * kchunks));
        if (m < M) {
            float xf[8];
            bf16x8_to_f32(row(i), xf);
            if (on) {
                const Mx8 qz = mxfp4_quant8<true>(xf);
                if (inb) {
                    mcodes[m * kchunks + c] = qz.code;
                    rcodes[m * kchunks + c] = qz.rcode;
                    if ((lane & 3) == 0) {
                        mscales[soff] = (uint8_t)qz.sb;
                        rscales[soff] = (uint8_t)qz.rb;
                    }
                }
            } else {
                const Mx8 qz = mxfp4_quant8<false>(xf);
                if (inb) {
                    mcodes[m * kchunks + c] = qz.code;
                    rcodes[m * kchunks + c] = 0u;
                    if ((lane & 3) == 0) {
                        mscales[soff] = (uint8_t)qz.sb;
                        rscales[soff] = 0;
                    }
                }
            }
        } else if (LAYOUT == RFQ_SCALE_MMA && (lane & 3) == 0 && inb) {
            // rows M .. of the last tile are the layout's padding rows
            mscales[soff] = 0;
            rscales[soff] = 0;
        }
    }
}

// Any bf16 with an all-ones exponent field (Inf or NaN) sets the status word.
__global__ void __launch_bounds__(256) check_finite_kernel(const uint4 *__restrict__ x, int64_t n8,
                                                          int32_t *__restrict__ status)
{
    bool bad = false;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8; i += (int64_t)gridDim.x * blockDim.x) {
        const uint4 v = __ldcs(x + i);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)   // both halves: exponent bits all ones
            bad |= ((w[j] & 0x7F800000u) == 0x7F800000u) || ((w[j] & 0x00007F80u) == 0x00007F80u);
    }
    if (__any_sync(0xFFFFFFFFu, bad) && (threadIdx.x & 31) == 0)
        atomicCAS(status, kDevOk, kDevNonFinite);
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
        if (LAYOUT == RFQ_SCALE_MMA && RFQ_IN_BOUNDS(scale_index<LAYOUT>(n, b, kblocks), scale_bytes<LAYOUT>(N, K)))
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
    if (!RFQ_IN_BOUNDS(n * (K >> 1) + b * 16 + 15, N * (K >> 1)) ||
        !RFQ_IN_BOUNDS(scale_index<LAYOUT>(n, b, kblocks), scale_bytes<LAYOUT>(N, K)))
        return;
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

cudaError_t launch_check_finite(const void *x, int64_t n8, int32_t *status, cudaStream_t st)
{
    check_finite_kernel<<<grid_for(n8, 256, 152 * 16), 256, 0, st>>>(static_cast<const uint4 *>(x), n8, status);
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
    if (mode == RFQ_FALLBACK_AMAX && p_s == 128 && r_s == 256 && K % 256 == 0) {
        // the GEMMs' phi granularity: one fused kernel (X read once)
        const unsigned tiles = (unsigned)(np * nr);
        auto *xi = static_cast<const uint4 *>(x);
        auto *mc = static_cast<uint32_t *>(mcodes);
        auto *ms = static_cast<uint8_t *>(mscales);
        auto *rc = static_cast<uint32_t *>(rcodes);
        auto *rs = static_cast<uint8_t *>(rscales);
        constexpr int smem = 128 * 256 * 2;   // the tile, staged in shared memory
        auto k = layout == RFQ_SCALE_MMA ? act_quant_mxfp4_amax_kernel<RFQ_SCALE_MMA>
                                         : act_quant_mxfp4_amax_kernel<RFQ_SCALE_ROWMAJOR>;
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess)
            return e;
        k<<<tiles, 256, smem, st>>>(xi, M, K, mc, ms, rc, rs, phi, tau);
        return cudaGetLastError();
    }
    if (mode == RFQ_FALLBACK_AMAX) {
        phi_amax_kernel<<<(unsigned)(np * nr), 256, 0, st>>>((const __nv_bfloat16 *)x, M, K, p_s, r_s, tau, phi);
    } else if (phi) {
        fill_u8_kernel<<<grid_for(np * nr, 256, 1024), 256, 0, st>>>(phi, np * nr, mode == RFQ_FALLBACK_ALL ? 1 : 0);
    }
    const int64_t pad = layout == RFQ_SCALE_MMA ? ((M + 127) / 128) * 128 - M : 0;
    const int64_t warps = M * ((K + kSeg - 1) / kSeg);
    const int64_t work = warps * 32 > pad * (K / 32) ? warps * 32 : pad * (K / 32);
    auto *xi = static_cast<const uint4 *>(x);
    auto *mc = static_cast<uint32_t *>(mcodes);
    auto *ms = static_cast<uint8_t *>(mscales);
    auto *rc = static_cast<uint32_t *>(rcodes);
    auto *rs = static_cast<uint8_t *>(rscales);
    // As many 256-thread blocks as are resident at once (registers limit
    // it), each warp looping over items: a grid beyond that runs a second,
    // partial wave (10% slower at six blocks per SM against four).
    auto grid = [&](auto kern) {
        return grid_for(work, 256, num_sms() * resident_blocks_per_sm((const void *)kern, 256, 0));
    };
#define RFQ_AQ(RES, PHI, LAY)                                                                                     \
    act_quant_mxfp4_kernel<RES, PHI, LAY><<<grid(act_quant_mxfp4_kernel<RES, PHI, LAY>), 256, 0, st>>>(            \
        xi, M, K, mc, ms, rc, rs, phi, p_s, r_s, pad)
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

RFQ_DEBUG_WORD_ACCESSOR(debug_word_quant_mxfp4)

} // namespace rfq
