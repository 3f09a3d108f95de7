// mma_peak.cu -- the dense block-scaled FP4 tensor rate of this GPU, measured
// with MMAs alone: the ceiling the RFQ GEMM's main and residual products
// (kind::mxf4, Algorithm 1 / Eq. rfq) are held against.
//
// Every SM (or CTA pair) issues `iters` back-to-back tcgen05 MMAs from one
// shared-memory operand tile into one TMEM accumulator, cycling through the
// four K = 64 steps of a 128-byte swizzled row as the GEMM does, with no
// copies, scale writes or epilogue: the kernel's time is the tensor pipe's.
// The operand bytes are a fixed pseudo-random pattern (E2M1 codes of every
// value and sign) and the scale bytes 2^0, so the pipe switches as it does on
// real data (an all-zero operand draws less power and would read faster
// under the power cap).
//   pair = 0: one CTA per SM, cta_group::1, 128 x 256 x 64 per MMA
//   pair = 1: clusters of two, cta_group::2, 256 x 256 x 64 per MMA (the
//             RFQ GEMM's form)
// The final wait is bounded (kWaitLimitNs); on expiry the kernel records
// kDevTimeout in the workspace and returns.
#include <cuda_runtime.h>
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace rfq {
namespace {

constexpr int A_BYTES = 128 * 128;   // 128 rows x 256 E2M1 codes
constexpr int B_BYTES = 256 * 128;   // 256 rows (pair: 128 per CTA, 256 staged anyway)
constexpr int THREADS = 128;
constexpr int TMEM_COLS = 512;
constexpr int SF_COL = 256;          // scale columns after the 256-column accumulator
// Dynamic shared memory per CTA: the tiles plus padding that keeps one CTA
// per SM (two would share TMEM and the tensor pipe).
constexpr size_t kSmemBytes = 160 * 1024;

struct Smem {
    alignas(1024) uint8_t a[A_BYTES];
    alignas(1024) uint8_t b[B_BYTES];
    uint64_t done;
    uint32_t tmem_base;
};
static_assert(sizeof(Smem) + 1024 <= kSmemBytes, "shared memory budget");

template <bool PAIR>
__global__ void __launch_bounds__(THREADS, 1) fp4_mma_peak_kernel(int64_t iters, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool lead = !PAIR || cluster_ctarank() == 0;

    // operand tiles: a multiplicative hash of the byte index
    for (int i = threadIdx.x; i < (A_BYTES + B_BYTES) / 4; i += THREADS) {
        const uint32_t v = (uint32_t)i * 2654435761u;
        if (i < A_BYTES / 4)
            reinterpret_cast<uint32_t *>(S.a)[i] = v ^ (v >> 15);
        else
            reinterpret_cast<uint32_t *>(S.b)[i - A_BYTES / 4] = v ^ (v >> 13);
    }
    fence_proxy_async_smem();
    if (threadIdx.x == 0) {
        mbar_init(&S.done, 1);
        fence_mbar_init();
    }
    if (warp == 0) {
        if (PAIR) {
            tmem_alloc_pair(&S.tmem_base, TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(&S.tmem_base, TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if (PAIR)
        cluster_sync();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    // scale words 2^0 (E8M0 127) in the 32 scale columns, every lane quarter
    {
        const uint32_t one = 0x7f7f7f7fu;
        const uint32_t t = tmem + ((uint32_t)(warp * 32) << 16) + SF_COL;
#pragma unroll
        for (int c = 0; c < 32; c += 4)
            tmem_st_32x32b_x4(t + c, one, one, one, one);
        tmem_st_wait();
    }
    tc_fence_before();
    __syncthreads();
    if (PAIR)
        cluster_sync();
    tc_fence_after();

    if (warp == 0 && lane == 0 && lead) {
        const uint32_t a0 = smem_u32(S.a), b0 = smem_u32(S.b);
        for (int64_t i = 0; i < iters; ++i) {
            const int j = (int)(i & 3);
            const uint64_t ad = sdesc_k_sw128(a0 + 32 * j), bd = sdesc_k_sw128(b0 + 32 * j);
            if (PAIR)
                tc_mma_mxf4_pair(tmem, ad, bd, idesc_mxf4(256, 256, 2 * (j & 1), 2 * (j & 1)), tmem + SF_COL,
                                 tmem + SF_COL + 16, i != 0);
            else
                tc_mma_mxf4(tmem, ad, bd, idesc_mxf4(128, 256, 2 * (j & 1), 2 * (j & 1)), tmem + SF_COL,
                            tmem + SF_COL + 16, i != 0);
        }
        if (PAIR)
            tc_commit_pair_mc(&S.done, 0x3);
        else
            tc_commit(&S.done);
    }
    if (warp == 0 && lane == 0) {
        // (pair: the commit arrives on both CTAs' barriers)
        if (!mbar_wait(&S.done, 0, kWaitLimitNs))
            atomicExch(status, kDevTimeout);
    }
    tc_fence_before();
    __syncthreads();
    if (PAIR)
        cluster_sync();
    if (warp == 0) {
        tc_fence_after();
        if (PAIR)
            tmem_dealloc_pair(tmem, TMEM_COLS);
        else
            tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <bool PAIR>
cudaError_t launch_peak(int64_t iters, int32_t *status, double *flop, cudaStream_t st)
{
    auto kern = fp4_mma_peak_kernel<PAIR>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    int grid = num_sms();
    if (PAIR) {
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cudaLaunchConfig_t lc = {};
        lc.gridDim = dim3(2 * (grid / 2));
        lc.blockDim = dim3(THREADS);
        lc.dynamicSmemBytes = kSmemBytes;
        lc.stream = st;
        lc.attrs = at;
        lc.numAttrs = 1;
        int n = 0;   // clusters of two resident at once
        e = cudaOccupancyMaxActiveClusters(&n, kern, &lc);
        if (e != cudaSuccess)
            return e;
        grid = 2 * (n > 0 ? n : 1);
        lc.gridDim = dim3(grid);
        *flop = 2.0 * 256 * 256 * 64 * (double)iters * (grid / 2);
        return cudaLaunchKernelEx(&lc, kern, iters, status);
    }
    *flop = 2.0 * 128 * 256 * 64 * (double)iters * grid;
    kern<<<grid, THREADS, kSmemBytes, st>>>(iters, status);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_fp4_mma_peak(int pair, int64_t iters, int32_t *status, double *flop, cudaStream_t st)
{
    return pair ? launch_peak<true>(iters, status, flop, st) : launch_peak<false>(iters, status, flop, st);
}

} // namespace rfq
