// gemm_mxf4_fused.cu -- RFQ linear layer with the activation quantizer fused
// into the GEMM (the on-the-fly residual of Sec. 4.3; Algorithm 1 with the
// quantization of each X block done where the block is consumed):
//   Y = Q(X) W~ + phi Q(X - Q(X)) W~,   X bf16 read straight from HBM.
//
// Persistent kernel, one CTA per SM over 128 x 256 output tiles (704 threads):
//   warp 0       TMA producer of the W~ tile (128-byte swizzle) and its scale
//                atoms (bulk copies), three 68 KB stages
//   warp 1       MMA issuer: main + residual kind::mxf4 MMA per K=64 step
//                into one TMEM accumulator
//   warps 2-9    epilogue (TMEM -> bf16 / fp32 Y through shared memory and
//                TMA stores)
//   warps 10-13  scale writers: the stage's scale atoms from shared memory
//                into TMEM with tcgen05.st
//   warps 14-21  converters: for each 256-element k-stage, read the tile's
//                128 rows of bf16 X, quantize them (main codes and E8M0
//                bytes, residual codes and bytes: the same per-lane
//                arithmetic as the activation quantizer) and write the codes
//                straight into the swizzled A / R tiles and the bytes into
//                the scale atoms, then release the stage to the MMA thread.
// Every output tile re-quantizes its 128 rows of X for each N tile, so the
// converters' ALU work grows with N / 256: the variant pays off when N is
// small, and on wide layers the two-kernel path (quantizer + GEMM) is faster.
//
// fallback: ALL (phi = 1, residual everywhere) or NONE (plain W4A4).
//
// Every mbarrier wait is bounded (kWaitLimitNs, or the limit in the caller's
// workspace) and also gives up as soon as any CTA has recorded a timeout in
// the caller's status word; the CTA then drains its in-flight copies and MMAs
// (bounded), frees TMEM and returns.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"
#include "mxfp4_math.cuh"
#include "ptx.cuh"

namespace rfq {
namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 256;                // k-elements per stage (two 128-element chunks)
constexpr int ROW = BK / 2;            // bytes of codes per row per stage
constexpr int A_BYTES = BM * ROW;
constexpr int B_BYTES = BN * ROW;
constexpr int STAGES = 3;
constexpr int ATOM = 512;              // scale bytes of 128 rows x one 128-element chunk
constexpr int TMEM_COLS = 512;
constexpr int SF_COL0 = 256;           // TMEM columns [256, 384): scale slots
constexpr int SF_SLOT_COLS = 32;       // A chunk c at 4c, R at 8 + 4c, W~ at 16 + 8c (+4: rows 128-255)
constexpr int SF_SLOTS = 4;
constexpr int EPI_WARPS = 8;
constexpr int SF_WARPS = 4;
constexpr int CONV_WARPS = 8;
constexpr int CONV_WARP0 = 2 + EPI_WARPS + SF_WARPS;
constexpr int THREADS = 32 * (CONV_WARP0 + CONV_WARPS);
constexpr int YSTAGE = 2048;          // per epilogue warp: 32 rows x 64 bytes of Y
static_assert(SF_COL0 + SF_SLOTS * SF_SLOT_COLS <= TMEM_COLS, "TMEM budget");
static_assert(SF_SLOTS >= STAGES, "a scale slot is rewritten only after its stage's MMAs completed");
static_assert(BM % CONV_WARPS == 0, "converter rows");

struct alignas(1024) Stage {
    uint8_t a[A_BYTES];                // X~ codes, 128-byte swizzled K-major rows
    uint8_t r[A_BYTES];                // X^ codes
    uint8_t b[B_BYTES];                // W~ codes
    uint8_t sfa[2 * ATOM];             // chunk c at c * ATOM
    uint8_t sfr[2 * ATOM];
    uint8_t sfb[4 * ATOM];             // W~ rows 128 h..128 h + 127: chunk c at (2 h + c) * ATOM
};

struct Smem {
    Stage st[STAGES];
    alignas(1024) uint8_t ystage[EPI_WARPS * YSTAGE];
    uint64_t full[STAGES];            // W~ codes and scale atoms landed
    uint64_t conv[STAGES];            // the converters wrote the stage's A / R codes and scale atoms
    uint64_t empty[STAGES];           // the stage's MMAs completed
    uint64_t acc_full;
    uint64_t acc_empty;
    uint64_t drain;
    uint64_t sf_ready[SF_SLOTS];
    uint32_t tmem_base;
    uint64_t wait_ns;             // limit of the bounded waits (workspace word 1, else wl)
    int32_t abort_flag;
    int32_t issued;
};
constexpr size_t kSmemBytes = sizeof(Smem) + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

__device__ __forceinline__ void flag_timeout(Smem &S, int32_t *status)
{
    S.abort_flag = 1;
    atomicExch(status, kDevTimeout);
}

template <bool RES, bool OUT_BF16>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_mxf4_fused_kernel(const uint4 *__restrict__ x, const __grid_constant__ CUtensorMap tmB,
                           const __grid_constant__ CUtensorMap tmY, const uint8_t *__restrict__ sfb, int M, int N,
                           int K, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const volatile int32_t *gstat = status;

    // A bounded wait of an earlier CTA or call gave up: do nothing.
    if (threadIdx.x == 0) {
        S.abort_flag = *gstat;
        S.wait_ns = ws_wait_limit_ns(status);
    }
    __syncthreads();
    if (S.abort_flag != 0)
        return;
    const uint64_t wl = S.wait_ns;
    __syncthreads();

    const int kc = K >> 7;                 // 128-element chunks
    const int nks = (kc + 1) >> 1;         // k-stages (the last may hold one chunk)
    const int n_tiles = (N + BN - 1) / BN;
    const int m_tiles = (M + BM - 1) / BM;
    const int tiles = n_tiles * m_tiles;
    const int n_atoms = (N + 127) >> 7;    // 128-row scale atoms of W~

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.conv[s], CONV_WARPS);
            mbar_init(&S.empty[s], 1);
        }
        mbar_init(&S.acc_full, 1);
        mbar_init(&S.acc_empty, EPI_WARPS);
        mbar_init(&S.drain, 1);
        for (int i = 0; i < SF_SLOTS; ++i)
            mbar_init(&S.sf_ready[i], SF_WARPS);
        S.issued = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmB);
        prefetch_tmap(&tmY);
    }
    if (warp == 1) {
        tmem_alloc(&S.tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer (W~)
        if (lane == 0) {
            int p = 0;
            bool stop = false;
            if (!held_start_wait(status, wl)) { // a test-held start never opened
                flag_timeout(S, status);
                stop = true;
            }
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
                const int n_tile = tile % n_tiles;
                const int atom0 = n_tile * 2;
                const int nb = atom0 + 1 < n_atoms ? 2 : 1;
                for (int ks = 0; ks < nks; ++ks, ++p) {
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    const int c0 = 2 * ks, nch = min(2, kc - c0);
                    const uint32_t sfbytes = (uint32_t)nch * ATOM;
                    Stage &st = S.st[slot];
                    uint64_t *bar = &S.full[slot];
                    mbar_arrive_expect_tx(bar, B_BYTES + nb * sfbytes);
                    tma_load_2d(st.b, &tmB, bar, c0 * 64, n_tile * BN);
                    for (int h = 0; h < nb; ++h)
                        bulk_load(st.sfb + h * 2 * ATOM, sfb + ((int64_t)(atom0 + h) * kc + c0) * ATOM, sfbytes, bar);
                }
            }
            S.issued = p;
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int p = 0, it = 0;
            bool stop = false;
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x, ++it) {
                if (!mbar_wait(&S.acc_empty, (it & 1) ^ 1, wl, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                tc_fence_after();
                for (int ks = 0; ks < nks; ++ks, ++p) {
                    const int slot = p % STAGES, sfs = p % SF_SLOTS;
                    if (!mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat) ||
                        !mbar_wait(&S.conv[slot], (p / STAGES) & 1, wl, gstat) ||
                        !mbar_wait(&S.sf_ready[sfs], (p / SF_SLOTS) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    const int c0 = 2 * ks, nch = min(2, kc - c0);
                    const uint32_t sf = tmem + SF_COL0 + SF_SLOT_COLS * sfs;
                    const Stage &st = S.st[slot];
                    const uint32_t a0 = smem_u32(st.a), r0 = smem_u32(st.r), b0 = smem_u32(st.b);
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int c = j >> 1;
                        if (c >= nch)
                            break;
                        const uint32_t id = idesc_mxf4(BM, BN, 2 * (j & 1), 2 * (j & 1));
                        const uint64_t bd = sdesc_k_sw128(b0 + 32 * j);
                        const uint32_t sfb_t = sf + 16 + 8 * c;
                        tc_mma_mxf4(tmem, sdesc_k_sw128(a0 + 32 * j), bd, id, sf + 4 * c, sfb_t, (ks | j) != 0);
                        if (RES)
                            tc_mma_mxf4(tmem, sdesc_k_sw128(r0 + 32 * j), bd, id, sf + 8 + 4 * c, sfb_t, 1);
                    }
                    tc_commit(&S.empty[slot]);
                }
                if (!stop)
                    tc_commit(&S.acc_full);
            }
            if (S.abort_flag) {
                // wait (bounded) until every MMA issued above has completed
                tc_commit(&S.drain);
                (void)mbar_wait(&S.drain, 0, wl);
            }
        }
    } else if (warp < 2 + EPI_WARPS) {
        // ------------------------------------------------ epilogue (warps 2..9)
        const int q = warp & 3;          // TMEM lane quarter this warp may access
        const int h = (warp - 2) >> 2;   // column half of the tile
        uint8_t *stg = S.ystage + (warp - 2) * YSTAGE;
        const uint32_t sw = (uint32_t)((lane >> 1) & 3);   // 64B swizzle: chunk j of row r at (j ^ ((r >> 1) & 3))
        int it = 0;
        for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
            const int m_tile = tile / n_tiles, n_tile = tile - m_tile * n_tiles;
            // warp-uniform outcome: the tcgen05 loads below need the whole warp
            if (!__all_sync(0xffffffffu, mbar_wait(&S.acc_full, it & 1, wl, gstat))) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            tc_fence_after();
            const int row0 = m_tile * BM + q * 32;
            const uint32_t tcol = tmem + ((uint32_t)(q * 32) << 16) + h * (BN / 2);
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                // two 32-column chunks in flight; the accumulator goes back to
                // the MMA thread after the last load of the tile
                uint32_t v[2][32];
#pragma unroll
                for (int c = 0; c < 2; ++c)
                    tmem_ld_32x32b_x32(tcol + (2 * half + c) * 32, v[c]);
                tmem_ld_wait();
                if (half == 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive(&S.acc_empty);
                }
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    const int col = n_tile * BN + h * (BN / 2) + (2 * half + c) * 32;
                    if (col >= N || row0 >= M)
                        continue;
                    if (OUT_BF16) {
                        if (lane == 0)
                            bulk_wait_group_read<0>();
                        __syncwarp();
                        uint32_t pk[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(v[c][2 * i]),
                                                                      __uint_as_float(v[c][2 * i + 1]));
                            pk[i] = *reinterpret_cast<uint32_t *>(&b2);
                        }
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            *reinterpret_cast<uint4 *>(stg + lane * 64 + ((j ^ sw) << 4)) =
                                make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tmY, stg, col * 2, row0);
                            bulk_commit_group();
                        }
                    } else {
#pragma unroll
                        for (int hb = 0; hb < 2; ++hb) { // 16 fp32 columns (64 bytes) per store
                            if (col + 16 * hb >= N)
                                break;
                            if (lane == 0)
                                bulk_wait_group_read<0>();
                            __syncwarp();
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                *reinterpret_cast<uint4 *>(stg + lane * 64 + ((j ^ sw) << 4)) =
                                    make_uint4(v[c][16 * hb + 4 * j], v[c][16 * hb + 4 * j + 1],
                                               v[c][16 * hb + 4 * j + 2], v[c][16 * hb + 4 * j + 3]);
                            fence_proxy_async_smem();
                            __syncwarp();
                            if (lane == 0) {
                                tma_store_2d(&tmY, stg, (col + 16 * hb) * 4, row0);
                                bulk_commit_group();
                            }
                        }
                    }
                }
            }
            if (S.abort_flag)
                break;
        }
        if (lane == 0)
            bulk_wait_group<0>(); // every TMA store of this warp has completed
    } else if (warp < CONV_WARP0) {
        // ------------------------------------------------ scale writers (warps 10..13)
        // Warp quarter q writes TMEM lanes 32q..32q+31; every quarter holds
        // the same scale words (the MMA reads row 32 j + i from column j of
        // lane i of the quarter that computes it).
        const int q = warp & 3;
        int p = 0;
        bool stop = false;
        for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
            for (int ks = 0; ks < nks; ++ks, ++p) {
                const int slot = p % STAGES, sfs = p % SF_SLOTS;
                // warp-uniform outcome: the tcgen05 stores below need the whole warp
                if (!__all_sync(0xffffffffu, mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat) &&
                                                 mbar_wait(&S.conv[slot], (p / STAGES) & 1, wl, gstat))) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    stop = true;
                    break;
                }
                tc_fence_after();
                const int nch = min(2, kc - 2 * ks);
                const Stage &st = S.st[slot];
                const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + SF_COL0 + SF_SLOT_COLS * sfs;
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    if (c >= nch)
                        break;
                    const uint4 va = *reinterpret_cast<const uint4 *>(st.sfa + c * ATOM + lane * 16);
                    const uint4 vb0 = *reinterpret_cast<const uint4 *>(st.sfb + c * ATOM + lane * 16);
                    const uint4 vb1 = *reinterpret_cast<const uint4 *>(st.sfb + (2 + c) * ATOM + lane * 16);
                    tmem_st_32x32b_x4(tb + 4 * c, va.x, va.y, va.z, va.w);
                    if (RES) {
                        const uint4 vr = *reinterpret_cast<const uint4 *>(st.sfr + c * ATOM + lane * 16);
                        tmem_st_32x32b_x4(tb + 8 + 4 * c, vr.x, vr.y, vr.z, vr.w);
                    }
                    tmem_st_32x32b_x4(tb + 16 + 8 * c, vb0.x, vb0.y, vb0.z, vb0.w);
                    tmem_st_32x32b_x4(tb + 20 + 8 * c, vb1.x, vb1.y, vb1.z, vb1.w);
                }
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&S.sf_ready[sfs]);
            }
        }
    } else {
        // ------------------------------------------------ converters (warps 14..21)
        // Converter w handles rows w, w + 8, ... of the 128-row tile; one row
        // of a k-stage is 256 elements = one 16-byte load per lane, lanes
        // 4b..4b+3 forming the 32-element block b.
        const int w = warp - CONV_WARP0;
        const int64_t kchunks = K >> 3;    // 8-element chunks per row of X
        int p = 0;
        bool stop = false;
        for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
            const int m_tile = tile / n_tiles;
            for (int ks = 0; ks < nks; ++ks, ++p) {
                const int slot = p % STAGES;
                const int c0 = 2 * ks, nch = min(2, kc - c0);
                const bool lane_in = (lane >> 4) < nch;   // lanes 16..31 hold the second 128-element chunk
                // the stage's A / R / scale buffers are free once its previous MMAs completed
                if (!__all_sync(0xffffffffu, mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, wl, gstat))) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    stop = true;
                    break;
                }
                Stage &st = S.st[slot];
                const int j16 = lane >> 2;                    // 16-byte chunk of the 128-byte code row
                const int b = lane >> 2;                      // 32-element block of the stage
#pragma unroll 2
                for (int i = 0; i < BM / CONV_WARPS; i += 4) {
                    uint4 v[4];
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int r = w + CONV_WARPS * (i + u);
                        const int64_t m = (int64_t)m_tile * BM + r;
                        v[u] = (m < M && lane_in) ? __ldg(x + m * kchunks + (int64_t)c0 * 16 + lane)
                                                  : make_uint4(0, 0, 0, 0);
                    }
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int r = w + CONV_WARPS * (i + u);
                        float xf[8];
                        bf16x8_to_f32(v[u], xf);
                        const Mx8 qz = mxfp4_quant8<RES>(xf);
                        const int off = r * ROW + ((j16 ^ (r & 7)) << 4) + (lane & 3) * 4;   // 128-byte swizzle
                        *reinterpret_cast<uint32_t *>(st.a + off) = qz.code;
                        if (RES)
                            *reinterpret_cast<uint32_t *>(st.r + off) = qz.rcode;
                        if ((lane & 3) == 0) {
                            // scale atom: chunk b / 4, byte 16 (r % 32) + 4 ((r / 32) % 4) + b % 4
                            const int so = (b >> 2) * ATOM + (r & 31) * 16 + ((r >> 5) & 3) * 4 + (b & 3);
                            st.sfa[so] = (uint8_t)qz.sb;
                            if (RES)
                                st.sfr[so] = (uint8_t)qz.rb;
                        }
                    }
                }
                // codes are read by the tensor core (async proxy), scales by the writers
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&S.conv[slot]);
            }
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && S.abort_flag) {
        // wait (bounded) for the copies of the last stages still in flight
        const int issued = S.issued;
        for (int p = max(0, issued - STAGES); p < issued; ++p)
            (void)mbar_wait(&S.full[p % STAGES], (p / STAGES) & 1, wl);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <bool RES, bool OUT>
cudaError_t launch_variant(const GemmFusedArgs &a, const CUtensorMap &tb, const CUtensorMap &ty, cudaStream_t st)
{
    auto kern = gemm_mxf4_fused_kernel<RES, OUT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    const int64_t tiles = ((a.N + BN - 1) / BN) * ((a.M + BM - 1) / BM);
    const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
    kern<<<grid, THREADS, kSmemBytes, st>>>((const uint4 *)a.x, tb, ty, (const uint8_t *)a.b_sf, (int)a.M,
                                            (int)a.N, (int)a.K, a.status);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_gemm_mxf4_fused(const GemmFusedArgs &a, cudaStream_t st)
{
    CUtensorMap tb, ty;
    const uint64_t kb = (uint64_t)a.K / 2;
    if (!encode_tmap_2d_u8(&tb, a.b_codes, kb, (uint64_t)a.N, kb, ROW, BN, 128))
        return cudaErrorInvalidValue;
    // Y [M][N] (bf16 or fp32) as bytes; boxes of 64 bytes x 32 rows, 64B swizzle
    const uint64_t yrow = (uint64_t)a.N * (a.out_bf16 ? 2 : 4);
    if (!encode_tmap_2d_u8(&ty, a.y, yrow, (uint64_t)a.M, yrow, 64, 32, 64))
        return cudaErrorInvalidValue;
    if (a.residual)
        return a.out_bf16 ? launch_variant<true, true>(a, tb, ty, st) : launch_variant<true, false>(a, tb, ty, st);
    return a.out_bf16 ? launch_variant<false, true>(a, tb, ty, st) : launch_variant<false, false>(a, tb, ty, st);
}

} // namespace rfq
