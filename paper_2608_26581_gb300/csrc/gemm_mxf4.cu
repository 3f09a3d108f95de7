// gemm_mxf4.cu -- RFQ GEMM on the sm_103a tensor cores (Algorithm 1,
// Eq. rfq):  Y = X~ W~ + phi X^ W~.
//
// Persistent kernel: one CTA per SM walks output tiles of 128 x 256.  Per
// 128-element k-stage the TMA producer stages the main A tile (X~ codes), the
// residual A tile (X^ codes), the W~ tile and their E8M0 scale atoms in
// shared memory (six stages in flight).  The MMA thread copies the scales into
// TMEM (tcgen05.cp) and issues, per K=64 step, the main MMA and the residual
// MMA against the SAME shared-memory W~ tile into the SAME TMEM accumulator:
// W~ is read once for both products and the correction costs only MMA issue
// (the on-the-fly residual accumulation of Sec. 4.3).  Residual MMAs of
// k-tiles with phi = 0 are not issued and their A tiles are not loaded.
// Eight epilogue warps drain the fp32 accumulator (TMEM -> registers ->
// fp32 or bf16 Y); the producer keeps loading the next tile meanwhile, and the
// MMA thread starts it as soon as the accumulator has been read.
//
// Scale layout in TMEM (per 128-element k-chunk): 4 columns per 128 rows,
// column j of lane i holding the four scales of row 32 j + i (written by
// tcgen05.cp 32x128b.warpx4 from one 512-byte MMA-layout atom).
//
// Every mbarrier wait is bounded (kWaitLimitNs) and also gives up as soon as
// any CTA has recorded a timeout in the caller's status word; the CTA then
// drains its in-flight copies and MMAs (bounded), frees TMEM and returns.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace rfq {
namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 128; // elements per k-stage: 64 bytes of codes per row
constexpr int STAGES = 6;
constexpr int A_BYTES = BM * BK / 2;
constexpr int B_BYTES = BN * BK / 2;
constexpr int ATOM = 512;              // scale bytes of 128 rows x one 128-element chunk
constexpr int TMEM_COLS = 512;
constexpr int SF_COL0 = 256;           // TMEM columns [256, 320): four scale slots of 16 columns
constexpr int EPI_WARPS = 8;
constexpr int THREADS = 64 + 32 * EPI_WARPS;

struct alignas(1024) Stage {
    uint8_t a[A_BYTES];
    uint8_t r[A_BYTES];
    uint8_t b[B_BYTES];
    uint8_t sfa[ATOM];
    uint8_t sfr[ATOM];
    uint8_t sfb[2 * ATOM];
};

struct Smem {
    Stage st[STAGES];
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t acc_full;
    uint64_t acc_empty;
    uint64_t drain;
    uint32_t tmem_base;
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

template <bool RES, bool PHI, bool OUT_BF16>
__global__ void __launch_bounds__(THREADS, 1)
    gemm_mxf4_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmR,
                     const __grid_constant__ CUtensorMap tmB, const uint8_t *__restrict__ sfa,
                     const uint8_t *__restrict__ sfr, const uint8_t *__restrict__ sfb,
                     const uint8_t *__restrict__ phi, int phi_chunks, int phi_cols, void *__restrict__ Y, int M,
                     int N, int K, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const volatile int32_t *gstat = status;

    // A bounded wait of an earlier CTA or call gave up: do nothing.
    if (threadIdx.x == 0)
        S.abort_flag = *gstat;
    __syncthreads();
    if (S.abort_flag != 0)
        return;
    __syncthreads();

    const int kc = K >> 7;                 // k-stages (128-element chunks)
    const int n_tiles = (N + BN - 1) / BN;
    const int m_tiles = (M + BM - 1) / BM;
    const int tiles = n_tiles * m_tiles;
    const int n_atoms = (N + 127) >> 7;    // 128-row scale atoms of W~

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.empty[s], 1);
        }
        mbar_init(&S.acc_full, 1);
        mbar_init(&S.acc_empty, EPI_WARPS);
        mbar_init(&S.drain, 1);
        S.issued = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA);
        if (RES)
            prefetch_tmap(&tmR);
        prefetch_tmap(&tmB);
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
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int p = 0; // stages issued so far (ring position)
            bool stop = false;
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
                const int m_tile = tile / n_tiles, n_tile = tile - m_tile * n_tiles;
                for (int ks = 0; ks < kc; ++ks, ++p) {
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, kWaitLimitNs, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    const bool res_on =
                        RES && (!PHI || phi[(int64_t)m_tile * phi_cols + ks / phi_chunks] != 0);
                    uint32_t bytes = A_BYTES + B_BYTES + ATOM;
                    if (res_on)
                        bytes += A_BYTES + ATOM;
                    const int atom0 = n_tile * 2;
                    bytes += (atom0 + 1 < n_atoms ? 2 : 1) * ATOM;
                    Stage &st = S.st[slot];
                    uint64_t *bar = &S.full[slot];
                    mbar_arrive_expect_tx(bar, bytes);
                    tma_load_2d(st.a, &tmA, bar, ks * (BK / 2), m_tile * BM);
                    if (res_on)
                        tma_load_2d(st.r, &tmR, bar, ks * (BK / 2), m_tile * BM);
                    tma_load_2d(st.b, &tmB, bar, ks * (BK / 2), n_tile * BN);
                    bulk_load(st.sfa, sfa + ((int64_t)m_tile * kc + ks) * ATOM, ATOM, bar);
                    if (res_on)
                        bulk_load(st.sfr, sfr + ((int64_t)m_tile * kc + ks) * ATOM, ATOM, bar);
                    bulk_load(st.sfb, sfb + ((int64_t)atom0 * kc + ks) * ATOM, ATOM, bar);
                    if (atom0 + 1 < n_atoms)
                        bulk_load(st.sfb + ATOM, sfb + ((int64_t)(atom0 + 1) * kc + ks) * ATOM, ATOM, bar);
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
                const int m_tile = tile / n_tiles;
                if (!mbar_wait(&S.acc_empty, (it & 1) ^ 1, kWaitLimitNs, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                tc_fence_after();
                for (int ks = 0; ks < kc; ++ks, ++p) {
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.full[slot], (p / STAGES) & 1, kWaitLimitNs, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    tc_fence_after();
                    const bool res_on =
                        RES && (!PHI || phi[(int64_t)m_tile * phi_cols + ks / phi_chunks] != 0);
                    const Stage &st = S.st[slot];
                    const uint32_t sf = tmem + SF_COL0 + 16 * (p & 3); // [0,4) A, [4,8) R, [8,16) B
                    tc_cp_32x128b_warpx4(sf, sdesc_rows16(smem_u32(st.sfa)));
                    if (res_on)
                        tc_cp_32x128b_warpx4(sf + 4, sdesc_rows16(smem_u32(st.sfr)));
                    tc_cp_32x128b_warpx4(sf + 8, sdesc_rows16(smem_u32(st.sfb)));
                    tc_cp_32x128b_warpx4(sf + 12, sdesc_rows16(smem_u32(st.sfb + ATOM)));
                    const uint32_t a0 = smem_u32(st.a), r0 = smem_u32(st.r), b0 = smem_u32(st.b);
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const uint32_t id = idesc_mxf4(BM, BN, 2 * j, 2 * j);
                        const uint64_t bd = sdesc_k_sw64(b0 + 32 * j);
                        tc_mma_mxf4(tmem, sdesc_k_sw64(a0 + 32 * j), bd, id, sf, sf + 8, (ks | j) != 0);
                        if (res_on)
                            tc_mma_mxf4(tmem, sdesc_k_sw64(r0 + 32 * j), bd, id, sf + 4, sf + 8, 1);
                    }
                    tc_commit(&S.empty[slot]);
                }
                if (!stop)
                    tc_commit(&S.acc_full);
            }
            if (S.abort_flag) {
                // wait (bounded) until every MMA issued above has completed
                tc_commit(&S.drain);
                (void)mbar_wait(&S.drain, 0, kWaitLimitNs);
            }
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..9)
        const int q = warp & 3;          // TMEM lane quarter this warp may access
        const int h = (warp - 2) >> 2;   // column half of the tile
        int it = 0;
        for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
            const int m_tile = tile / n_tiles, n_tile = tile - m_tile * n_tiles;
            if (!mbar_wait(&S.acc_full, it & 1, kWaitLimitNs, gstat)) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            tc_fence_after();
            const int row = m_tile * BM + q * 32 + lane;
            const bool store = row < M;
#pragma unroll 1
            for (int c = 0; c < BN / 64; ++c) {
                const int col0 = h * (BN / 2) + c * 32;
                uint32_t v[32];
                tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + col0, v);
                tmem_ld_wait();
                if (c == BN / 64 - 1) {
                    // the accumulator is in registers: hand it back to the MMA thread
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive(&S.acc_empty);
                }
                const int col = n_tile * BN + col0;
                if (!store || col >= N)
                    continue;
                const int nvalid = min(32, N - col); // 16 or 32 (N % 16 == 0)
                if (OUT_BF16) {
                    uint4 *dst =
                        reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(Y) + (int64_t)row * N + col);
                    uint32_t pk[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        __nv_bfloat162 b2 =
                            __floats2bfloat162_rn(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
                        pk[i] = *reinterpret_cast<uint32_t *>(&b2);
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (i * 8 < nvalid)
                            dst[i] = make_uint4(pk[4 * i], pk[4 * i + 1], pk[4 * i + 2], pk[4 * i + 3]);
                } else {
                    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<float *>(Y) + (int64_t)row * N + col);
#pragma unroll
                    for (int i = 0; i < 8; ++i)
                        if (i * 4 < nvalid)
                            dst[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
                }
            }
            if (S.abort_flag)
                break;
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && S.abort_flag) {
        // wait (bounded) for the copies of the last stages still in flight
        const int issued = S.issued;
        for (int p = max(0, issued - STAGES); p < issued; ++p)
            (void)mbar_wait(&S.full[p % STAGES], (p / STAGES) & 1, kWaitLimitNs);
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <bool RES, bool PHI, bool OUT>
cudaError_t launch_variant(const CUtensorMap &ta, const CUtensorMap &tr, const CUtensorMap &tb,
                           const GemmMxf4Args &a, cudaStream_t st)
{
    auto kern = gemm_mxf4_kernel<RES, PHI, OUT>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    const int64_t tiles = ((a.N + BN - 1) / BN) * ((a.M + BM - 1) / BM);
    const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
    const int phi_chunks = a.phi_r_s / 128;
    const int phi_cols = a.phi ? (int)((a.K + a.phi_r_s - 1) / a.phi_r_s) : 0;
    kern<<<grid, THREADS, kSmemBytes, st>>>(ta, tr, tb, (const uint8_t *)a.a_sf, (const uint8_t *)a.r_sf,
                                            (const uint8_t *)a.b_sf, a.phi, phi_chunks, phi_cols, a.y, (int)a.M,
                                            (int)a.N, (int)a.K, a.status);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_gemm_mxf4(const GemmMxf4Args &a, cudaStream_t st)
{
    CUtensorMap ta, tr, tb;
    const uint64_t kb = (uint64_t)a.K / 2;
    if (!encode_tmap_2d_u8(&ta, a.a_codes, kb, (uint64_t)a.M, kb, BK / 2, BM, 64))
        return cudaErrorInvalidValue;
    if (!encode_tmap_2d_u8(&tb, a.b_codes, kb, (uint64_t)a.N, kb, BK / 2, BN, 64))
        return cudaErrorInvalidValue;
    if (a.r_codes) {
        if (!encode_tmap_2d_u8(&tr, a.r_codes, kb, (uint64_t)a.M, kb, BK / 2, BM, 64))
            return cudaErrorInvalidValue;
    } else {
        tr = ta;
    }
    const bool res = a.r_codes != nullptr, phi = res && a.phi != nullptr;
#define RFQ_GV(R, P, O) return launch_variant<R, P, O>(ta, tr, tb, a, st)
    if (!res) {
        if (a.out_bf16) RFQ_GV(false, false, true);
        RFQ_GV(false, false, false);
    }
    if (phi) {
        if (a.out_bf16) RFQ_GV(true, true, true);
        RFQ_GV(true, true, false);
    }
    if (a.out_bf16) RFQ_GV(true, false, true);
    RFQ_GV(true, false, false);
#undef RFQ_GV
}

} // namespace rfq
