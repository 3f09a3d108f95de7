// gemm_mxf4.cu -- RFQ GEMM on the sm_103a tensor cores (Algorithm 1,
// Eq. rfq):  Y = X~ W~ + phi X^ W~.
//
// One CTA computes a 128 x 256 output tile.  Per 256-element k-stage the TMA
// producer stages the main A tile (X~ codes), the residual A tile (X^
// codes), the W~ tile and the three E8M0 scale blocks in shared memory; the
// MMA thread copies the scales into TMEM (tcgen05.cp) and issues, for each
// K=64 step, the main MMA and the residual MMA against the SAME shared-memory
// W~ tile into the SAME TMEM accumulator.  W~ is therefore read once for both
// products, and the correction costs only MMA issue (the "streaming" residual
// accumulation of Sec. 4.3).  Residual MMAs of k-tiles with phi = 0 are not
// issued and their A tiles are not loaded.  Four epilogue warps read the
// fp32 accumulator from TMEM and store fp32 or bf16 Y.
//
// Scale layout in TMEM (per 128-element k-chunk): 4 columns per 128 rows,
// column j of lane i holding the four scales of row 32 j + i (written by
// tcgen05.cp 32x128b.warpx4 from the 512-byte MMA-layout atom).
//
// Every mbarrier wait is bounded (kWaitLimitNs); on expiry the CTA records
// kDevTimeout in the caller's workspace, drains its in-flight copies and
// MMAs (again with bounded waits), frees TMEM and returns.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace rfq {
namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 256;  // elements per k-stage (128 bytes of codes per row)
constexpr int STAGES = 3;
constexpr int A_BYTES = BM * BK / 2;
constexpr int B_BYTES = BN * BK / 2;
constexpr int SFA_BYTES = BM * BK / 32;
constexpr int SFB_BYTES = BN * BK / 32;
constexpr int TMEM_COLS = 512;
constexpr int SF_COL0 = 256;   // TMEM columns [256, 320): two scale slots of 32 columns

struct alignas(1024) Stage {
    uint8_t a[A_BYTES];
    uint8_t r[A_BYTES];
    uint8_t b[B_BYTES];
    uint8_t sfa[SFA_BYTES];
    uint8_t sfr[SFA_BYTES];
    uint8_t sfb[SFB_BYTES];
};

struct Smem {
    Stage st[STAGES];
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t acc_full;
    uint32_t tmem_base;
    int32_t abort_flag;
    int32_t issued;
};

constexpr size_t kSmemBytes = sizeof(Smem) + 1024;

__device__ __forceinline__ void flag_timeout(Smem &S, int32_t *status)
{
    S.abort_flag = 1;
    atomicExch(status, kDevTimeout);
}

__device__ __forceinline__ bool phi_on(const uint8_t *phi, int phi_cols, int m_tile, int chunk, int phi_chunks)
{
    return phi[(int64_t)m_tile * phi_cols + chunk / phi_chunks] != 0;
}

template <bool RES, bool PHI, bool OUT_BF16>
__global__ void __launch_bounds__(192, 1)
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
    const int n_tile = blockIdx.x, m_tile = blockIdx.y;
    const int kc = K >> 7;              // 128-element k-chunks
    const int nst = (kc + 1) >> 1;      // k-stages of 256 (the last may hold one chunk)
    const int n_atoms = (N + 127) >> 7; // 128-row scale atoms of W~

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.empty[s], 1);
        }
        mbar_init(&S.acc_full, 1);
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
            int s = 0;
            for (; s < nst; ++s) {
                const int slot = s % STAGES;
                const uint32_t ph = (s / STAGES) & 1;
                if (!mbar_wait(&S.empty[slot], ph ^ 1, kWaitLimitNs, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                const int nch = min(2, kc - 2 * s);
                bool res_on = RES;
                if (RES && PHI) {
                    res_on = phi_on(phi, phi_cols, m_tile, 2 * s, phi_chunks) ||
                             (nch > 1 && phi_on(phi, phi_cols, m_tile, 2 * s + 1, phi_chunks));
                }
                uint32_t bytes = A_BYTES + B_BYTES + nch * 512;
                if (res_on)
                    bytes += A_BYTES + nch * 512;
                for (int h = 0; h < 2; ++h)
                    if (n_tile * 2 + h < n_atoms)
                        bytes += nch * 512;
                Stage &st = S.st[slot];
                mbar_arrive_expect_tx(&S.full[slot], bytes);
                tma_load_2d(st.a, &tmA, &S.full[slot], s * (BK / 2), m_tile * BM);
                if (res_on)
                    tma_load_2d(st.r, &tmR, &S.full[slot], s * (BK / 2), m_tile * BM);
                tma_load_2d(st.b, &tmB, &S.full[slot], s * (BK / 2), n_tile * BN);
                bulk_load(st.sfa, sfa + ((int64_t)m_tile * kc + 2 * s) * 512, nch * 512, &S.full[slot]);
                if (res_on)
                    bulk_load(st.sfr, sfr + ((int64_t)m_tile * kc + 2 * s) * 512, nch * 512, &S.full[slot]);
                for (int h = 0; h < 2; ++h) {
                    const int atom = n_tile * 2 + h;
                    if (atom < n_atoms)
                        bulk_load(st.sfb + h * 1024, sfb + ((int64_t)atom * kc + 2 * s) * 512, nch * 512,
                                  &S.full[slot]);
                }
            }
            S.issued = s;
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            for (int s = 0; s < nst; ++s) {
                const int slot = s % STAGES;
                const uint32_t ph = (s / STAGES) & 1;
                if (!mbar_wait(&S.full[slot], ph, kWaitLimitNs, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                tc_fence_after();
                const int nch = min(2, kc - 2 * s);
                const Stage &st = S.st[slot];
                const uint32_t sf = tmem + SF_COL0 + (s & 1) * 32; // [0,8) A, [8,16) R, [16,32) B
                bool ron[2] = {RES, RES};
                if (RES && PHI) {
                    ron[0] = phi_on(phi, phi_cols, m_tile, 2 * s, phi_chunks);
                    ron[1] = nch > 1 && phi_on(phi, phi_cols, m_tile, 2 * s + 1, phi_chunks);
                }
                for (int c = 0; c < nch; ++c) {
                    tc_cp_32x128b_warpx4(sf + 4 * c, sdesc_rows16(smem_u32(st.sfa + 512 * c)));
                    if (ron[c])
                        tc_cp_32x128b_warpx4(sf + 8 + 4 * c, sdesc_rows16(smem_u32(st.sfr + 512 * c)));
                    tc_cp_32x128b_warpx4(sf + 16 + 8 * c, sdesc_rows16(smem_u32(st.sfb + 512 * c)));
                    tc_cp_32x128b_warpx4(sf + 16 + 8 * c + 4, sdesc_rows16(smem_u32(st.sfb + 1024 + 512 * c)));
                }
                const uint32_t a0 = smem_u32(st.a), r0 = smem_u32(st.r), b0 = smem_u32(st.b);
                for (int j = 0; j < 2 * nch; ++j) {
                    const int c = j >> 1;
                    const uint32_t id = idesc_mxf4(BM, BN, (j & 1) * 2, (j & 1) * 2);
                    const uint64_t bd = sdesc_k_sw128(b0 + 32 * j);
                    tc_mma_mxf4(tmem, sdesc_k_sw128(a0 + 32 * j), bd, id, sf + 4 * c, sf + 16 + 8 * c,
                                (s | j) != 0);
                    if (ron[c])
                        tc_mma_mxf4(tmem, sdesc_k_sw128(r0 + 32 * j), bd, id, sf + 8 + 4 * c, sf + 16 + 8 * c, 1);
                }
                tc_commit(&S.empty[slot]);
            }
            // Tracks every MMA issued above (also after an abort), so the
            // epilogue never reads, and teardown never frees, a busy TMEM.
            tc_commit(&S.acc_full);
        }
    } else {
        // ------------------------------------------------ epilogue (warps 2..5)
        const bool ok = mbar_wait(&S.acc_full, 0, kWaitLimitNs, gstat);
        if (!ok && lane == 0)
            flag_timeout(S, status);
        tc_fence_after();
        const int q = warp & 3; // TMEM lane quarter this warp may access
        const int row = m_tile * BM + q * 32 + lane;
        const bool store = ok && !S.abort_flag && row < M;
        for (int c = 0; c < BN / 32; ++c) {
            uint32_t v[32];
            tmem_ld_32x32b_x32(tmem + ((uint32_t)(q * 32) << 16) + c * 32, v);
            tmem_ld_wait();
            const int col = n_tile * BN + c * 32;
            if (!store || col >= N)
                continue;
            const int nvalid = min(32, N - col); // 16 or 32 (N % 16 == 0)
            if (OUT_BF16) {
                uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(Y) + (int64_t)row * N + col);
                uint32_t p[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) {
                    __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(v[2 * i]), __uint_as_float(v[2 * i + 1]));
                    p[i] = *reinterpret_cast<uint32_t *>(&h);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (i * 8 < nvalid)
                        dst[i] = make_uint4(p[4 * i], p[4 * i + 1], p[4 * i + 2], p[4 * i + 3]);
            } else {
                uint4 *dst = reinterpret_cast<uint4 *>(static_cast<float *>(Y) + (int64_t)row * N + col);
#pragma unroll
                for (int i = 0; i < 8; ++i)
                    if (i * 4 < nvalid)
                        dst[i] = make_uint4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
            }
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && S.abort_flag) {
        // wait (bounded) for the copies of the last stages still in flight
        const int issued = S.issued;
        for (int s = max(0, issued - STAGES); s < issued; ++s)
            (void)mbar_wait(&S.full[s % STAGES], (s / STAGES) & 1, kWaitLimitNs);
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
    dim3 grid((unsigned)((a.N + BN - 1) / BN), (unsigned)((a.M + BM - 1) / BM));
    const int phi_chunks = a.phi_r_s / 128;
    const int phi_cols = a.phi ? (int)((a.K + a.phi_r_s - 1) / a.phi_r_s) : 0;
    kern<<<grid, 192, kSmemBytes, st>>>(ta, tr, tb, (const uint8_t *)a.a_sf, (const uint8_t *)a.r_sf,
                                       (const uint8_t *)a.b_sf, a.phi, phi_chunks, phi_cols, a.y, (int)a.M,
                                       (int)a.N, (int)a.K, a.status);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_gemm_mxf4(const GemmMxf4Args &a, cudaStream_t st)
{
    CUtensorMap ta, tr, tb;
    const uint64_t kb = (uint64_t)a.K / 2;
    if (!encode_tmap_2d_u8(&ta, a.a_codes, kb, (uint64_t)a.M, kb, BK / 2, BM, true))
        return cudaErrorInvalidValue;
    if (!encode_tmap_2d_u8(&tb, a.b_codes, kb, (uint64_t)a.N, kb, BK / 2, BN, true))
        return cudaErrorInvalidValue;
    if (a.r_codes) {
        if (!encode_tmap_2d_u8(&tr, a.r_codes, kb, (uint64_t)a.M, kb, BK / 2, BM, true))
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
