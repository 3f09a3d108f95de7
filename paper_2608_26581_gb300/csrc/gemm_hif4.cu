// gemm_hif4.cu -- RFQ GEMM with HiF4 activations (Sec. 3.3, Sec. 4.3,
// Algorithm 1):  Y = X~ W~ + phi X^ W~.
//
// HiF4 has no tensor-core format (its macro scale carries a 2-bit mantissa
// and the per-4-element exponents are finer than any block scale), but every
// HiF4 value is exactly a bf16: k (3 bits) times S (3 significant bits) times
// a power of two.  So the GEMM runs bf16 tcgen05 MMAs (kind::f16) on exact
// expansions:
//   - W~ comes as its bf16 expansion [N][K] (done once, rfq_dequant), loaded
//     by TMA with the 128-byte swizzle;
//   - the main and residual activation tiles are loaded as HiF4 codes plus
//     block metadata and expanded to bf16 in shared memory by eight converter
//     warps, written directly in the swizzled layout the MMA reads.
// Per 64-element k-stage (one HiF4 block per row) the MMA thread issues four
// K=16 MMAs for X~ and four for X^ against the same W~ tile into the same
// TMEM accumulator.  The accumulator is double-buffered (2 x 256 columns; no
// scale columns are needed), so four epilogue warps drain tile t while the
// MMAs of tile t+1 run.  Waits are bounded as in the MXFP4 GEMM.
//
// Selective phi: stages of phi = 0 skip the residual load and MMAs.  As in
// the CTA-pair MXFP4 GEMM, an extra warp writes one record per output tile (a
// bit per k-stage, set when phi = 1, and their count), the producer issues
// the residual stages first and publishes the count with every stage, and
// the MMA thread runs two loops with compile-time residual flags: a branch
// on a per-stage flag in the MMA thread slows its MMA issue.
#include <cuda_bf16.h>
#include <cstdint>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace rfq {
namespace {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;                        // elements per k-stage = one HiF4 block
constexpr int STAGES = 3;
constexpr int CODE_BYTES = BM * BK / 2;       // 4 KB of codes per 128 rows
constexpr int META_BYTES = BM * 4;
constexpr int A16_BYTES = BM * BK * 2;        // 16 KB bf16 tile
constexpr int B16_BYTES = BN * BK * 2;        // 32 KB bf16 tile
constexpr int CONV_WARPS = 8;
constexpr int EPI_WARPS = 4;
constexpr int THREADS = 64 + 32 * EPI_WARPS + 32 * CONV_WARPS;
constexpr int PHI_WARP = THREADS / 32;        // the phi reader: one warp beyond THREADS
constexpr int REC_WORDS = 64;                 // phi record: up to 2048 k-stages (K <= 131072)

// Selective phi, one output tile: bit ks of bits set when the residual of
// k-stage ks applies; count = the number of set bits.
struct PhiRec {
    uint32_t bits[REC_WORDS];
    uint32_t count;
};
constexpr int TMEM_COLS = 512;

struct alignas(1024) Stage {
    uint8_t b[B16_BYTES];      // W~ bf16, 128B-swizzled (TMA)
    uint8_t a16[A16_BYTES];    // X~ bf16, 128B-swizzled (converters)
    uint8_t r16[A16_BYTES];    // X^ bf16
    uint8_t acode[CODE_BYTES]; // X~ HiF4 codes, 32 bytes per row
    uint8_t rcode[CODE_BYTES];
    uint32_t ameta[BM];
    uint32_t rmeta[BM];
};

// Operands already expanded to bf16 (X~, X^ and W~ all loaded by TMA).
struct alignas(1024) Stage16 {
    uint8_t b[B16_BYTES];
    uint8_t a16[A16_BYTES];
    uint8_t r16[A16_BYTES];
};

constexpr int YSTAGE = 2048; // per epilogue warp: 32 rows x 64 bytes of Y

template <bool CONV>
struct Smem {
    typename std::conditional<CONV, Stage, Stage16>::type st[STAGES];
    alignas(1024) uint8_t ystage[CONV ? 16 : EPI_WARPS * YSTAGE];
    uint64_t full[STAGES];
    uint64_t conv[STAGES];
    uint64_t empty[STAGES];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t drain;
    uint64_t phi_full[2];      // the phi reader filled the record
    uint64_t phi_empty[2];     // the producer consumed the record
    PhiRec rec[2];
    uint32_t stage_info[STAGES]; // the tile's residual-stage count | (this stage's residual applies) << 31
    uint32_t tmem_base;
    uint64_t wait_ns;             // limit of the bounded waits (workspace word 1, else wl)
    int32_t abort_flag;
    int32_t issued;
};

template <bool CONV>
constexpr size_t smem_bytes() { return sizeof(Smem<CONV>) + 1024; }
static_assert(smem_bytes<true>() <= 227 * 1024 && smem_bytes<false>() <= 227 * 1024, "shared memory budget");

template <class SM>
__device__ __forceinline__ void flag_timeout(SM &S, int32_t *status)
{
    S.abort_flag = 1;
    atomicExch(status, kDevTimeout);
}

// 8 HiF4 codes of group g of a block -> 8 bf16 (exact), packed in a uint4.
__device__ __forceinline__ uint4 hif4_group_to_bf16(uint32_t cw, uint32_t meta, int g)
{
    const int E = (int)((meta >> 2) & 63), Mm = (int)(meta & 3);
    const float S = __uint_as_float(((uint32_t)(E - 48 + 127) << 23) | ((uint32_t)Mm << 21));
    const int e18 = (int)((meta >> (8 + g)) & 1);
    const float s0 = 0.25f * S * (float)(1 << (e18 + (int)((meta >> (16 + 2 * g)) & 1)));
    const float s1 = 0.25f * S * (float)(1 << (e18 + (int)((meta >> (17 + 2 * g)) & 1)));
    uint32_t out[4];
#pragma unroll
    for (int p = 0; p < 4; ++p) {
        const uint32_t c0 = (cw >> (8 * p)) & 0xF, c1 = (cw >> (8 * p + 4)) & 0xF;
        const float st = p < 2 ? s0 : s1;
        // k as float via the 2^23 magic (exact), times the step (exact), sign from the code
        float v0 = (__uint_as_float(0x4B000000u | (c0 & 7)) - 8388608.f) * st;
        float v1 = (__uint_as_float(0x4B000000u | (c1 & 7)) - 8388608.f) * st;
        const uint32_t b0 = (__float_as_uint(v0) >> 16) | ((c0 & 8) << 12);
        const uint32_t b1 = (__float_as_uint(v1) & 0xFFFF0000u) | ((c1 & 8) << 28);
        out[p] = b0 | b1;
    }
    return make_uint4(out[0], out[1], out[2], out[3]);
}

// CONV: the activation operands are HiF4 codes + metadata expanded in the
// kernel; otherwise they are bf16 expansions loaded by TMA like W~.
template <bool B>
struct Bool {
    static constexpr bool value = B;
};

template <bool CONV, bool RES, bool PHI, bool OUT_BF16>
__global__ void __launch_bounds__(PHI ? THREADS + 32 : THREADS, 1)
    gemm_hif4_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmR,
                     const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmY,
                     const uint32_t *__restrict__ ameta,
                     const uint32_t *__restrict__ rmeta, const uint8_t *__restrict__ phi, int phi_blocks,
                     int phi_cols, void *__restrict__ Y, int M, int N, int K, int32_t *status)
{
    extern __shared__ uint8_t smem_raw[];
    Smem<CONV> &S =
        *reinterpret_cast<Smem<CONV> *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const volatile int32_t *gstat = status;

    if (threadIdx.x == 0) {
        S.abort_flag = *gstat;
        S.wait_ns = ws_wait_limit_ns(status);
    }
    __syncthreads();
    if (S.abort_flag != 0)
        return;
    const uint64_t wl = S.wait_ns;
    __syncthreads();

    const int nks = K / BK;
    const int n_tiles = (N + BN - 1) / BN;
    const int m_tiles = (M + BM - 1) / BM;
    const int tiles = n_tiles * m_tiles;
    const int64_t mpad = (int64_t)m_tiles * BM; // rows of the block-major metadata

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.conv[s], CONV ? CONV_WARPS : 1);
            mbar_init(&S.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&S.acc_full[b], 1);
            mbar_init(&S.acc_empty[b], EPI_WARPS);
        }
        mbar_init(&S.drain, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&S.phi_full[i], 32);
            mbar_init(&S.phi_empty[i], 1);
        }
        S.issued = 0;
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA);
        if (RES)
            prefetch_tmap(&tmR);
        prefetch_tmap(&tmB);
        if (!CONV)
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
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int p = 0, it = 0;
            bool stop = false;
            if (!held_start_wait(status, wl)) { // a test-held start never opened
                flag_timeout(S, status);
                stop = true;
            }
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x, ++it) {
                const int m_tile = tile / n_tiles, n_tile = tile - m_tile * n_tiles;
                // one k-stage: wait for its ring slot, publish the tile's info and
                // the stage's residual flag, issue the copies
                auto produce = [&](int ks, uint32_t count, auto res_t) {
                    constexpr bool ron = decltype(res_t)::value;
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    S.stage_info[slot] = count | (ron ? 1u << 31 : 0u);
                    auto &st = S.st[slot];
                    uint64_t *bar = &S.full[slot];
                    if constexpr (CONV) {
                        uint32_t bytes = B16_BYTES + CODE_BYTES + META_BYTES;
                        if (ron)
                            bytes += CODE_BYTES + META_BYTES;
                        mbar_arrive_expect_tx(bar, bytes);
                        tma_load_2d(st.b, &tmB, bar, ks * BK * 2, n_tile * BN);
                        tma_load_2d(st.acode, &tmA, bar, ks * BK / 2, m_tile * BM);
                        bulk_load(st.ameta, ameta + ks * mpad + (int64_t)m_tile * BM, META_BYTES, bar);
                        if (ron) {
                            tma_load_2d(st.rcode, &tmR, bar, ks * BK / 2, m_tile * BM);
                            bulk_load(st.rmeta, rmeta + ks * mpad + (int64_t)m_tile * BM, META_BYTES, bar);
                        }
                    } else {
                        mbar_arrive_expect_tx(bar, B16_BYTES + A16_BYTES + (ron ? A16_BYTES : 0));
                        tma_load_2d(st.b, &tmB, bar, ks * BK * 2, n_tile * BN);
                        tma_load_2d(st.a16, &tmA, bar, ks * BK * 2, m_tile * BM);
                        if (ron)
                            tma_load_2d(st.r16, &tmR, bar, ks * BK * 2, m_tile * BM);
                    }
                    ++p;
                };
                if constexpr (!PHI) {
                    for (int ks = 0; ks < nks && !stop; ++ks)
                        produce(ks, 0u, Bool<RES>{});
                } else {
                    const int r = it & 1;
                    if (!mbar_wait(&S.phi_full[r], (it >> 1) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    const PhiRec &rec = S.rec[r];
                    const uint32_t count = rec.count;
                    // stages with a residual, then the others, each in k order
                    for (int w = 0; 32 * w < nks && !stop; ++w) {
                        uint32_t x = rec.bits[w];
                        while (x != 0 && !stop) {
                            const int b = __ffs(x) - 1;
                            x &= x - 1;
                            produce(32 * w + b, count, Bool<true>{});
                        }
                    }
                    for (int w = 0; 32 * w < nks && !stop; ++w) {
                        const int left = nks - 32 * w;
                        uint32_t x = ~rec.bits[w] & (left >= 32 ? 0xffffffffu : (1u << left) - 1u);
                        while (x != 0 && !stop) {
                            const int b = __ffs(x) - 1;
                            x &= x - 1;
                            produce(32 * w + b, count, Bool<false>{});
                        }
                    }
                    mbar_arrive(&S.phi_empty[r]);
                }
            }
            S.issued = p;
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        if (lane == 0) {
            int p = 0, it = 0;
            bool stop = false;
            const uint32_t idesc = idesc_bf16(BM, BN);
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x, ++it) {
                const int buf = it & 1;
                if (!mbar_wait(&S.acc_empty[buf], ((it >> 1) & 1) ^ 1, wl, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                tc_fence_after();
                const uint32_t acc = tmem + 256 * buf;
                // the MMAs of the stage at position pos of the tile
                auto mma_stage = [&](int pos, auto res_t) {
                    constexpr bool ron = decltype(res_t)::value;
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat) ||
                        (CONV && !mbar_wait(&S.conv[slot], (p / STAGES) & 1, wl, gstat))) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    tc_fence_after();
                    const auto &st = S.st[slot];
                    const uint32_t a0 = smem_u32(st.a16), r0 = smem_u32(st.r16), b0 = smem_u32(st.b);
#pragma unroll
                    for (int j = 0; j < BK / 16; ++j) {
                        const uint64_t bd = sdesc_k_sw128(b0 + 32 * j);
                        tc_mma_f16(acc, sdesc_k_sw128(a0 + 32 * j), bd, idesc, (pos | j) != 0);
                        if (ron)
                            tc_mma_f16(acc, sdesc_k_sw128(r0 + 32 * j), bd, idesc, 1);
                    }
                    tc_commit(&S.empty[slot]);
                    ++p;
                };
                if constexpr (!PHI) {
                    for (int ks = 0; ks < nks && !stop; ++ks)
                        mma_stage(ks, Bool<RES>{});
                } else {
                    // the tile's residual-stage count arrives with its first stage
                    if (!mbar_wait(&S.full[p % STAGES], (p / STAGES) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        break;
                    }
                    const int n_res = (int)(S.stage_info[p % STAGES] & 0x7fffffffu);
                    int pos = 0;
                    for (; pos < n_res && !stop; ++pos)
                        mma_stage(pos, Bool<true>{});
                    for (; pos < nks && !stop; ++pos)
                        mma_stage(pos, Bool<false>{});
                }
                if (!stop)
                    tc_commit(&S.acc_full[buf]);
            }
            if (S.abort_flag) {
                tc_commit(&S.drain);
                (void)mbar_wait(&S.drain, 0, wl);
            }
        }
    } else if (warp < 2 + EPI_WARPS) {
        // ------------------------------------------------ epilogue (warps 2..5)
        const int q = warp & 3;
        int it = 0;
        for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++it) {
            const int m_tile = tile / n_tiles, n_tile = tile - m_tile * n_tiles;
            const int buf = it & 1;
            if (!mbar_wait(&S.acc_full[buf], (it >> 1) & 1, wl, gstat)) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            tc_fence_after();
            const int row = m_tile * BM + q * 32 + lane;
            const bool store = row < M;
            const uint32_t acc = tmem + 256 * buf + ((uint32_t)(q * 32) << 16);
            uint8_t *stg = S.ystage + (CONV ? 0 : (warp - 2) * YSTAGE);
#pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                uint32_t v[32];
                tmem_ld_32x32b_x32(acc + c * 32, v);
                tmem_ld_wait();
                if (c == BN / 32 - 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0)
                        mbar_arrive(&S.acc_empty[buf]);
                }
                const int col = n_tile * BN + c * 32;
                if (col >= N)
                    continue;
                if (!CONV) {
                    // shared-memory stage (64B swizzle) + TMA store, clipped at M and N
                    const uint32_t sw = (uint32_t)((lane >> 1) & 3);
#pragma unroll
                    for (int hb = 0; hb < (OUT_BF16 ? 1 : 2); ++hb) {
                        if (col + 16 * hb >= N)
                            break;
                        if (lane == 0)
                            bulk_wait_group_read<0>();
                        __syncwarp();
                        uint32_t pk[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            if (OUT_BF16) {
                                __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(v[2 * i]),
                                                                          __uint_as_float(v[2 * i + 1]));
                                pk[i] = *reinterpret_cast<uint32_t *>(&b2);
                            } else {
                                pk[i] = v[16 * hb + i];
                            }
                        }
#pragma unroll
                        for (int j = 0; j < 4; ++j)
                            *reinterpret_cast<uint4 *>(stg + lane * 64 + ((j ^ sw) << 4)) =
                                make_uint4(pk[4 * j], pk[4 * j + 1], pk[4 * j + 2], pk[4 * j + 3]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tmY, stg, OUT_BF16 ? col * 2 : (col + 16 * hb) * 4, m_tile * BM + q * 32);
                            bulk_commit_group();
                        }
                    }
                    continue;
                }
                if (!store)
                    continue;
                const int nvalid = min(32, N - col);
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
        if (!CONV && lane == 0)
            bulk_wait_group<0>(); // every TMA store of this warp has completed
    } else if (warp < PHI_WARP) {
        if constexpr (CONV) {
        // ------------------------------------------------ converters (warps 6..13)
        // 2 x 128 rows x 8 groups of 8 elements per stage; thread u handles
        // chunks u, u + 256, ... (row = chunk / 8, group = chunk % 8).
        const int u = threadIdx.x - 32 * (2 + EPI_WARPS);
        int p = 0;
        bool stop = false;
        for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
            for (int ks = 0; ks < nks; ++ks, ++p) {
                const int slot = p % STAGES;
                if (!mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat)) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    stop = true;
                    break;
                }
                auto &st = S.st[slot];
                const bool ron = RES && (!PHI || (S.stage_info[slot] >> 31) != 0);
#pragma unroll 2
                for (int ch = u; ch < 2 * BM * 8; ch += 32 * CONV_WARPS) {
                    const bool isr = ch >= BM * 8;
                    if (isr && !ron)
                        break;
                    const int cc = isr ? ch - BM * 8 : ch;
                    const int row = cc >> 3, g = cc & 7;
                    const uint32_t cw = *reinterpret_cast<const uint32_t *>((isr ? st.rcode : st.acode) + row * 32 + g * 4);
                    const uint32_t md = (isr ? st.rmeta : st.ameta)[row];
                    const uint4 v = hif4_group_to_bf16(cw, md, g);
                    uint8_t *dst = (isr ? st.r16 : st.a16) + row * 128 + ((g ^ (row & 7)) << 4);
                    *reinterpret_cast<uint4 *>(dst) = v;
                }
                // make the generic-proxy stores visible to the tensor core (async proxy)
                asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&S.conv[slot]);
            }
        }
        }
    }
    if constexpr (PHI) {
        if (warp == PHI_WARP) {
            // -------------------------------------------- phi reader
            // Record of the CTA's j-th tile: stage ks of row tile m needs its
            // residual when phi[m][ks / phi_blocks] is non-zero.
            const int my_tiles =
                (int)blockIdx.x < tiles ? (tiles - (int)blockIdx.x + (int)gridDim.x - 1) / (int)gridDim.x : 0;
            for (int j = 0; j < my_tiles; ++j) {
                const int r = j & 1;
                if (j >= 2 && !__all_sync(0xffffffffu, mbar_wait(&S.phi_empty[r], ((j >> 1) - 1) & 1,
                                                                 wl, gstat))) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    break;
                }
                const int m_tile = ((int)blockIdx.x + j * (int)gridDim.x) / n_tiles;
                PhiRec &rec = S.rec[r];
                uint32_t count = 0;
                for (int w = 0; 32 * w < nks; ++w) {
                    const int ks = 32 * w + lane;
                    const bool on = ks < nks && __ldg(phi + (int64_t)m_tile * phi_cols + ks / phi_blocks) != 0;
                    const uint32_t word = __ballot_sync(0xffffffffu, on);
                    if (lane == 0)
                        rec.bits[w] = word;
                    count += __popc(word);
                }
                if (lane == 0)
                    rec.count = count;
                mbar_arrive(&S.phi_full[r]);
            }
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && S.abort_flag) {
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

template <bool CONV, bool RES, bool PHI, bool OUT>
cudaError_t launch_variant(const CUtensorMap &ta, const CUtensorMap &tr, const CUtensorMap &tb,
                           const CUtensorMap &ty, const GemmHif4Args &a, cudaStream_t st)
{
    auto kern = gemm_hif4_kernel<CONV, RES, PHI, OUT>;
    constexpr size_t smem = smem_bytes<CONV>();
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess)
        return e;
    const int64_t tiles = ((a.N + BN - 1) / BN) * ((a.M + BM - 1) / BM);
    const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
    const int phi_blocks = a.phi_r_s / BK;
    const int phi_cols = a.phi ? (int)((a.K + a.phi_r_s - 1) / a.phi_r_s) : 0;
    kern<<<grid, PHI ? THREADS + 32 : THREADS, smem, st>>>(ta, tr, tb, ty, (const uint32_t *)a.a_meta, (const uint32_t *)a.r_meta, a.phi,
                                      phi_blocks, phi_cols, a.y, (int)a.M, (int)a.N, (int)a.K, a.status);
    return cudaGetLastError();
}

template <bool CONV>
cudaError_t launch_conv(const GemmHif4Args &a, cudaStream_t st)
{
    CUtensorMap ta, tr, tb, ty;
    const uint64_t kb = CONV ? (uint64_t)a.K / 2 : (uint64_t)a.K * 2; // bytes per activation row
    const uint32_t box = CONV ? BK / 2 : BK * 2;
    const int swz = CONV ? 0 : 128;
    if (!encode_tmap_2d_u8(&ta, a.a_codes, kb, (uint64_t)a.M, kb, box, BM, swz))
        return cudaErrorInvalidValue;
    if (!encode_tmap_2d_u8(&tb, a.b_bf16, (uint64_t)a.K * 2, (uint64_t)a.N, (uint64_t)a.K * 2, BK * 2, BN, 128))
        return cudaErrorInvalidValue;
    if (a.r_codes) {
        if (!encode_tmap_2d_u8(&tr, a.r_codes, kb, (uint64_t)a.M, kb, box, BM, swz))
            return cudaErrorInvalidValue;
    } else {
        tr = ta;
    }
    const uint64_t yrow = (uint64_t)a.N * (a.out_bf16 ? 2 : 4);
    if (!encode_tmap_2d_u8(&ty, a.y, yrow, (uint64_t)a.M, yrow, 64, 32, 64))
        return cudaErrorInvalidValue;
    // Beyond REC_WORDS * 32 k-stages the record does not fit: every residual
    // product is then issued (exact: phi = 0 residuals are zero).
    const bool res = a.r_codes != nullptr;
    const bool phi = res && a.phi != nullptr && a.K / BK <= REC_WORDS * 32;
#define RFQ_GV(R, P, O) return launch_variant<CONV, R, P, O>(ta, tr, tb, ty, a, st)
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

} // namespace

cudaError_t launch_gemm_hif4(const GemmHif4Args &a, cudaStream_t st)
{
    return a.a_bf16 ? launch_conv<false>(a, st) : launch_conv<true>(a, st);
}

} // namespace rfq
