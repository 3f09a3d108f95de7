// gemm_mxf4.cu -- RFQ GEMM on the sm_103a tensor cores (Algorithm 1,
// Eq. rfq):  Y = X~ W~ + phi X^ W~.
//
// Persistent kernel: one CTA per SM walks output tiles of 128 x 256 (of
// one matrix, or of G row groups each with its own W~: the grouped form).  Per
// 256-element k-stage the TMA producer stages the main A tile (X~ codes), the
// residual A tile (X^ codes), the W~ tile (128-byte rows, 128-byte swizzle)
// and their E8M0 scale atoms (bulk copies) in shared memory, three 68 KB
// stages in flight.  Four scale-writer warps (one per TMEM lane quarter) move
// each stage's scale words from shared memory into a ring of four TMEM scale
// slots with tcgen05.st (a scale copy issued by the MMA thread would wait for
// its earlier MMAs).  With four slots and three stages, a slot is rewritten
// only after its previous stage's MMAs completed: the writers wait for the
// stage's scale copies (issued ahead of its operand tiles, on a barrier of
// their own, so that the scale words reach TMEM while the tiles still land),
// which the producer issued after those MMAs released the shared-memory
// stage.  The MMA
// thread issues, per K=64 step, the main MMA and the residual MMA against the
// SAME shared-memory W~ tile into the SAME TMEM accumulator: W~ is read once
// for both products and the correction costs only MMA issue (the on-the-fly
// residual accumulation of Sec. 4.3).  Residual MMAs of k-chunks with
// phi = 0 are not issued and their A tiles are not loaded.  With selective
// phi an extra warp writes one record per output tile (a bit per 256-element
// k-stage, set when either chunk's phi is 1, and their count; a global load
// issued by the producer would wait behind the stage copies in flight); the
// producer issues the residual stages first and publishes the count with
// every stage, so the MMA thread and the scale writers run loops with
// compile-time residual masks (a branch on a per-stage mask in the MMA
// thread slows its MMA issue; the sum over k does not depend on its order;
// a phi = 0 chunk beside a phi = 1 one adds exact zeros).  Eight epilogue
// warps drain the fp32 accumulator; with bf16 Y each warp first loads and
// packs all 128 of its columns, hands the accumulator back to the MMA thread,
// then stages and stores them (shared memory + TMA stores), so the next
// tile's MMAs start after the loads only.
//
// Scale layout in TMEM (per 128-element k-chunk): 4 columns per 128 rows,
// column j of lane i (of every lane quarter) holding the four scales of row
// 32 j + i, i.e. lane i of a quarter takes bytes [16 i, 16 i + 16) of the
// 512-byte MMA-layout atom.  A slot holds one stage: A chunk c at 4c, R at
// 8 + 4c, W~ rows 0-127 at 16 + 8c and rows 128-255 at 20 + 8c.
//
// Every mbarrier wait is bounded (kWaitLimitNs, or the limit in the caller's
// workspace) and also gives up as soon as any CTA has recorded a timeout in
// the caller's status word; the CTA then drains its in-flight copies and MMAs
// (bounded), frees TMEM and returns.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"
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
constexpr int SF_SLOT_COLS = 32;
constexpr int SF_SLOTS = 4;
constexpr int EPI_WARPS = 8;
constexpr int SF_WARPS = 4;
constexpr int THREADS = 64 + 32 * EPI_WARPS + 32 * SF_WARPS;
constexpr int PHI_WARP = THREADS / 32;  // the phi reader: one warp beyond THREADS
constexpr int REC_WORDS = 64;           // phi record: up to 2048 full k-stages (K <= 524288)
constexpr int GRP_MAX = 128;            // groups of the grouped GEMM
static_assert(SF_COL0 + SF_SLOTS * SF_SLOT_COLS <= TMEM_COLS, "TMEM budget");
static_assert(SF_SLOTS >= STAGES, "a scale slot is rewritten only after its stage's MMAs completed");

struct alignas(1024) Stage {
    uint8_t a[A_BYTES];
    uint8_t r[A_BYTES];
    uint8_t b[B_BYTES];
    uint8_t sfa[2 * ATOM];             // chunk c at c * ATOM
    uint8_t sfr[2 * ATOM];
    uint8_t sfb[4 * ATOM];             // W~ rows 128 h..128 h + 127: chunk c at (2 h + c) * ATOM
};

constexpr int YSTAGE = 2048;          // per epilogue warp: 32 rows x 64 bytes of Y

// Selective phi, one output tile: bit ks of bits (ks < K / 256, the full
// k-stages) set when phi is 1 for either 128-element chunk of stage ks;
// info = the number of set bits | (phi of the odd last chunk, when K / 128
// is odd) << 31.
struct PhiRec {
    uint32_t bits[REC_WORDS];
    uint32_t info;
};

struct Smem {
    Stage st[STAGES];
    alignas(1024) uint8_t ystage[EPI_WARPS * YSTAGE]; // 64B-swizzled staging for the TMA stores of Y
    uint64_t full[STAGES];            // a stage's operand tiles landed
    uint64_t sf_full[STAGES];         // a stage's scale atoms landed (issued first, awaited apart)
    uint64_t empty[STAGES];
    uint64_t acc_full;
    uint64_t acc_empty;
    uint64_t drain;
    uint64_t sf_ready[SF_SLOTS];      // the scale writers filled the slot
    uint64_t phi_full[2];             // the phi reader filled the record
    uint64_t phi_empty[2];            // the producer consumed the record
    PhiRec rec[2];
    uint32_t stage_info[STAGES];      // the tile's info (PhiRec::info), published with each stage
    uint32_t tmem_base;
    uint64_t wait_ns;             // limit of the bounded waits (workspace word 1, else wl)
    int32_t abort_flag;
    int32_t issued;
    int32_t grp_off[GRP_MAX + 1];     // grouped GEMM: first row of each group (and the end)
    int32_t grp_tiles[GRP_MAX + 1];   // grouped GEMM: 128-row tiles of the groups before each group
    int32_t grp_bad;
};

constexpr size_t kSmemBytes = sizeof(Smem) + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

__device__ __forceinline__ void flag_timeout(Smem &S, int32_t *status)
{
    S.abort_flag = 1;
    atomicExch(status, kDevTimeout);
}

template <bool B>
struct Bool {
    static constexpr bool value = B;
};
template <uint32_t V>
struct Mask {
    static constexpr uint32_t value = V;
};

// An output tile: its first A row, the end of its rows' group (M without
// groups), its first W~ row, its first Y column and the end of its group's
// W~ scale atoms.
struct TileCoord {
    int a_row0, row_end, w_row0, col0, wa_end;
};

// GRP: the grouped (mixture-of-experts) form: G groups of rows with their own
// W~ (row offsets read on the device), tiles of 128 rows inside each group;
// the plain form is compiled without any of it.
template <bool RES, bool PHI, bool OUT_BF16, bool GRP>
__global__ void __launch_bounds__(PHI ? THREADS + 32 : THREADS, 1)
    gemm_mxf4_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmR,
                     const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmY,
                     const uint8_t *__restrict__ sfa, const uint8_t *__restrict__ sfr,
                     const uint8_t *__restrict__ sfb, const uint8_t *__restrict__ phi, int phi_chunks,
                     int phi_cols, int M, int N, int K, int32_t *status, const int32_t *__restrict__ group_off,
                     int G, void *__restrict__ y)
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
    const int nf = kc >> 1;                // stages with two chunks
    const int n_tiles = (N + BN - 1) / BN;
    const int m_tiles = (M + BM - 1) / BM;
    const int n_atoms = (N + 127) >> 7;    // 128-row scale atoms of W~ (one group's with G > 0)

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.sf_full[s], 1);
            mbar_init(&S.empty[s], 1);
        }
        mbar_init(&S.acc_full, 1);
        mbar_init(&S.acc_empty, EPI_WARPS);
        mbar_init(&S.drain, 1);
        for (int i = 0; i < SF_SLOTS; ++i)
            mbar_init(&S.sf_ready[i], SF_WARPS);
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
        prefetch_tmap(&tmY);
    }
    if (warp == 1) {
        tmem_alloc(&S.tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    if (GRP && warp == 2) {
        // Grouped GEMM: rows [group_off[g], group_off[g+1]) of X and Y belong
        // to group g, whose W~ rows are [g N, (g+1) N).  Every group start
        // must be a multiple of 128 with the offsets non-decreasing and
        // group_off[G] <= M; otherwise the kernel records kDevBadGroups and
        // computes nothing.  The prefix of 128-row tiles maps a tile index
        // to its group.
        int bad = 0;
        for (int e = lane; e <= G; e += 32)
            S.grp_off[e] = __ldg(group_off + e);
        __syncwarp();
        int carry = 0;
        if (lane == 0)
            S.grp_tiles[0] = 0;
        for (int base = 0; base < G; base += 32) {
            const int e = base + lane;
            int cnt = 0;
            if (e < G) {
                const int a = S.grp_off[e], b = S.grp_off[e + 1];
                if (a < 0 || (a & (BM - 1)) != 0 || b < a || b > M)
                    bad = 1;
                else
                    cnt = (b - a + BM - 1) / BM;
            }
            int v = cnt;
#pragma unroll
            for (int d = 1; d < 32; d <<= 1) {
                const int t = __shfl_up_sync(0xffffffffu, v, d);
                if (lane >= d)
                    v += t;
            }
            if (e < G)
                S.grp_tiles[e + 1] = carry + v;
            carry += __shfl_sync(0xffffffffu, v, 31);
        }
        bad = __any_sync(0xffffffffu, bad);
        if (bad && lane == 0)
            atomicExch(status, kDevBadGroups);
        if (lane == 0)
            S.grp_bad = bad;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    // bad group offsets: no tile (every role skips straight to the teardown)
    const int tiles = n_tiles * (GRP ? (S.grp_bad ? 0 : S.grp_tiles[G]) : m_tiles);
    auto coord = [&](int tile) {
        const int mi = tile / n_tiles, nt = tile - mi * n_tiles;
        TileCoord c;
        c.col0 = nt * BN;
        if (!GRP) {
            c.a_row0 = mi * BM;
            c.row_end = M;
            c.w_row0 = nt * BN;
            c.wa_end = n_atoms;
        } else {
            int lo = 0, hi = G; // grp_tiles[lo] <= mi < grp_tiles[hi]
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (S.grp_tiles[mid] <= mi)
                    lo = mid;
                else
                    hi = mid;
            }
            c.a_row0 = S.grp_off[lo] + (mi - S.grp_tiles[lo]) * BM;
            c.row_end = S.grp_off[lo + 1];
            c.w_row0 = lo * N + nt * BN;
            c.wa_end = (lo + 1) * n_atoms;
        }
        return c;
    };

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            int p = 0, it = 0; // p: stages issued so far (ring position)
            bool stop = false;
            if (!held_start_wait(status, wl)) { // a test-held start never opened
                flag_timeout(S, status);
                stop = true;
            }
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x, ++it) {
                const TileCoord tc = coord(tile);
                const int m_tile = tc.a_row0 / BM;    // scale atoms and A rows
                const int atom0 = tc.w_row0 >> 7;
                const int nb = atom0 + 1 < tc.wa_end ? 2 : 1;
                // one k-stage: wait for its ring slot, publish the tile's info,
                // issue the copies
                auto produce = [&](int ks, int nch, uint32_t info, auto res_t) {
                    constexpr bool res_on = decltype(res_t)::value;
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    const int c0 = 2 * ks;
                    if (PHI)
                        S.stage_info[slot] = info;
                    const uint32_t sfbytes = (uint32_t)nch * ATOM;
                    Stage &st = S.st[slot];
                    // the scale atoms first, on their own barrier: the scale
                    // writers move them into TMEM while the operand tiles land
                    uint64_t *sbar = &S.sf_full[slot];
                    mbar_arrive_expect_tx(sbar, (1 + nb) * sfbytes + (res_on ? sfbytes : 0));
                    bulk_load(st.sfa, sfa + ((int64_t)m_tile * kc + c0) * ATOM, sfbytes, sbar);
                    if (res_on)
                        bulk_load(st.sfr, sfr + ((int64_t)m_tile * kc + c0) * ATOM, sfbytes, sbar);
                    for (int h = 0; h < nb; ++h)
                        bulk_load(st.sfb + h * 2 * ATOM, sfb + ((int64_t)(atom0 + h) * kc + c0) * ATOM, sfbytes, sbar);
                    uint64_t *bar = &S.full[slot];
                    mbar_arrive_expect_tx(bar, A_BYTES + B_BYTES + (res_on ? A_BYTES : 0));
                    tma_load_2d(st.a, &tmA, bar, c0 * 64, tc.a_row0);
                    if (res_on)
                        tma_load_2d(st.r, &tmR, bar, c0 * 64, tc.a_row0);
                    tma_load_2d(st.b, &tmB, bar, c0 * 64, tc.w_row0);
                    ++p;
                };
                if constexpr (!PHI) {
                    // full stages, then an odd last chunk (chunk counts known at compile time)
                    for (int ks = 0; ks < nf && !stop; ++ks)
                        produce(ks, 2, 0u, Bool<RES>{});
                    if (nf < nks && !stop)
                        produce(nf, 1, 0u, Bool<RES>{});
                } else {
                    const int r = it & 1;
                    if (!mbar_wait(&S.phi_full[r], (it >> 1) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        break;
                    }
                    const PhiRec &rec = S.rec[r];
                    const uint32_t info = rec.info;
                    // stages with a residual, then the others, each in k order
                    for (int w = 0; 32 * w < nf && !stop; ++w) {
                        uint32_t x = rec.bits[w];
                        while (x != 0 && !stop) {
                            const int b = __ffs(x) - 1;
                            x &= x - 1;
                            produce(32 * w + b, 2, info, Bool<true>{});
                        }
                    }
                    for (int w = 0; 32 * w < nf && !stop; ++w) {
                        const int left = nf - 32 * w;
                        uint32_t x = ~rec.bits[w] & (left >= 32 ? 0xffffffffu : (1u << left) - 1u);
                        while (x != 0 && !stop) {
                            const int b = __ffs(x) - 1;
                            x &= x - 1;
                            produce(32 * w + b, 2, info, Bool<false>{});
                        }
                    }
                    if (nf < nks && !stop) {   // the odd last chunk
                        if (info >> 31)
                            produce(nf, 1, info, Bool<true>{});
                        else
                            produce(nf, 1, info, Bool<false>{});
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
            for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x, ++it) {
                if (!mbar_wait(&S.acc_empty, (it & 1) ^ 1, wl, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                tc_fence_after();
                // the MMAs of the stage at position pos of the tile, with residual
                // mask rm (bit c: chunk c's residual product) known at compile time
                auto mma_stage = [&](int pos, int nch, auto rm_t) {
                    constexpr uint32_t rm = decltype(rm_t)::value;
                    const int slot = p % STAGES, sfs = p % SF_SLOTS;
                    if (!mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat) ||
                        !mbar_wait(&S.sf_ready[sfs], (p / SF_SLOTS) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    tc_fence_after();
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
                        tc_mma_mxf4(tmem, sdesc_k_sw128(a0 + 32 * j), bd, id, sf + 4 * c, sfb_t, (pos | j) != 0);
                        if ((rm >> c) & 1)
                            tc_mma_mxf4(tmem, sdesc_k_sw128(r0 + 32 * j), bd, id, sf + 8 + 4 * c, sfb_t, 1);
                    }
                    tc_commit(&S.empty[slot]);
                    ++p;
                };
                if constexpr (!PHI) {
                    for (int ks = 0; ks < nf && !stop; ++ks)
                        mma_stage(ks, 2, Mask<RES ? 3u : 0u>{});
                    if (nf < nks && !stop)
                        mma_stage(nf, 1, Mask<RES ? 1u : 0u>{});
                } else {
                    // the tile's residual-stage count arrives with its first stage
                    if (!mbar_wait(&S.full[p % STAGES], (p / STAGES) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        break;
                    }
                    const uint32_t info = S.stage_info[p % STAGES];
                    const int n_res = (int)(info & 0x7fffffffu);
                    int pos = 0;
                    for (; pos < n_res && !stop; ++pos)
                        mma_stage(pos, 2, Mask<3u>{});
                    for (; pos < nf && !stop; ++pos)
                        mma_stage(pos, 2, Mask<0u>{});
                    if (nf < nks && !stop) {
                        if (info >> 31)
                            mma_stage(pos, 1, Mask<1u>{});
                        else
                            mma_stage(pos, 1, Mask<0u>{});
                    }
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
            // warp-uniform outcome: the tcgen05 loads below need the whole warp
            if (!__all_sync(0xffffffffu, mbar_wait(&S.acc_full, it & 1, wl, gstat))) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            tc_fence_after();
            const TileCoord tc = coord(tile);
            const int row0 = tc.a_row0 + q * 32;
            const uint32_t tcol = tmem + ((uint32_t)(q * 32) << 16) + h * (BN / 2);
            if (OUT_BF16) {
                // all 128 columns of this warp into registers as packed bf16,
                // then the accumulator goes back to the MMA thread
                uint32_t pk[64];
                {
                    // all four 32-column loads in flight, one wait
                    uint32_t v[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        tmem_ld_32x32b_x32(tcol + 32 * c, v[c]);
                    tmem_ld_wait();
#pragma unroll
                    for (int c = 0; c < 4; ++c)
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(v[c][2 * i]),
                                                                      __uint_as_float(v[c][2 * i + 1]));
                            pk[16 * c + i] = *reinterpret_cast<uint32_t *>(&b2);
                        }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&S.acc_empty);
#pragma unroll
                for (int c = 0; c < 4; ++c) {   // 32-column chunks: one 64-byte TMA box row per lane
                    const int col = tc.col0 + h * (BN / 2) + 32 * c;
                    if (col >= N || row0 >= tc.row_end)
                        break;
                    if (GRP && row0 + 32 > tc.row_end && tc.row_end < M) {
                        // a group ends inside this 32-row box: rows past it are
                        // another group's or padding, so each lane stores its own row
                        if (row0 + lane < tc.row_end) {
                            uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(y) +
                                                                   (int64_t)(row0 + lane) * N + col);
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                dst[j] = make_uint4(pk[16 * c + 4 * j], pk[16 * c + 4 * j + 1],
                                                    pk[16 * c + 4 * j + 2], pk[16 * c + 4 * j + 3]);
                        }
                        continue;
                    }
                    if (lane == 0)
                        bulk_wait_group_read<0>();
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 4; ++j)
                        *reinterpret_cast<uint4 *>(stg + lane * 64 + ((j ^ sw) << 4)) =
                            make_uint4(pk[16 * c + 4 * j], pk[16 * c + 4 * j + 1], pk[16 * c + 4 * j + 2],
                                       pk[16 * c + 4 * j + 3]);
                    fence_proxy_async_smem();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_2d(&tmY, stg, col * 2, row0);
                        bulk_commit_group();
                    }
                }
            } else {
#pragma unroll
                for (int half = 0; half < 2; ++half) {
                    // two 32-column chunks in flight; the accumulator goes back
                    // to the MMA thread after the last load of the tile
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
                        const int col = tc.col0 + h * (BN / 2) + (2 * half + c) * 32;
                        if (col >= N || row0 >= tc.row_end)
                            continue;
#pragma unroll
                        for (int hb = 0; hb < 2; ++hb) { // 16 fp32 columns (64 bytes) per store
                            if (col + 16 * hb >= N)
                                break;
                            if (GRP && row0 + 32 > tc.row_end && tc.row_end < M) {
                                // a group ends inside this 32-row box (see the bf16 path)
                                if (row0 + lane < tc.row_end) {
                                    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<float *>(y) +
                                                                           (int64_t)(row0 + lane) * N + col + 16 * hb);
#pragma unroll
                                    for (int j = 0; j < 4; ++j)
                                        dst[j] = make_uint4(v[c][16 * hb + 4 * j], v[c][16 * hb + 4 * j + 1],
                                                            v[c][16 * hb + 4 * j + 2], v[c][16 * hb + 4 * j + 3]);
                                }
                                continue;
                            }
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
    } else if (warp < PHI_WARP) {
        // ------------------------------------------------ scale writers (warps 10..13)
        // Warp quarter q writes TMEM lanes 32q..32q+31; every quarter holds
        // the same scale words (the MMA reads row 32 j + i from column j of
        // lane i of the quarter that computes it).
        const int q = warp & 3;
        int p = 0;
        bool stop = false;
        for (int tile = blockIdx.x; tile < tiles && !stop; tile += gridDim.x) {
            // the tile's second W~ scale atom exists (else zeros: its W~ rows
            // are past N, or another group's)
            const TileCoord tc = coord(tile);
            const bool b1_in = (tc.w_row0 >> 7) + 1 < tc.wa_end;
            // the scale words of the next stage (in the producer's order), with
            // the residual mask rm known at compile time
            auto write_stage = [&](int nch, auto rm_t) {
                constexpr uint32_t rm = decltype(rm_t)::value;
                const int slot = p % STAGES, sfs = p % SF_SLOTS;
                // warp-uniform outcome: the tcgen05 stores below need the whole warp
                if (!__all_sync(0xffffffffu, mbar_wait(&S.sf_full[slot], (p / STAGES) & 1, wl, gstat))) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    stop = true;
                    return;
                }
                tc_fence_after();
                const Stage &st = S.st[slot];
                const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + SF_COL0 + SF_SLOT_COLS * sfs;
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    if (c >= nch)
                        break;
                    const uint4 va = *reinterpret_cast<const uint4 *>(st.sfa + c * ATOM + lane * 16);
                    const uint4 vb0 = *reinterpret_cast<const uint4 *>(st.sfb + c * ATOM + lane * 16);
                    const uint4 vb1 = b1_in ? *reinterpret_cast<const uint4 *>(st.sfb + (2 + c) * ATOM + lane * 16)
                                            : make_uint4(0, 0, 0, 0);
                    tmem_st_32x32b_x4(tb + 4 * c, va.x, va.y, va.z, va.w);
                    if ((rm >> c) & 1) {
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
                ++p;
            };
            if constexpr (!PHI) {
                for (int ks = 0; ks < nf && !stop; ++ks)
                    write_stage(2, Mask<RES ? 3u : 0u>{});
                if (nf < nks && !stop)
                    write_stage(1, Mask<RES ? 1u : 0u>{});
            } else {
                // the tile's residual-stage count arrives with its first stage
                if (!__all_sync(0xffffffffu, mbar_wait(&S.sf_full[p % STAGES], (p / STAGES) & 1, wl, gstat))) {
                    if (lane == 0)
                        flag_timeout(S, status);
                    break;
                }
                const uint32_t info = S.stage_info[p % STAGES];
                const int n_res = (int)(info & 0x7fffffffu);
                int pos = 0;
                for (; pos < n_res && !stop; ++pos)
                    write_stage(2, Mask<3u>{});
                for (; pos < nf && !stop; ++pos)
                    write_stage(2, Mask<0u>{});
                if (nf < nks && !stop) {
                    if (info >> 31)
                        write_stage(1, Mask<1u>{});
                    else
                        write_stage(1, Mask<0u>{});
                }
            }
        }
    } else if (PHI) {
        // ------------------------------------------------ phi reader (warp 14)
        // Record of the CTA's j-th tile: chunk c of row tile m needs its
        // residual when phi[m][c / phi_chunks] is non-zero.
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
            const uint8_t *row = phi + (int64_t)(coord((int)blockIdx.x + j * (int)gridDim.x).a_row0 / BM) * phi_cols;
            PhiRec &rec = S.rec[r];
            uint32_t n_res = 0;
            for (int w = 0; 32 * w < nf; ++w) {
                const int ks = 32 * w + lane;
                const bool on = ks < nf && (__ldg(row + (2 * ks) / phi_chunks) != 0 ||
                                            __ldg(row + (2 * ks + 1) / phi_chunks) != 0);
                const uint32_t word = __ballot_sync(0xffffffffu, on);
                if (lane == 0)
                    rec.bits[w] = word;
                n_res += __popc(word);
            }
            const uint32_t tail = nf < nks && __ldg(row + (2 * nf) / phi_chunks) != 0 ? 1u : 0u;
            if (lane == 0)
                rec.info = n_res | tail << 31;
            mbar_arrive(&S.phi_full[r]);
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (threadIdx.x == 0 && S.abort_flag) {
        // wait (bounded) for the copies of the last stages still in flight
        const int issued = S.issued;
        for (int p = max(0, issued - STAGES); p < issued; ++p) {
            (void)mbar_wait(&S.full[p % STAGES], (p / STAGES) & 1, wl);
            (void)mbar_wait(&S.sf_full[p % STAGES], (p / STAGES) & 1, wl);
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, TMEM_COLS);
    }
}

template <bool RES, bool PHI, bool OUT, bool GRP>
cudaError_t launch_variant(const CUtensorMap &ta, const CUtensorMap &tr, const CUtensorMap &tb,
                           const CUtensorMap &ty, const GemmMxf4Args &a, cudaStream_t st)
{
    auto kern = gemm_mxf4_kernel<RES, PHI, OUT, GRP>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    // grouped: the tile count depends on the device-side row offsets; every
    // CTA of the grid walks the tiles that exist
    const int64_t tiles = GRP ? INT64_MAX : ((a.N + BN - 1) / BN) * ((a.M + BM - 1) / BM);
    const int grid = (int)(tiles < num_sms() ? tiles : num_sms());
    const int phi_chunks = a.phi_r_s / 128;
    const int phi_cols = a.phi ? (int)((a.K + a.phi_r_s - 1) / a.phi_r_s) : 0;
    kern<<<grid, PHI ? THREADS + 32 : THREADS, kSmemBytes, st>>>(
        ta, tr, tb, ty, (const uint8_t *)a.a_sf, (const uint8_t *)a.r_sf, (const uint8_t *)a.b_sf, a.phi, phi_chunks,
        phi_cols, (int)a.M, (int)a.N, (int)a.K, a.status, a.group_off, a.groups, a.y);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_gemm_mxf4(const GemmMxf4Args &a, cudaStream_t st)
{
    // More than one 128-row tile: CTA pairs (M = 256 MMAs, half the W~ bytes
    // per SM); E4M3 operands run on the pair kernel at every M.  Grouped
    // MXFP4: 128-row tiles inside each group here while the groups average
    // fewer than 2048 stacked rows.  A group's 256-row pairs compute 64 rows
    // past its 128-row tiles on average, which for short groups costs more
    // than the pair saves (Qwen3-VL-30B experts, ~320 rows each: 0.106 ms
    // here against 0.112 ms on pairs).
    const bool grp = a.groups > 0;
    const bool grp_single = grp && !a.f8 && a.M < (int64_t)2048 * a.groups;
    if ((a.M > BM && !grp_single) || a.f8 || (grp && !grp_single))
        return launch_gemm_mxf4_pair(a, st);
    CUtensorMap ta, tr, tb;
    const uint64_t kb = (uint64_t)a.K / 2;
    const uint64_t w_rows = (uint64_t)a.N * (grp ? (uint64_t)a.groups : 1u);
    if (!encode_tmap_2d_u8(&ta, a.a_codes, kb, (uint64_t)a.M, kb, ROW, BM, 128))
        return cudaErrorInvalidValue;
    if (!encode_tmap_2d_u8(&tb, a.b_codes, kb, w_rows, kb, ROW, BN, 128))
        return cudaErrorInvalidValue;
    if (a.r_codes) {
        if (!encode_tmap_2d_u8(&tr, a.r_codes, kb, (uint64_t)a.M, kb, ROW, BM, 128))
            return cudaErrorInvalidValue;
    } else {
        tr = ta;
    }
    // Y [M][N] (bf16 or fp32) as bytes; boxes of 64 bytes x 32 rows, 64B swizzle
    CUtensorMap ty;
    const uint64_t yrow = (uint64_t)a.N * (a.out_bf16 ? 2 : 4);
    if (!encode_tmap_2d_u8(&ty, a.y, yrow, (uint64_t)a.M, yrow, 64, 32, 64))
        return cudaErrorInvalidValue;
    // Beyond REC_WORDS * 32 full k-stages the record does not fit: every
    // residual product is then issued (exact: phi = 0 residuals are zero).
    const bool res = a.r_codes != nullptr;
    const bool phi = res && a.phi != nullptr && a.K / 256 <= REC_WORDS * 32;
#define RFQ_GV(R, P, O)                                                                                           \
    return grp ? launch_variant<R, P, O, true>(ta, tr, tb, ty, a, st) : launch_variant<R, P, O, false>(ta, tr, tb, ty, a, st)
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
