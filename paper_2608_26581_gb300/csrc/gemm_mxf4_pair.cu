// gemm_mxf4_pair.cu -- RFQ GEMM on CTA pairs (Algorithm 1, Eq. rfq):
//   Y = X~ W~ + phi X^ W~
// with tcgen05 cta_group::2 MMAs: the two CTAs of a cluster compute one
// 256 x 256 output tile.  Each CTA stages its own 128 rows of X~ and X^ and
// HALF of the tile's 256 W~ rows; one thread of the even CTA issues M = 256
// MMAs that read the A rows and W~ halves of both CTAs.  Per 256-element
// k-stage an SM streams 52 KB (codes and scale atoms) for 1,024 cycles of MMA
// work, 24% less than the 68 KB of a single-CTA 128 x 256 tile.
//
// Per CTA (448 threads, 480 with selective phi; one CTA per SM):
//   warp 0      TMA producer.  The codes (own A and R rows, own W~ half) are
//               CTA-pair copies that complete on the EVEN CTA's stage
//               barrier, which the even CTA's producer arms with the bytes of
//               both CTAs; the scale atoms (own A / R rows, both 128-row W~
//               atoms of the tile) are bulk copies into this CTA's shared
//               memory, on its own barrier.
//   warp 1      even CTA: MMA issuer (main + residual MMA per K=64 step,
//               same W~ descriptor, same accumulator: Sec. 4.3)
//   warps 2-9   epilogue: TMEM -> registers -> bf16 / fp32 -> shared-memory
//               staging -> TMA stores of this CTA's 128 rows
//   warps 10-13 scale writers: this CTA's scale words from shared memory into
//               its TMEM with tcgen05.st, one warp per TMEM lane quarter
//   warp 14     (selective phi only) phi reader: one record per output tile
//               of this CTA (double-buffered) with a bit per k-stage, set
//               when the stage needs its residual, and their count
// TMEM (512 columns per CTA): a 256-column accumulator (this CTA's 128 rows
// of the tile) and four 32-column scale slots; each CTA holds the scales of
// its own A / R rows and of ALL 256 W~ rows of the tile (the layout the pair
// MMA reads).  A slot is rewritten four stages after its last use, after the
// stage's copies, which the producer issued once the MMAs of that earlier
// stage had completed.
//
// Cross-CTA signals (the odd CTA's scale writers and epilogue warps telling
// the even CTA's MMA thread that a scale slot is filled or the accumulator
// drained) are relaxed arrives on the even CTA's barriers, issued after the
// signalling warp's own tcgen05 stores / loads have completed (wait::st /
// wait::ld); the MMA thread observes them with cluster-scope acquire waits
// and orders its MMAs after them with tcgen05.fence.  A release arrive at
// cluster scope would stall the arriving warp for hundreds of cycles.
//
// Selective phi: the residual loads and MMAs of a 256-element k-stage are
// skipped when phi is 0 for both of its 128-element chunks in both row tiles
// of the pair (the stored residual of a phi = 0 tile is zero, so including a
// phi = 0 chunk or row tile beside a phi = 1 one adds exact zeros).  Each
// tile's stages run in a data-dependent ORDER -- the stages with a residual
// first, then those without, each in k order, an odd last chunk last -- so
// the MMA thread and the scale writers run two loops with compile-time
// residual masks and data-dependent trip counts (the sum over k does not
// depend on its order).  A branch on a per-stage mask value in the MMA
// thread slowed its MMA issue by ~150 cycles per stage; the loop bounds cost
// nothing measurable.  Only the producer follows the order, from the bits of
// the tile's record; it publishes the tile's residual-stage count with every
// stage.  The records come from a warp of their own, a tile ahead: a global
// load issued by the producer waits behind the stage copies in flight on its
// SM (thousands of cycles).
//
// Every mbarrier wait is bounded (kWaitLimitNs, or the limit in the caller's
// workspace) and also gives up when any CTA has recorded a timeout in the
// caller's status word.  Neither CTA of a pair leaves before the final
// cluster barrier, so the peer never signals a CTA that has exited; the even
// CTA drains its MMAs before that barrier.
#include <cuda_bf16.h>
#include <cstdint>

#include "internal.h"
#include "mxfp4_math.cuh"
#include "ptx.cuh"

namespace rfq {
namespace {

RFQ_DEBUG_WORD_DECL

constexpr int BM = 128;                  // rows per CTA (256 per pair)
constexpr int BN = 256;                  // output columns per pair tile
constexpr int BN_HALF = BN / 2;          // W~ rows staged per CTA
constexpr int ROW = 128;                 // bytes of codes per row per stage (256 elements)
constexpr int STAGES = 4;
constexpr int A_BYTES = BM * ROW;
constexpr int B_BYTES = BN_HALF * ROW;
constexpr int ATOM = 512;                // scale bytes of 128 rows x one 128-element chunk
constexpr int TMEM_COLS = 512;
constexpr int SF_COL0 = BN;              // scale slots after the accumulator
constexpr int SF_SLOT_COLS = 32;         // A chunk c at 4c, R at 8 + 4c, W~ at 16 + 8c (+4: rows 128-255)
constexpr int SF_SLOTS = 4;
constexpr int EPI_WARPS = 8;
constexpr int SF_WARPS = 4;
constexpr int THREADS = 64 + 32 * (EPI_WARPS + SF_WARPS);
constexpr int PHI_WARP = THREADS / 32;   // the phi reader: one warp beyond THREADS
constexpr int REC_WORDS = 64;            // phi record: up to 2048 full k-stages (K <= 524288)
constexpr int GRP_MAX = 128;             // groups of the grouped GEMM
constexpr int YSTAGE = 2048;             // per epilogue warp: 32 rows x 64 bytes of Y
constexpr int FQ_ROWS = 8;               // fused quantizer: rows of X per conversion unit
constexpr int FQ_SUB = BM / FQ_ROWS;     // units per (128-row tile, k-stage)
constexpr int FQ_CALL = 4;               // rows quantized per step of a converting warp (loads in flight)
static_assert(FQ_ROWS % FQ_CALL == 0, "whole steps per unit");
static_assert(SF_COL0 + SF_SLOTS * SF_SLOT_COLS <= TMEM_COLS, "TMEM budget");
static_assert(SF_SLOTS >= STAGES, "a scale slot is rewritten only after its stage's MMAs completed");

struct alignas(1024) Stage {
    uint8_t a[A_BYTES];
    uint8_t r[A_BYTES];
    uint8_t b[B_BYTES];
    uint8_t sfa[2 * ATOM];               // chunk c at c * ATOM
    uint8_t sfr[2 * ATOM];
    uint8_t sfb[4 * ATOM];               // W~ rows 128 h..128 h + 127 of the tile: chunk c at (2 h + c) * ATOM
};
static_assert(sizeof(Stage) % 1024 == 0, "stages keep the 1024-byte swizzle alignment");

// Selective phi, one output tile: bit ks of bits (ks < K / 256, the full
// k-stages) set when phi is 1 for either 128-element chunk of stage ks in
// either row tile; info = the number of set bits | (phi of the odd last
// chunk, when K / 128 is odd) << 31.
struct PhiRec {
    uint32_t bits[REC_WORDS];
    uint32_t info;
};

struct Smem {
    Stage st[STAGES];
    alignas(1024) uint8_t ystage[EPI_WARPS * YSTAGE];
    uint64_t full[STAGES];        // (even CTA) both CTAs' code copies landed
    uint64_t sf_full[STAGES];     // this CTA's scale atoms landed
    uint64_t w4_full[STAGES];     // mixed rate: this CTA's packed W~ half landed
    uint64_t empty[STAGES];       // the stage's MMAs completed (both CTAs)
    uint64_t sf_ready[SF_SLOTS];  // (even CTA) both CTAs' scale writers filled the slot
    uint64_t acc_full;            // accumulator complete (both CTAs)
    uint64_t acc_empty;           // (even CTA) both CTAs' epilogue warps drained it
    uint64_t drain;
    uint64_t phi_full[2];         // the phi reader filled the record
    uint64_t phi_empty[2];        // the producer consumed the record
    PhiRec rec[2];
    uint32_t stage_info[STAGES];  // the tile's residual-stage count | odd last chunk's residual << 31
    int32_t grp_off[GRP_MAX + 1];   // grouped GEMM: first row of each group (and the end)
    int32_t grp_pairs[GRP_MAX + 1]; // grouped GEMM: 256-row pairs of the groups before each group
    int32_t grp_bad;                // grouped GEMM: the row offsets break the contract
    uint32_t tmem_base;
    int32_t fq_last;              // fused quantizer: this CTA is the grid's last to finish
    uint64_t wait_ns;             // limit of the bounded waits (workspace word 1, else wl)
    int32_t abort_flag;
};
constexpr size_t kSmemBytes = sizeof(Smem) + 1024;
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");

// Fused quantizer (FQ): the activation quantizer of Sec. 4.3 (X~ = Q(X), the
// residual dX = X - X~ and X^ = Q(dX), per 32-element block along K) runs
// inside the GEMM.  X is cut into units of FQ_ROWS rows x one k-stage (256
// columns, or the odd last 128); the epilogue warps, between draining
// accumulators, take units in order from a global counter, quantize them
// into a scratch copy of the codes and MMA-layout scales (the layout the
// quantizer kernel writes), and count each finished unit for its (128-row
// tile, k-stage).  The producer issues a stage's A / R copies once that
// count is complete.  Every element of X is quantized once, however many
// output tiles read it.  The scratch is a ring of `ring` slots of 256 rows:
// the rows of 256-row block p live in slot p % ring, and a converter fills
// block p only once every output tile of block p - ring has loaded its
// operands (counted by the MMA thread after the tile's last stage), so the
// scratch stays in L2 (the tile walk is row-block major).  A converter never
// blocks on a slot: it keeps its unit and goes back to its accumulator
// wait.  The grid's last CTA to finish zeroes the counters for the next call.
struct FqArgs {
    const uint4 *x;               // bf16 X [M][K], 8 elements per uint4
    uint32_t *mcodes, *rcodes;    // scratch codes [ring * 256][K/8] words (X~, X^)
    uint8_t *msf, *rsf;           // scratch scales, MMA layout, [ring * 256] rows
    int32_t *ctr;                 // [0] next unit, [1] CTAs finished, [2, 2 + m_tiles) units done per
                                  // 128-row tile, then [m_tiles][k-stages] units done per (tile, stage),
                                  // then [m_pairs] output tiles that finished loading each 256-row block
    int ring;                     // slots of 256 rows in the scratch
};

__device__ __forceinline__ void flag_timeout(Smem &S, int32_t *status)
{
    S.abort_flag = 1;
    atomicExch(status, kDevTimeout);
}

// Where an output tile lives: the pair's first A row, the end of its rows
// (the group's end, or M), its first W~ row and Y column, and the end of
// its group's 128-row W~ scale atoms.
struct TileCoord {
    int a_row0, row_end, w_row0, col0, wa_end;
};

template <bool B>
struct Bool {
    static constexpr bool value = B;
};
template <uint32_t V>
struct Mask {
    static constexpr uint32_t value = V;
};

// F8 (operand form): 0 -- every operand E2M1 (kind::mxf4); 1 -- every
// operand holds E4M3 codes (one byte per element, kind::mxf8f6f4 MMAs of
// K = 32 with one scale per row each), a stage is then one 128-element chunk
// (the same 128-byte rows); 2 -- the FP4-to-FP8 residual at two rates
// (Sec. 4.2, 4.3): a stage is one 128-element chunk holding X~ and W~ packed
// (E2M1, 64-byte rows, 64-byte swizzle: the main product on kind::mxf4, two
// K = 64 MMAs), X^ as E4M3 and W~ again in the padded 4-bit form (128-byte
// rows: the residual product on kind::mxf8f6f4, E4M3 x E2M1, four K = 32
// MMAs), into the same accumulator with the same scale words.  The scale
// writers expand the packed W~ tile into the padded one in shared memory,
// so a stage reads 32 KB from L2 for 768 MMA cycles (1,024 when the main
// product also runs on kind::mxf8f6f4).
constexpr int F8_MIXED = 2;
// F8 == F8_W4: the E4M3 form with W~ kept as MXFP4 -- every product on
// kind::mxf8f6f4 as E4M3 x E2M1, W~'s tile copied from its packed codes in
// the padded 4-bit form (64 bytes read per 128-byte row).
constexpr int F8_W4 = 3;
// GRP: the grouped (mixture-of-experts) form, G groups of rows with their
// own W~ (row offsets read on the device); the plain form is compiled
// without any of it.
// FQ: the fused quantizer above (MXFP4 operands, no phi records, no groups).
// PROF: the MMA thread of each even CTA counts its SM clock cycles and
// wall-clock nanoseconds from its first wait to its drain, the cycles it
// waits for a drained accumulator, for a stage's copies and for a stage's
// scale words, and its stages and tiles, and adds them to the 64-bit
// workspace words 4..11 (a measurement of where the tensor pipe idles).
template <bool RES, bool PHI, bool OUT_BF16, int F8, bool GRP, bool FQ = false, bool PROF = false>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(PHI ? THREADS + 32 : THREADS, 1)
    gemm_mxf4_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmR,
                          const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmY,
                          const __grid_constant__ CUtensorMap tmB4,
                          const uint8_t *__restrict__ sfa, const uint8_t *__restrict__ sfr,
                          const uint8_t *__restrict__ sfb, const uint8_t *__restrict__ phi, int phi_chunks,
                          int phi_cols, int M, int N, int K, int32_t *status,
                          const int32_t *__restrict__ group_off, int G, void *__restrict__ y, const FqArgs fq)
{
    static_assert(!FQ || (!PHI && !F8 && !GRP), "the fused quantizer takes plain MXFP4 operands");
    static_assert(F8 != F8_MIXED || (RES && !GRP && !FQ), "the mixed-rate form is the RFQ with a residual");
    constexpr int B_TX = F8 == F8_W4 ? B_BYTES / 2 : B_BYTES;   // bytes a W~ tile copy reads
    extern __shared__ uint8_t smem_raw[];
    Smem &S = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool lead = rank == 0;
    const volatile int32_t *gstat = status;

    const int kc = K >> 7;                  // 128-element chunks
    constexpr int CPS = F8 ? 1 : 2;        // 128-element chunks per stage (128-byte rows either way)
    const int nks = (kc + CPS - 1) / CPS;   // stages (with MXFP4 the last may hold one chunk)
    const int nf = kc / CPS;                // stages with CPS chunks
    const int n_tiles = (N + BN - 1) / BN;
    const int m_tiles = (M + BM - 1) / BM;  // 128-row tiles: scale atoms and phi rows
    const int m_pairs = (M + 2 * BM - 1) / (2 * BM);
    const int n_atoms = (N + 127) >> 7;     // 128-row scale atoms of W~ (one group's with G > 0)
    const int pair = blockIdx.x >> 1, pairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&S.full[s], 1);
            mbar_init(&S.sf_full[s], 1);
            mbar_init(&S.w4_full[s], 1);
            mbar_init(&S.empty[s], 1);
        }
        for (int i = 0; i < SF_SLOTS; ++i)
            mbar_init(&S.sf_ready[i], 2 * SF_WARPS);
        mbar_init(&S.acc_full, 1);
        mbar_init(&S.acc_empty, 2 * EPI_WARPS);
        mbar_init(&S.drain, 1);
        for (int i = 0; i < 2; ++i) {
            mbar_init(&S.phi_full[i], 32);
            mbar_init(&S.phi_empty[i], 1);
        }
        // A bounded wait of an earlier CTA or call gave up: skip the work
        // (both CTAs still meet at the cluster barriers).
        S.abort_flag = *gstat;
        S.wait_ns = ws_wait_limit_ns(status);
        fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tmap(&tmA);
        if (RES)
            prefetch_tmap(&tmR);
        prefetch_tmap(&tmB);
        prefetch_tmap(&tmY);
        if (F8 == F8_MIXED)
            prefetch_tmap(&tmB4);
    }
    if (warp == 1) {
        tmem_alloc_pair(&S.tmem_base, TMEM_COLS);
        tmem_relinquish_pair();
    }
    if (GRP && warp == 2) {
        // Grouped GEMM (G > 0): rows [group_off[g], group_off[g+1]) of X and Y
        // belong to group g, whose W~ rows are [g N, (g+1) N).  Every group
        // start must be a multiple of 128 with the offsets non-decreasing and
        // group_off[G] <= M; otherwise the kernel records kDevBadGroups and
        // computes nothing.  The prefix of 256-row pairs maps a tile index to
        // its group.
        int bad = 0;
        if (G > 0) {
            for (int e = lane; e <= G; e += 32)
                S.grp_off[e] = __ldg(group_off + e);
            __syncwarp();
            int carry = 0;
            if (lane == 0)
                S.grp_pairs[0] = 0;
            for (int base = 0; base < G; base += 32) {
                const int e = base + lane;
                int cnt = 0;
                if (e < G) {
                    const int a = S.grp_off[e], b = S.grp_off[e + 1];
                    if (a < 0 || (a & (BM - 1)) != 0 || b < a || b > M)
                        bad = 1;
                    else
                        cnt = (b - a + 2 * BM - 1) / (2 * BM);
                }
                int v = cnt;
#pragma unroll
                for (int d = 1; d < 32; d <<= 1) {
                    const int t = __shfl_up_sync(0xffffffffu, v, d);
                    if (lane >= d)
                        v += t;
                }
                if (e < G)
                    S.grp_pairs[e + 1] = carry + v;
                carry += __shfl_sync(0xffffffffu, v, 31);
            }
            bad = __any_sync(0xffffffffu, bad);
            if (bad && lane == 0)
                atomicExch(status, kDevBadGroups);
        }
        if (lane == 0)
            S.grp_bad = bad;
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync(); // both CTAs' barriers initialised and TMEM allocated
    tc_fence_after();
    const uint32_t tmem = S.tmem_base;
    const bool skip = S.abort_flag != 0 || (GRP && S.grp_bad != 0);
    const uint64_t wl = S.wait_ns;
    const int tiles = n_tiles * (GRP ? S.grp_pairs[G] : m_pairs);
    auto coord = [&](int tile) {
        const int pi = tile / n_tiles, nt = tile - pi * n_tiles;
        TileCoord c;
        c.col0 = nt * BN;
        if (!GRP) {
            c.a_row0 = pi * 2 * BM;
            c.row_end = M;
            c.w_row0 = nt * BN;
            c.wa_end = n_atoms;
        } else {
            int lo = 0, hi = G; // grp_pairs[lo] <= pi < grp_pairs[hi]
            while (hi - lo > 1) {
                const int mid = (lo + hi) >> 1;
                if (S.grp_pairs[mid] <= pi)
                    lo = mid;
                else
                    hi = mid;
            }
            c.a_row0 = S.grp_off[lo] + (pi - S.grp_pairs[lo]) * 2 * BM;
            c.row_end = S.grp_off[lo + 1];
            c.w_row0 = lo * N + nt * BN;
            c.wa_end = (lo + 1) * n_atoms;
        }
        return c;
    };

    if (warp == 0) {
        // ------------------------------------------------ TMA producer (both CTAs)
        if (lane == 0 && !skip) {
            const uint32_t full0 = mapa_shared(smem_u32(&S.full[0]), 0);   // the even CTA's barriers
            int p = 0, it = 0;
            bool stop = false;
            int fq_tile_ok = -1;   // FQ: a 128-row tile whose every unit is quantized
            if (!held_start_wait(status, wl)) { // a test-held start never opened
                flag_timeout(S, status);
                stop = true;
            }
            for (int tile = pair; tile < tiles && !stop; tile += pairs, ++it) {
                const TileCoord tc = coord(tile);
                const int a_row = tc.a_row0 + (int)rank * BM;   // this CTA's first A row
                const int m_tile = a_row / BM;
                const bool rows_in = a_row < tc.row_end;
                // FQ: the ring slot holding these rows (rows past M: a box past the ring, zero fill)
                const int fq_slot = FQ ? (tc.a_row0 >> 8) % fq.ring : 0;
                const int a_y = !FQ ? a_row : rows_in ? fq_slot * 2 * BM + (int)rank * BM : fq.ring * 2 * BM;
                const int sf_tile = FQ ? fq_slot * 2 + (int)rank : m_tile;
                const int atom0 = tc.w_row0 >> 7;
                const int nb = atom0 + 1 < tc.wa_end ? 2 : 1;
                // one k-stage: wait for its ring slot, publish the tile's info,
                // issue the copies (codes: both CTAs' copies complete on the even
                // CTA's barrier; scale atoms: this CTA's own barrier)
                auto produce = [&](int ks, int nch, uint32_t info, auto res_t) {
                    constexpr bool res_on = decltype(res_t)::value;
                    const int slot = p % STAGES;
                    if (!mbar_wait(&S.empty[slot], ((p / STAGES) & 1) ^ 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    if constexpr (FQ) {
                        // the stage's rows of X quantized (every unit of this 128-row
                        // tile and k-stage counted, or the whole tile): acquire the
                        // counts, then order the TMA reads after them
                        if (rows_in && fq_tile_ok != m_tile) {
                            const int32_t *dn = fq.ctr + 2 + m_tile;
                            const int32_t *fl = fq.ctr + 2 + m_tiles + (int64_t)m_tile * nks + ks;
                            const uint64_t t0 = globaltimer_ns();
                            for (uint32_t i = 0;; ++i) {
                                const int32_t a = ld_acquire_gpu(dn), b = ld_acquire_gpu(fl);
                                if (a == nks * FQ_SUB) {
                                    fq_tile_ok = m_tile;
                                    break;
                                }
                                if (b == FQ_SUB)
                                    break;
                                if ((i & 15) == 15 && (globaltimer_ns() - t0 > wl || *gstat != 0)) {
                                    flag_timeout(S, status);
                                    stop = true;
                                    return;
                                }
                                __nanosleep(128);
                            }
                            fence_proxy_async_global();
                        }
                    }
                    const int c0 = CPS * ks, cx = c0 * (F8 ? 128 : 64); // first chunk, its byte column
                    if (PHI)
                        S.stage_info[slot] = info;
                    Stage &st = S.st[slot];
                    const uint32_t bar = full0 + 8 * slot;
                    const uint32_t sfbytes = (uint32_t)nch * ATOM;
                    uint64_t *sbar = &S.sf_full[slot];
                    if (F8 == F8_MIXED) {
                        // X~ and W~ packed (64-byte rows) side by side in the A tile;
                        // with a residual, X^ as E4M3 in the R tile.  The W~ half lands
                        // on this CTA's own barrier: its scale writers expand it into
                        // the B tile in the padded 4-bit form the residual MMAs read
                        if (lead)
                            mbar_arrive_expect_tx(&S.full[slot], 2 * (A_BYTES / 2 + (res_on ? A_BYTES : 0)));
                        tma_load_2d_pair(st.a, &tmA, bar, c0 * 64, a_y);
                        mbar_arrive_expect_tx(&S.w4_full[slot], A_BYTES / 2);
                        tma_load_2d(st.a + A_BYTES / 2, &tmB4, &S.w4_full[slot], c0 * 64,
                                    tc.w_row0 + (int)rank * BN_HALF);
                        if (res_on)
                            tma_load_2d_pair(st.r, &tmR, bar, cx, a_y);
                    } else {
                        if (lead)
                            mbar_arrive_expect_tx(&S.full[slot], 2 * (A_BYTES + B_TX + (res_on ? A_BYTES : 0)));
                        tma_load_2d_pair(st.a, &tmA, bar, cx, a_y);
                        if (res_on)
                            tma_load_2d_pair(st.r, &tmR, bar, cx, a_y);
                        tma_load_2d_pair(st.b, &tmB, bar, cx, tc.w_row0 + (int)rank * BN_HALF);
                    }
                    mbar_arrive_expect_tx(sbar, nb * sfbytes + (rows_in ? (res_on ? 2 : 1) * sfbytes : 0));
                    if (rows_in) {
                        bulk_load(st.sfa, sfa + ((int64_t)sf_tile * kc + c0) * ATOM, sfbytes, sbar);
                        if (res_on)
                            bulk_load(st.sfr, sfr + ((int64_t)sf_tile * kc + c0) * ATOM, sfbytes, sbar);
                    }
                    for (int h = 0; h < nb; ++h)
                        bulk_load(st.sfb + h * 2 * ATOM, sfb + ((int64_t)(atom0 + h) * kc + c0) * ATOM, sfbytes,
                                  sbar);
                    ++p;
                };
                if constexpr (!PHI) {
                    // full stages, then an odd last chunk (chunk counts known at compile time)
                    for (int ks = 0; ks < nf && !stop; ++ks)
                        produce(ks, CPS, 0u, Bool<RES>{});
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
                            produce(32 * w + b, CPS, info, Bool<true>{});
                        }
                    }
                    for (int w = 0; 32 * w < nf && !stop; ++w) {
                        const int left = nf - 32 * w;
                        uint32_t x = ~rec.bits[w] & (left >= 32 ? 0xffffffffu : (1u << left) - 1u);
                        while (x != 0 && !stop) {
                            const int b = __ffs(x) - 1;
                            x &= x - 1;
                            produce(32 * w + b, CPS, info, Bool<false>{});
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
            if (stop || S.abort_flag)
                // wait (bounded) until the copies of the last stages landed: this
                // CTA's scale atoms, and (even CTA) both CTAs' codes
                for (int q = max(0, p - STAGES); q < p; ++q) {
                    (void)mbar_wait(&S.sf_full[q % STAGES], (q / STAGES) & 1, wl);
                    if (F8 == F8_MIXED)
                        (void)mbar_wait(&S.w4_full[q % STAGES], (q / STAGES) & 1, wl);
                    if (lead)
                        (void)mbar_wait(&S.full[q % STAGES], (q / STAGES) & 1, wl);
                }
        }
    } else if (warp == 1) {
        if (lane == 0 && !skip && lead) {
            // -------------------------------------------- MMA issuer (even CTA)
            int p = 0, it = 0;
            bool stop = false;
            const int64_t c_start = PROF ? clock64() : 0;
            const uint64_t g_start = PROF ? globaltimer_ns() : 0;
            int64_t w_acc = 0, w_full = 0, w_sf = 0;
            for (int tile = pair; tile < tiles && !stop; tile += pairs, ++it) {
                const int64_t ta = PROF ? clock64() : 0;
                if (!mbar_wait<true>(&S.acc_empty, (it & 1) ^ 1, wl, gstat)) {
                    flag_timeout(S, status);
                    break;
                }
                if (PROF)
                    w_acc += clock64() - ta;
                tc_fence_after();
                // the MMAs of the stage at position pos of the tile, with residual
                // mask rm (bit c: chunk c's residual product) known at compile time
                auto mma_stage = [&](int pos, int nch, auto rm_t) {
                    constexpr uint32_t rm = decltype(rm_t)::value;
                    const int slot = p % STAGES, sfs = p % SF_SLOTS;
                    const int64_t t1 = PROF ? clock64() : 0;
                    const bool full_ok = mbar_wait(&S.full[slot], (p / STAGES) & 1, wl, gstat);
                    const int64_t t2 = PROF ? clock64() : 0;
                    if (!full_ok || !mbar_wait<true>(&S.sf_ready[sfs], (p / SF_SLOTS) & 1, wl, gstat)) {
                        flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    if (PROF) {
                        w_full += t2 - t1;
                        w_sf += clock64() - t2;
                    }
                    tc_fence_after();
                    const uint32_t sf = tmem + SF_COL0 + SF_SLOT_COLS * sfs;
                    const Stage &st = S.st[slot];
                    const uint32_t a0 = smem_u32(st.a), r0 = smem_u32(st.r), b0 = smem_u32(st.b);
                    if constexpr (F8 == F8_MIXED) {
                        // main: X~ W~ packed, two K = 64 kind::mxf4 MMAs (scale bytes 0-1, 2-3)
#pragma unroll
                        for (int j = 0; j < 2; ++j)
                            tc_mma_mxf4_pair(tmem, sdesc_k_sw64(a0 + 32 * j), sdesc_k_sw64(a0 + A_BYTES / 2 + 32 * j),
                                             idesc_mxf4(2 * BM, BN, 2 * j, 2 * j), sf, sf + 16, (pos | j) != 0);
                        // residual: X^ (E4M3) times W~ (padded E2M1), four K = 32
                        // kind::mxf8f6f4 MMAs (scale byte j)
                        if (rm & 1) {
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                tc_mma_mxf8_pair(tmem, sdesc_k_sw128(r0 + 32 * j), sdesc_k_sw128(b0 + 32 * j),
                                                 idesc_mxf8_e4m3_e2m1(2 * BM, BN, j, j), sf + 8, sf + 16, 1);
                        }
                    } else {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const int c = F8 ? 0 : j >> 1;
                        if (c >= nch)
                            break;
                        // MXFP4: K = 64 per MMA, scale bytes 2 (j & 1) and up; E4M3: K = 32, byte j
                        const uint32_t id = F8 == F8_W4 ? idesc_mxf8_e4m3_e2m1(2 * BM, BN, j, j)
                                            : F8        ? idesc_mxf8(2 * BM, BN, j, j)
                                                        : idesc_mxf4(2 * BM, BN, 2 * (j & 1), 2 * (j & 1));
                        const uint64_t bd = sdesc_k_sw128(b0 + 32 * j);
                        const uint32_t sfb_t = sf + 16 + 8 * c;
                        if (F8)
                            tc_mma_mxf8_pair(tmem, sdesc_k_sw128(a0 + 32 * j), bd, id, sf + 4 * c, sfb_t,
                                             (pos | j) != 0);
                        else
                            tc_mma_mxf4_pair(tmem, sdesc_k_sw128(a0 + 32 * j), bd, id, sf + 4 * c, sfb_t,
                                             (pos | j) != 0);
                        if ((rm >> c) & 1)
                        {
                            if (F8)
                                tc_mma_mxf8_pair(tmem, sdesc_k_sw128(r0 + 32 * j), bd, id, sf + 8 + 4 * c, sfb_t, 1);
                            else
                                tc_mma_mxf4_pair(tmem, sdesc_k_sw128(r0 + 32 * j), bd, id, sf + 8 + 4 * c, sfb_t, 1);
                        }
                    }
                    }
                    tc_commit_pair_mc(&S.empty[slot], 0x3);
                    ++p;
                };
                if constexpr (!PHI) {
                    for (int ks = 0; ks < nf && !stop; ++ks)
                        mma_stage(ks, CPS, Mask<RES ? 3u : 0u>{});
                    if (nf < nks && !stop)
                        mma_stage(nf, 1, Mask<RES ? 1u : 0u>{});
                    if constexpr (FQ) {
                        // every stage of the tile landed (both CTAs' codes and scale
                        // atoms): its 256-row block's ring slot has one reader fewer
                        if (!stop)
                            red_release_add_gpu(fq.ctr + 2 + m_tiles + m_tiles * nks + tile / n_tiles, 1);
                    }
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
                        mma_stage(pos, CPS, Mask<3u>{});
                    for (; pos < nf && !stop; ++pos)
                        mma_stage(pos, CPS, Mask<0u>{});
                    if (nf < nks && !stop) {
                        if (info >> 31)
                            mma_stage(pos, 1, Mask<1u>{});
                        else
                            mma_stage(pos, 1, Mask<0u>{});
                    }
                }
                if (!stop)
                    tc_commit_pair_mc(&S.acc_full, 0x3);
            }
            // every MMA (and its commits to both CTAs) completes before the
            // final cluster barrier
            tc_commit_pair_mc(&S.drain, 0x1);
            (void)mbar_wait(&S.drain, 0, wl);
            if (PROF) {
                unsigned long long *w = reinterpret_cast<unsigned long long *>(status) + 4;
                atomicAdd(w + 0, (unsigned long long)(clock64() - c_start));
                atomicAdd(w + 1, (unsigned long long)(globaltimer_ns() - g_start));
                atomicAdd(w + 2, (unsigned long long)w_acc);
                atomicAdd(w + 3, (unsigned long long)w_full);
                atomicAdd(w + 4, (unsigned long long)w_sf);
                atomicAdd(w + 5, (unsigned long long)p);
                atomicAdd(w + 6, 1ull);
                atomicAdd(w + 7, (unsigned long long)it);
            }
        }
    } else if (warp < 2 + EPI_WARPS) {
        // ------------------------------------------------ epilogue (warps 2..9)
        const int q = warp & 3;          // TMEM lane quarter this warp may access
        const int h = (warp - 2) >> 2;   // column half of the tile
        const uint32_t acc_empty_lead = mapa_shared(smem_u32(&S.acc_empty), 0);
        uint8_t *stg = S.ystage + (warp - 2) * YSTAGE;
        const uint32_t sw = (uint32_t)((lane >> 1) & 3);   // 64B swizzle: chunk j of row r at (j ^ ((r >> 1) & 3))
        // FQ: the conversion unit this warp holds (-1: none) and its next row
        int fq_u = -1, fq_row = 0, fq_free = -1;   // fq_free: a 256-row block whose ring slot is free
        bool fq_done = !FQ;
        const int fq_units = m_tiles * nks * FQ_SUB;
        // FQ_CALL rows of the held unit (taking the next unit first if none is
        // held): lane l quantizes the 32-element block l % 8 of the stage's
        // columns in row l / 8 of the step (Sec. 3.2 Eq. 3-4 and the residual
        // of Sec. 4.3, the quantizer kernel's arithmetic), stores its 16 bytes
        // of codes and its E8M0 bytes into the scratch.  Returns false when
        // the unit's ring slot is still being read (nothing done).
        auto fq_rows = [&]() -> bool {
            if constexpr (FQ) {
                static_assert(FQ_CALL * 8 == 32, "a step is one block per lane");
                if (fq_u < 0) {
                    int u = 0;
                    if (lane == 0)
                        u = atomicAdd(fq.ctr, 1);
                    u = __shfl_sync(0xffffffffu, u, 0);
                    if (u >= fq_units) {
                        fq_done = true;
                        return true;
                    }
                    fq_u = u;
                    fq_row = 0;
                }
                const int t = fq_u / FQ_SUB, sub = fq_u - t * FQ_SUB;   // t: (128-row tile, k-stage)
                const int mt = t / nks, ks = t - mt * nks;
                const int mp = mt >> 1;                                 // 256-row block
                if (mp >= fq.ring && fq_free != mp) {
                    // the slot's previous block: every output tile has loaded it?
                    int ok = 0;
                    if (lane == 0)
                        ok = ld_acquire_gpu(fq.ctr + 2 + m_tiles + m_tiles * nks + (mp - fq.ring)) == n_tiles;
                    if (!__shfl_sync(0xffffffffu, ok, 0))
                        return false;   // keep the unit, try again later
                    fence_proxy_async_global();
                    fq_free = mp;
                }
                const int kb = K >> 5;                                  // 32-element blocks per row
                const int m = mt * BM + sub * FQ_ROWS + fq_row + (lane >> 3);
                const int mr = (mp % fq.ring) * 2 * BM + (m & (2 * BM - 1));   // its row in the ring
                const int b = ks * 8 + (lane & 7);                      // this lane's block
                const bool ok = m < M && b < kb;                        // (the odd last chunk: 4 blocks)
                uint32_t w[16];
                if (ok) {
                    const uint4 *px = fq.x + (int64_t)m * (K >> 3) + (int64_t)b * 4;
                    uint32_t t0[8], t1[8];
                    ldg256_stream(px, t0);
                    ldg256_stream(px + 2, t1);
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
                // rows past M get zero codes and scale bytes (zero input)
                if (b < kb && RFQ_IN_BOUNDS((int64_t)mr * kb + b, (int64_t)fq.ring * 2 * BM * kb)) {
                    reinterpret_cast<uint4 *>(fq.mcodes)[(int64_t)mr * kb + b] = qz.code;
                    if (RES)
                        reinterpret_cast<uint4 *>(fq.rcodes)[(int64_t)mr * kb + b] = qz.rcode;
                    const int64_t off = sf_mma_offset(mr, b, kc);
                    fq.msf[off] = (uint8_t)qz.sb;
                    if (RES)
                        fq.rsf[off] = (uint8_t)qz.rb;
                }
                fq_row += FQ_CALL;
                if (fq_row == FQ_ROWS) {
                    // the unit's stores before its count, for the TMA reads of other SMs
                    fence_proxy_async_global();
                    __syncwarp();
                    if (lane == 0) {
                        __threadfence();
                        atomicAdd(fq.ctr + 2 + m_tiles + t, 1);
                        atomicAdd(fq.ctr + 2 + mt, 1);
                    }
                    fq_u = -1;
                }
            }
            return true;
        };
        // the accumulator of the warp's next tile (warp-uniform outcome: the
        // tcgen05 loads need the whole warp); with FQ the warp quantizes
        // while it waits
        auto acc_wait = [&](uint32_t parity) -> bool {
            if constexpr (!FQ) {
                return __all_sync(0xffffffffu, mbar_wait(&S.acc_full, parity, wl, gstat));
            } else {
                const uint32_t a = smem_u32(&S.acc_full);
                const uint64_t t0 = globaltimer_ns();
                bool busy = true;   // the last conversion step did work
                for (uint32_t i = 0;; ++i) {
                    // test_wait returns at once; try_wait may suspend the warp, which
                    // would starve the conversion -- and backs off while the next
                    // unit's ring slot is still being read
                    const bool poll = !fq_done && busy;
                    if (__all_sync(0xffffffffu, poll ? mbar_test_wait(a, parity) : mbar_try_wait(a, parity)))
                        return true;
                    if (!fq_done)
                        busy = fq_rows();
                    if ((i & 63) == 63 && __any_sync(0xffffffffu, globaltimer_ns() - t0 > wl || *gstat != 0))
                        return false;
                }
            }
        };
        int it = 0;
        for (int tile = pair; tile < tiles && !skip; tile += pairs, ++it) {
            if (!acc_wait(it & 1)) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            tc_fence_after();
            const TileCoord tc = coord(tile);   // (computed here: fewer registers live across the wait)
            const int row0 = tc.a_row0 + (int)rank * BM + q * 32;
            const uint32_t tcol = tmem + ((uint32_t)(q * 32) << 16) + h * (BN / 2);
            auto release = [&]() {
                // the accumulator goes back to the MMA thread
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    if (lead)
                        mbar_arrive(&S.acc_empty);
                    else
                        mbar_arrive_remote_relaxed(acc_empty_lead);
                }
            };
            if (OUT_BF16) {
                // all 128 columns of this warp into registers as packed bf16
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
                release();
#pragma unroll
                for (int c = 0; c < 4; ++c) {   // 32-column chunks: one 64-byte TMA box row per lane
                    const int col = tc.col0 + h * (BN / 2) + 32 * c;
                    if (col >= N || row0 >= tc.row_end)
                        break;
                    if (GRP && row0 + 32 > tc.row_end && tc.row_end < M) {
                        // a group ends inside this 32-row box: rows past it are
                        // another group's or padding, so each lane stores its own row
                        if (row0 + lane < tc.row_end &&
                            RFQ_IN_BOUNDS((int64_t)(row0 + lane) * N + col + 31, (int64_t)M * N)) {
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
                    uint32_t v[2][32];
#pragma unroll
                    for (int c = 0; c < 2; ++c)
                        tmem_ld_32x32b_x32(tcol + (2 * half + c) * 32, v[c]);
                    tmem_ld_wait();
                    if (half == 1)
                        release();
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
                                if (row0 + lane < tc.row_end &&
                                    RFQ_IN_BOUNDS((int64_t)(row0 + lane) * N + col + 16 * hb + 15, (int64_t)M * N)) {
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
        if constexpr (FQ) {
            // units no warp has taken yet (this CTA has no tile left); a unit
            // whose ring slot is still being read waits here, bounded
            bool go = !skip && S.abort_flag == 0;
            const uint64_t t0 = globaltimer_ns();
            for (uint32_t i = 0; go && !fq_done; ++i) {
                if (!fq_rows())
                    __nanosleep(2000);
                if ((i & 63) == 63) {
                    if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > wl)) {
                        if (lane == 0)
                            flag_timeout(S, status);
                        break;
                    }
                    go = !__any_sync(0xffffffffu, *gstat != 0);
                }
            }
        }
        if (lane == 0)
            bulk_wait_group<0>(); // every TMA store of this warp has completed
    } else if (warp < PHI_WARP) {
        // ------------------------------------------------ scale writers (warps 10..13)
        // Warp quarter q writes TMEM lanes 32q..32q+31; every quarter holds
        // the same words: column j of lane i carries the four scales of row
        // 32 j + i (of this CTA's 128 A rows; of the tile's W~ rows).
        const int q = warp & 3;
        const uint32_t sf_ready_lead = mapa_shared(smem_u32(&S.sf_ready[0]), 0);
        int p = 0;
        bool stop = false;
        for (int tile = pair; tile < tiles && !stop && !skip; tile += pairs) {
            const TileCoord tc = coord(tile);
            const bool rows_in = tc.a_row0 + (int)rank * BM < tc.row_end;
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
                const uint4 z = make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    if (c >= nch)
                        break;
                    const uint4 va = rows_in ? *reinterpret_cast<const uint4 *>(st.sfa + c * ATOM + lane * 16) : z;
                    const uint4 vb0 = *reinterpret_cast<const uint4 *>(st.sfb + c * ATOM + lane * 16);
                    const uint4 vb1 = b1_in ? *reinterpret_cast<const uint4 *>(st.sfb + (2 + c) * ATOM + lane * 16) : z;
                    tmem_st_32x32b_x4(tb + 4 * c, va.x, va.y, va.z, va.w);
                    if ((rm >> c) & 1) {
                        const uint4 vr = rows_in ? *reinterpret_cast<const uint4 *>(st.sfr + c * ATOM + lane * 16) : z;
                        tmem_st_32x32b_x4(tb + 8 + 4 * c, vr.x, vr.y, vr.z, vr.w);
                    }
                    tmem_st_32x32b_x4(tb + 16 + 8 * c, vb0.x, vb0.y, vb0.z, vb0.w);
                    tmem_st_32x32b_x4(tb + 20 + 8 * c, vb1.x, vb1.y, vb1.z, vb1.w);
                }
                if constexpr (F8 == F8_MIXED) {
                    // this CTA's packed W~ half (the main MMAs read it from both
                    // CTAs, so the stage is ready only once it landed) and, for a
                    // residual stage, its padded 4-bit copy: lane l of quarter q
                    // takes row 32 q + l, 16-code chunk c (8 packed bytes, then an
                    // 8-byte gap the MMA skips) to 16-byte position c ^ (row & 7)
                    // of the 128-byte swizzled row, from the 64-byte swizzled
                    // packed row (16-byte chunk j at j ^ ((row >> 1) & 3))
                    if (!__all_sync(0xffffffffu, mbar_wait(&S.w4_full[slot], (p / STAGES) & 1, wl, gstat))) {
                        if (lane == 0)
                            flag_timeout(S, status);
                        stop = true;
                        return;
                    }
                    if (rm & 1) {
                        const int row = q * 32 + lane;
                        const uint32_t src = smem_u32(st.a + A_BYTES / 2) + row * 64;
                        const uint32_t dst = smem_u32(st.b) + row * 128;
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            uint32_t w0, w1, w2, w3;
                            asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                                         : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
                                         : "r"(src + ((j ^ ((row >> 1) & 3)) << 4)));
                            asm volatile("st.shared.v2.u32 [%0], {%1, %2};" ::"r"(dst + (((2 * j) ^ (row & 7)) << 4)),
                                         "r"(w0), "r"(w1)
                                         : "memory");
                            asm volatile("st.shared.v2.u32 [%0], {%1, %2};" ::"r"(dst + (((2 * j + 1) ^ (row & 7)) << 4)),
                                         "r"(w2), "r"(w3)
                                         : "memory");
                        }
                        fence_proxy_async_smem();   // generic-proxy writes, read by the MMAs
                    }
                }
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    if (lead)
                        mbar_arrive(&S.sf_ready[sfs]);
                    else
                        mbar_arrive_remote_relaxed(sf_ready_lead + 8 * sfs);
                }
                ++p;
            };
            if constexpr (!PHI) {
                for (int ks = 0; ks < nf && !stop; ++ks)
                    write_stage(CPS, Mask<RES ? 3u : 0u>{});
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
                    write_stage(CPS, Mask<3u>{});
                for (; pos < nf && !stop; ++pos)
                    write_stage(CPS, Mask<0u>{});
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
        // Record of the CTA's j-th tile: chunk c of the pair's row tile m
        // (128 rows) needs its residual when phi[m][c / phi_chunks] is non-zero.
        const int my_tiles = pair < tiles ? (tiles - pair + pairs - 1) / pairs : 0;
        auto chunk_on = [&](const TileCoord &tc, int c) {
            const int col = c / phi_chunks;
            bool on = false;
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                const int row = tc.a_row0 + r * BM, mt = row / BM;
                if (row < tc.row_end && mt < m_tiles && __ldg(phi + (int64_t)mt * phi_cols + col) != 0)
                    on = true;
            }
            return on;
        };
        for (int j = 0; j < (skip ? 0 : my_tiles); ++j) {
            const int r = j & 1;
            if (j >= 2 && !__all_sync(0xffffffffu, mbar_wait(&S.phi_empty[r], ((j >> 1) - 1) & 1,
                                                             wl, gstat))) {
                if (lane == 0)
                    flag_timeout(S, status);
                break;
            }
            const TileCoord tcj = coord(pair + j * pairs);
            PhiRec &rec = S.rec[r];
            uint32_t n_res = 0;
            for (int w = 0; 32 * w < nf; ++w) {
                const int ks = 32 * w + lane;
                const bool on = ks < nf && (chunk_on(tcj, CPS * ks) || (!F8 && chunk_on(tcj, CPS * ks + 1)));
                const uint32_t word = __ballot_sync(0xffffffffu, on);
                if (lane == 0)
                    rec.bits[w] = word;
                n_res += __popc(word);
            }
            const uint32_t tail = nf < nks && chunk_on(tcj, CPS * nf) ? 1u : 0u;
            if (lane == 0)
                rec.info = n_res | tail << 31;
            mbar_arrive(&S.phi_full[r]);
        }
    }

    // ---------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    cluster_sync(); // the peer no longer signals this CTA, the pair's MMAs are complete
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, TMEM_COLS);
    }
    if constexpr (FQ) {
        // the grid's last CTA to get here zeroes the counters for the next call
        if (threadIdx.x == 0) {
            __threadfence();
            S.fq_last = atomicAdd(fq.ctr + 1, 1) == (int)gridDim.x - 1;
        }
        __syncthreads();
        if (S.fq_last) {
            const int n = 2 + m_tiles + m_tiles * nks + m_pairs;
            for (int i = threadIdx.x; i < n; i += blockDim.x)
                if (i != 1)
                    fq.ctr[i] = 0;
            __syncthreads();
            if (threadIdx.x == 0) {
                __threadfence();
                fq.ctr[1] = 0;
            }
        }
    }
}

template <bool RES, bool PHI, bool OUT, int F8, bool GRP, bool FQ = false, bool PROF = false>
cudaError_t launch_variant(const CUtensorMap &ta, const CUtensorMap &tr, const CUtensorMap &tb,
                           const CUtensorMap &ty, const GemmMxf4Args &a, cudaStream_t st,
                           const CUtensorMap *tb4 = nullptr)
{
    auto kern = gemm_mxf4_pair_kernel<RES, PHI, OUT, F8, GRP, FQ, PROF>;
    static int max_pairs = 0; // per variant: clusters of two that fit on the device at once
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBytes);
    if (e != cudaSuccess)
        return e;
    if (max_pairs == 0) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(2 * (num_sms() / 2));
        cfg.blockDim = dim3(PHI ? THREADS + 32 : THREADS);
        cfg.dynamicSmemBytes = kSmemBytes;
        int n = 0;
        e = cudaOccupancyMaxActiveClusters(&n, kern, &cfg);
        if (e != cudaSuccess)
            return e;
        max_pairs = n > 0 ? n : 1;
    }
    // grouped: the tile count depends on the device-side row offsets; every
    // pair of the grid walks the tiles that exist
    const int64_t tiles = a.groups > 0 ? INT64_MAX : ((a.N + BN - 1) / BN) * ((a.M + 2 * BM - 1) / (2 * BM));
    const int grid = 2 * (int)(tiles < max_pairs ? tiles : max_pairs);
    const int phi_chunks = a.phi_r_s / 128;
    const int phi_cols = a.phi ? (int)((a.K + a.phi_r_s - 1) / a.phi_r_s) : 0;
    FqArgs fq = {};
    if (FQ) {
        fq.x = static_cast<const uint4 *>(a.fq_x);
        fq.mcodes = static_cast<uint32_t *>(const_cast<void *>(a.a_codes));
        fq.rcodes = static_cast<uint32_t *>(const_cast<void *>(a.r_codes));
        fq.msf = static_cast<uint8_t *>(const_cast<void *>(a.a_sf));
        fq.rsf = static_cast<uint8_t *>(const_cast<void *>(a.r_sf));
        fq.ctr = a.fq_ctr;
        fq.ring = a.fq_ring;
    }
    kern<<<grid, PHI ? THREADS + 32 : THREADS, kSmemBytes, st>>>(
        ta, tr, tb, ty, tb4 ? *tb4 : tb, (const uint8_t *)a.a_sf, (const uint8_t *)a.r_sf, (const uint8_t *)a.b_sf, a.phi, phi_chunks,
        phi_cols, (int)a.M, (int)a.N, (int)a.K, a.status, a.group_off, a.groups, a.y, fq);
    return cudaGetLastError();
}

} // namespace

cudaError_t launch_gemm_mxf4_pair(const GemmMxf4Args &a, cudaStream_t st)
{
    CUtensorMap ta, tr, tb, ty;
    if (a.b4_codes) {
        // the mixed-rate FP4-to-FP8 residual: X~ and W~ packed (64-byte boxes,
        // 64-byte swizzle), X^ as E4M3 (128-byte boxes); the kernel makes
        // the padded 4-bit W~ tile itself, so no map reads W~ in that form
        if (!a.r_codes || a.groups > 0 || a.fq_x || a.prof)
            return cudaErrorInvalidValue;
        CUtensorMap tb4;
        const uint64_t kp = (uint64_t)a.K / 2, k8 = (uint64_t)a.K, yrow = (uint64_t)a.N * (a.out_bf16 ? 2 : 4);
        if (!encode_tmap_2d_u8(&ta, a.a_codes, kp, (uint64_t)a.M, kp, 64, BM, 64) ||
            !encode_tmap_2d_u8(&tb4, a.b4_codes, kp, (uint64_t)a.N, kp, 64, BN_HALF, 64) ||
            !encode_tmap_2d_u8(&tr, a.r_codes, k8, (uint64_t)a.M, k8, ROW, BM, 128) ||
            !encode_tmap_2d_u8(&ty, a.y, yrow, (uint64_t)a.M, yrow, 64, 32, 64))
            return cudaErrorInvalidValue;
        tb = tb4;   // (unused by this form)
        const bool phi = a.phi != nullptr && a.K / 128 <= REC_WORDS * 32;
        if (phi)
            return a.out_bf16 ? launch_variant<true, true, true, F8_MIXED, false>(ta, tr, tb, ty, a, st, &tb4)
                              : launch_variant<true, true, false, F8_MIXED, false>(ta, tr, tb, ty, a, st, &tb4);
        return a.out_bf16 ? launch_variant<true, false, true, F8_MIXED, false>(ta, tr, tb, ty, a, st, &tb4)
                          : launch_variant<true, false, false, F8_MIXED, false>(ta, tr, tb, ty, a, st, &tb4);
    }
    const uint64_t kb = a.f8 ? (uint64_t)a.K : (uint64_t)a.K / 2; // code bytes per row
    const uint64_t w_rows = (uint64_t)a.N * (a.groups > 0 ? (uint64_t)a.groups : 1u);
    const uint64_t a_rows = a.fq_x ? (uint64_t)a.fq_ring * 2 * BM : (uint64_t)a.M;   // FQ: the ring
    if (a.w4 && !a.f8)
        return cudaErrorInvalidValue;
    if (!encode_tmap_2d_u8(&ta, a.a_codes, kb, a_rows, kb, ROW, BM, 128) ||
        !(a.w4 ? encode_tmap_2d_e2m1_padded(&tb, a.b_codes, (uint64_t)a.K, w_rows, BN_HALF)
               : encode_tmap_2d_u8(&tb, a.b_codes, kb, w_rows, kb, ROW, BN_HALF, 128)))
        return cudaErrorInvalidValue;
    if (a.r_codes) {
        if (!encode_tmap_2d_u8(&tr, a.r_codes, kb, a_rows, kb, ROW, BM, 128))
            return cudaErrorInvalidValue;
    } else {
        tr = ta;
    }
    // Y [M][N] (bf16 or fp32) as bytes; boxes of 64 bytes x 32 rows, 64B swizzle
    const uint64_t yrow = (uint64_t)a.N * (a.out_bf16 ? 2 : 4);
    if (!encode_tmap_2d_u8(&ty, a.y, yrow, (uint64_t)a.M, yrow, 64, 32, 64))
        return cudaErrorInvalidValue;
    // Beyond REC_WORDS * 32 full k-stages the record does not fit: every
    // residual product is then issued (exact: phi = 0 residuals are zero).
    const bool res = a.r_codes != nullptr;
    if (a.prof) {
        // the measuring instantiation: RFQ with a residual, no phi, MXFP4 operands
        if (!res || a.f8 || a.groups > 0 || a.phi || a.fq_x)
            return cudaErrorInvalidValue;
        return a.out_bf16 ? launch_variant<true, false, true, false, false, false, true>(ta, tr, tb, ty, a, st)
                          : launch_variant<true, false, false, false, false, false, true>(ta, tr, tb, ty, a, st);
    }
    if (a.fq_x) {
        // the fused quantizer: plain MXFP4 operands written by the kernel itself
        if (a.f8 || a.groups > 0 || a.phi)
            return cudaErrorInvalidValue;
        if (res)
            return a.out_bf16 ? launch_variant<true, false, true, false, false, true>(ta, tr, tb, ty, a, st)
                              : launch_variant<true, false, false, false, false, true>(ta, tr, tb, ty, a, st);
        return a.out_bf16 ? launch_variant<false, false, true, false, false, true>(ta, tr, tb, ty, a, st)
                          : launch_variant<false, false, false, false, false, true>(ta, tr, tb, ty, a, st);
    }
    const bool phi = res && a.phi != nullptr && a.K / (a.f8 ? 128 : 256) <= REC_WORDS * 32;
#define RFQ_GV_F(R, P, O, G)                                                                                      \
    (!a.f8 ? launch_variant<R, P, O, 0, G>(ta, tr, tb, ty, a, st)                                                 \
           : a.w4 ? launch_variant<R, P, O, F8_W4, G>(ta, tr, tb, ty, a, st)                                      \
                  : launch_variant<R, P, O, 1, G>(ta, tr, tb, ty, a, st))
#define RFQ_GV(R, P, O) return a.groups > 0 ? RFQ_GV_F(R, P, O, true) : RFQ_GV_F(R, P, O, false)
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
#undef RFQ_GV_F
}

RFQ_DEBUG_WORD_ACCESSOR(debug_word_gemm_mxf4_pair)

} // namespace rfq
