/*
 * rfq.h -- C ABI of the GB300 (sm_103a) Residual Fallback Quantization
 * (RFQ) linear layer: "Activation Outliers Matter: Robust Recovery for
 * Quantized Multimodal LLMs", Sec. 3.2-3.3 (formats), Sec. 4.3 and
 * Algorithm 1 (method).
 *
 * The layer computes Y = X W for an activation X [M x K] (bf16) and a weight
 * W [K x N] (bf16) as
 *
 *     Y = Q(X) Q(W) + phi * Q(X - Q(X)) Q(W)                  (Eq. rfq)
 *
 * where Q is a block quantizer to a 4-bit format (MXFP4 or HiF4) along K.
 * The paper writes Z = X Y with X [P x R], Y [R x Q]; here P = M, R = K,
 * Q = N and the paper's Y is W.
 *
 * Conventions shared by every entry point:
 *   - Every pointer named "device" is CUDA device memory on the current
 *     device, allocated and owned by the caller; the library never allocates
 *     device memory and never frees a caller's buffer.
 *   - Every device pointer must be 16-byte aligned (RFQ_ERR_ALIGNMENT).
 *   - Calls are asynchronous: they validate the arguments on the host,
 *     enqueue kernels on `stream` (a cudaStream_t; NULL = legacy default
 *     stream) and return.  On any argument error nothing is launched.
 *   - bf16 inputs must be finite; non-finite inputs give unspecified codes
 *     but never a fault.
 *   - The library needs an sm_103 device (GB300); otherwise RFQ_ERR_DEVICE.
 *
 * Storage of a quantized matrix (rfq_qtensor), rows x k, quantized along k:
 *   codes   [rows][k/2] bytes; element 2j of a row in the low nibble of byte
 *           j, element 2j+1 in the high nibble.
 *   MXFP4   E2M1 codes (sign, 2 exponent bits, 1 mantissa bit, Sec. 3.2.2)
 *           with one E8M0 scale byte 2^(byte-127) per 32 elements
 *           (Sec. 3.2 Eq. 3-4).  Scale layouts:
 *             RFQ_SCALE_ROWMAJOR  [rows][k/32] bytes (k % 32 == 0)
 *             RFQ_SCALE_MMA       the tensor-core layout consumed by
 *               rfq_linear (k % 128 == 0): rows padded to a multiple of 128
 *               and split into 512-byte atoms of 128 rows x 4 k-blocks; the
 *               byte for (row m, k-block b) lives at
 *                 ((m/128) * (k/128) + b/4) * 512 + (m%32)*16 + ((m/32)%4)*4 + b%4
 *               Bytes of padding rows (m >= rows) are 0.
 *   HiF4    S1P2 codes (sign, 1 integer bit, 2 fraction bits) with one
 *           32-bit metadata word per 64 elements (Sec. 3.3):
 *           bits [7:0] UE6M2 macro scale (E in [7:2], bias 48; M in [1:0]),
 *           bits [15:8] E1_8 (bit g: group of 8 elements g),
 *           bits [31:16] E1_16 (bit j: sub-group of 4 elements j).
 *           Metadata layouts (k % 64 == 0):
 *             RFQ_SCALE_ROWMAJOR  [rows][k/64] uint32
 *             RFQ_SCALE_MMA       block-major [k/64][rows rounded up to 128]
 *                                 uint32, the layout rfq_linear consumes
 *   BF16    an exact bf16 expansion of a quantized matrix, [rows][k]
 *           (codes = the bf16 data, scales unused): rfq_dequant writes it,
 *           and rfq_linear takes the HiF4 weight in this form.
 *   MXFP8   E4M3 codes (Sec. 3.2.1: sign, 4 exponent bits with bias 7, 3
 *           mantissa bits; exponent field 0 subnormal; no infinity;
 *           S.1111.111 is NaN; largest finite 448), one byte per element:
 *           codes [rows][k]; one E8M0 scale byte per 32 elements with the
 *           MXFP4 scale layouts.  The block exponent is floor(log2 amax) - 8
 *           (clamped to [-127, 127]); elements round to nearest even and
 *           saturate at +-448.  An MXFP4 tensor re-encoded by rfq_convert is
 *           an MXFP8 tensor holding the same values.
 */
#ifndef RFQ_H
#define RFQ_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define RFQ_API __attribute__((visibility("default")))
#else
#define RFQ_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RFQ_OK = 0,
    RFQ_ERR_INVALID_ARG = 1, /* NULL pointer or an enum value out of range */
    RFQ_ERR_SHAPE = 2,       /* sizes violate the call's constraints */
    RFQ_ERR_ALIGNMENT = 3,   /* a device pointer is not 16-byte aligned */
    RFQ_ERR_UNSUPPORTED = 4, /* valid but unimplemented combination */
    RFQ_ERR_CUDA = 5,        /* a CUDA runtime call or a launch failed */
    RFQ_ERR_TIMEOUT = 6,     /* a kernel's bounded wait expired (device status) */
    RFQ_ERR_DEVICE = 7,      /* the current device is not an sm_103 GPU */
    RFQ_ERR_NONFINITE = 8    /* rfq_check_finite found an Inf or NaN (device status) */
} rfq_status;

typedef enum { RFQ_FMT_MXFP4 = 0, RFQ_FMT_HIF4 = 1, RFQ_FMT_BF16 = 2, RFQ_FMT_MXFP8 = 3 } rfq_format;

typedef enum { RFQ_SCALE_ROWMAJOR = 0, RFQ_SCALE_MMA = 1 } rfq_scale_layout;

/* Fallback indicator phi(p, r) of Sec. 4.3 over tiles of p_s rows x r_s
 * columns of X.  The paper gives no formula for it:
 *   RFQ_FALLBACK_NONE  phi = 0: plain W4A4, no residual pathway
 *   RFQ_FALLBACK_ALL   phi = 1 on every tile (the default; Sec. 1 describes
 *                      RFQ as working without threshold-based selection)
 *   RFQ_FALLBACK_AMAX  phi(p, r) = 1 iff max |x| over the tile > tau */
typedef enum {
    RFQ_FALLBACK_NONE = 0,
    RFQ_FALLBACK_ALL = 1,
    RFQ_FALLBACK_AMAX = 2
} rfq_fallback_mode;

typedef enum { RFQ_OUT_F32 = 0, RFQ_OUT_BF16 = 1 } rfq_out_dtype;

typedef struct {
    int32_t fmt;          /* rfq_format */
    int32_t scale_layout; /* rfq_scale_layout (ignored for RFQ_FMT_BF16) */
    int64_t rows;         /* M for an activation, N for a weight */
    int64_t k;            /* length of the quantized (reduction) axis */
    void *codes;          /* device, see "Storage" above */
    void *scales;         /* device, see "Storage" above */
} rfq_qtensor;

typedef struct {
    int32_t mode; /* rfq_fallback_mode */
    float tau;    /* threshold for RFQ_FALLBACK_AMAX */
    int32_t p_s;  /* tile rows (>= 1); rfq_linear reads phi tiles of 128 rows */
    int32_t r_s;  /* tile columns, a multiple of 32; rfq_linear needs a multiple of 128 */
} rfq_fallback;

/* Human-readable name of a status code (static string, never NULL). */
RFQ_API const char *rfq_status_string(rfq_status s);

/* Byte sizes of the code and scale arrays of a rows x k quantized matrix in
 * the given format and scale layout (host only, no device work).
 * Errors: RFQ_ERR_INVALID_ARG (NULL outputs, bad enums), RFQ_ERR_SHAPE
 * (rows < 0, k not a multiple of the layout's granule). */
RFQ_API rfq_status rfq_qtensor_bytes(int32_t fmt, int32_t scale_layout, int64_t rows, int64_t k,
                             size_t *codes_bytes, size_t *scale_bytes);

/* Weight quantization W~ = Q(W) (Sec. 4.3; Algorithm 1 quantizes every
 * weight block).  W: device bf16 [K][N] row-major.  out->fmt,
 * out->scale_layout, out->codes and out->scales are set by the caller and
 * out->rows must equal N, out->k must equal K; codes are written K-major
 * ([N][K/2]; MXFP8: [N][K]).  Formats: MXFP4, HiF4, MXFP8 (the W8A8
 * baseline of Table 1).  Meant to run once per weight, off the hot path.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_quantize_weight(const void *w_bf16, int64_t K, int64_t N, rfq_qtensor *out,
                               void *stream);

/* RFQ activation decomposition in one pass over X (Sec. 4.3, Algorithm 1):
 *   X~ = Q(X), dX = X - X~, X^ = Q(dX) where phi = 1 (same format, Sec. 4.3),
 * with the E8M0 scale floor(log2 amax) - 2 clamped to [-127, 127] and
 * round-to-nearest-even, saturating element rounding (MXFP4); HiF4 per its
 * encoder.  X: device bf16 [M][K] row-major.  xq: main pathway output,
 * xr: residual pathway output (both with rows = M, k = K and the same fmt
 * and layout); xr may be NULL only when fb->mode == RFQ_FALLBACK_NONE.
 * Two more format combinations:
 *   xq MXFP4, xr MXFP8   the FP4-to-FP8 residual pathway named in Sec. 4.2:
 *                        X~ = Q_MXFP4(X), X^ = Q_MXFP8(X - X~) (E4M3 scale
 *                        floor(log2 amax) - 8), one pass over X;
 *   xq MXFP8, no residual (fb->mode == RFQ_FALLBACK_NONE; a residual
 *                        returns RFQ_ERR_UNSUPPORTED): X -> MXFP8, the
 *                        activation of the W4A8 / W8A8 baselines (Table 1).
 * Residual codes and scales of tiles with phi = 0 are written as zero.
 * phi: device bytes [ceil(M/p_s)][ceil(K/r_s)], may be NULL; fb may be
 * NULL (= RFQ_FALLBACK_ALL).  M may be 0 (nothing is launched).
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_quantize_act(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb,
                            rfq_qtensor *xq, rfq_qtensor *xr, uint8_t *phi, void *stream);

/* rfq_quantize_act that in the same pass over X also writes X~ (and X^) in
 * the form rfq_linear multiplies, replacing a separate conversion pass:
 *   xq, xr HiF4 (Sec. 3.3):  xq_op (and xr_op) receive the exact bf16 values
 *       of X~ (and X^), the products of rfq_dequant(xq) and rfq_dequant(xr):
 *       every HiF4 value has at most six significant bits and an exponent
 *       inside bf16's range.  RFQ_FMT_BF16 operands of rows = M, k = K
 *       (device bf16 [M][K] row-major, 16-byte aligned); xr_op is required
 *       with a residual and must be NULL when fb->mode == RFQ_FALLBACK_NONE.
 *       X^ values of phi = 0 tiles are zero.
 *   xq MXFP4, xr MXFP8 (the FP4-to-FP8 residual, Sec. 4.2):  xq_op receives
 *       X~ re-encoded as MXFP8 (RFQ_FMT_MXFP8, the layout of xq), the
 *       product of rfq_convert(xq): every E2M1 value is an E4M3 value, so
 *       the codes change and the scale bytes do not.  xr_op must be NULL
 *       (X^ is already MXFP8) and the mode must have a residual.
 * Other format combinations return RFQ_ERR_UNSUPPORTED.  xq, xr, phi and fb
 * as for rfq_quantize_act.  Asynchronous on `stream`.
 * Errors: as rfq_quantize_act. */
RFQ_API rfq_status rfq_quantize_act_expand(const void *x_bf16, int64_t M, int64_t K, const rfq_fallback *fb,
                                           rfq_qtensor *xq, rfq_qtensor *xr, uint8_t *phi, rfq_qtensor *xq_op,
                                           rfq_qtensor *xr_op, void *stream);

/* Bytes of device workspace rfq_linear needs (a status word, padded).  The
 * caller zeroes it.  Its int32 words: [0] the device status that
 * rfq_workspace_status reads; [1] the limit of the call's bounded waits in
 * microseconds (0: two seconds); [2] held start: when non-zero, the GEMM's
 * copy producers wait (within that limit) for word [3] to become non-zero
 * before their first copy and record RFQ_ERR_TIMEOUT if it stays zero -- a
 * way to run a kernel's timeout path with no copy or MMA in flight.  Every
 * GEMM entry point (rfq_linear, rfq_linear_fused, rfq_linear_grouped)
 * honours words [1] to [3]; leave them zero in normal use.  Bytes 32..95
 * receive rfq_linear_profile's counters.  With the environment variable
 * RFQ_DEBUG_SYNC set (to anything but "0") when the library first checks it,
 * every GEMM entry point synchronizes its stream after the launch and
 * returns the status the workspace then holds (as rfq_workspace_status
 * would), so a timeout surfaces at the call that caused it. */
RFQ_API size_t rfq_linear_workspace_bytes(void);

/* RFQ GEMM (Algorithm 1, Eq. rfq): Y = X~ W~ + phi X^ W~ with both products
 * accumulated into one fp32 accumulator per output tile, the weight tile read
 * once for both.  xq: [M x K] main codes; xr: [M x K] residual codes or NULL
 * (plain W4A4); phi: device bytes [ceil(M/128)][K/r_s] selecting the
 * residual k-tiles per 128-row tile, or NULL (= all ones); phi_r_s: the
 * column tile r_s of phi (a multiple of 128; ignored when phi is NULL).
 * The residual of every phi = 0 tile must be stored as zero, as
 * rfq_quantize_act writes it: phi only lets the GEMM skip residual loads and
 * products, at its own granularity (it may still include a phi = 0 tile that
 * shares a 256-row or 256-column block with a phi = 1 one).
 * wq: [N x K] weight.  MXFP4: every operand MXFP4 with RFQ_SCALE_MMA,
 * K % 128 == 0.  MXFP8: xq (and xr) MXFP8 (E4M3, kind::mxf8f6f4 MMAs)
 * with RFQ_SCALE_MMA, K % 128 == 0, and wq MXFP8 or MXFP4 -- the W8A8 and
 * W4A8 baselines and the FP4-to-FP8 RFQ (X~ re-encoded by rfq_convert, X^
 * from the MXFP8 residual pathway).  An MXFP4 wq (codes 32-byte aligned) is
 * multiplied as E2M1 (E4M3 x E2M1 MMAs) straight from its packed codes, half
 * the weight bytes of its E4M3 re-encoding, which gives the same Y.  HiF4 (Sec. 3.3): wq is the exact bf16 expansion of the HiF4
 * weight (RFQ_FMT_BF16, from rfq_dequant), K % 64 == 0, phi_r_s a multiple
 * of 64, and xq/xr are either HiF4 with RFQ_SCALE_MMA metadata (expanded
 * exactly to bf16 in shared memory inside the GEMM) or their exact bf16
 * expansions (RFQ_FMT_BF16, from rfq_dequant; faster when N spans several
 * tiles, since each activation tile is then expanded once instead of once
 * per output tile).  Both run on the bf16 tensor path.  N % 16 == 0, M >= 0.  y: device [M][N] row-major fp32 or bf16 (round-to-nearest-even
 * of the fp32 accumulator).  workspace: device, rfq_linear_workspace_bytes()
 * bytes, zeroed by the caller once; a kernel that gives up a bounded wait
 * records a timeout there (read it with rfq_workspace_status).  The record
 * is sticky: later calls with that workspace return without computing until
 * it is cleared.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_linear(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi,
                      int32_t phi_r_s, const rfq_qtensor *wq, void *y, int32_t out_dtype,
                      void *workspace, void *stream);

/* The RFQ linear layer end to end from host memory (Algorithm 1, Eq. rfq,
 * with X and Y in host memory): Y = X~ W~ + phi X^ W~ for a bf16 X on the
 * host.  The call copies X to the device, quantizes it (rfq_quantize_act,
 * MXFP4 main and residual pathways per fb), multiplies it by wq (rfq_linear)
 * and copies Y back, in chunks of chunk_rows rows: each chunk's
 * host-to-device copy runs on a copy stream of the library's, its two
 * kernels on `stream`, its device-to-host copy on a second copy stream, so
 * the copies of one chunk overlap the kernels and copies of the others.
 * `stream` then waits for the copy streams: y_host is complete once the
 * stream has passed the call (the call itself returns after enqueueing).
 * Y equals rfq_linear's on the same operands bit for bit (row chunking
 * does not change any output element's accumulation).
 *   x_host: host bf16 [M][K] row-major; page-locked memory lets the copies
 *           run asynchronously (pageable memory works, with copies that
 *           then block the host).
 *   y_host: host [M][N] row-major, bf16 or fp32 per out_dtype.
 *   fb: NULL (= RFQ_FALLBACK_ALL), RFQ_FALLBACK_NONE (plain W4A4; xr NULL)
 *       or RFQ_FALLBACK_AMAX with p_s = 128 and r_s a multiple of 128.
 *   wq: MXFP4 W~ [N x K] with RFQ_SCALE_MMA (device).
 *   chunk_rows: a multiple of 128; 0 selects 8192.  M = 0 does nothing
 *   (the host and device buffers may then be NULL).
 *   Device scratch, all the caller's (the library allocates no device
 *   memory; it creates two copy streams per device, kept for the process,
 *   and a few events per call): x_dev bf16 [M][K] (16-byte aligned); xq, xr
 *   MXFP4 qtensors of M x K with RFQ_SCALE_MMA (xr NULL exactly when fb is
 *   RFQ_FALLBACK_NONE); phi [ceil(M/128)][ceil(K/r_s)] bytes with
 *   RFQ_FALLBACK_AMAX, else ignored; y_dev [M][N]; workspace as for
 *   rfq_linear.  Nothing else may use these buffers until `stream` has
 *   passed the call.  Calls on one device share the two copy streams, so
 *   the copies of concurrent calls run one after another.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED (other formats or layouts), RFQ_ERR_CUDA,
 * RFQ_ERR_DEVICE; every check happens before the first copy is enqueued. */
RFQ_API rfq_status rfq_linear_host(const void *x_host, int64_t M, int64_t K, const rfq_fallback *fb,
                                   const rfq_qtensor *wq, void *y_host, int32_t out_dtype, int64_t chunk_rows,
                                   void *x_dev, rfq_qtensor *xq, rfq_qtensor *xr, uint8_t *phi, void *y_dev,
                                   void *workspace, void *stream);

/* Workspace bytes rfq_linear_fused needs for an M x K activation and the
 * fallback mode fb (NULL = RFQ_FALLBACK_ALL); 0 for sizes it rejects
 * (K % 128 != 0).  For M <= 128 it is rfq_linear_workspace_bytes(); beyond,
 * it adds the kernel's counters and a scratch ring for the quantized X of
 * at most 12 blocks of 256 rows: 256 R K (1 + 1/16) bytes with the residual
 * for R = min(12, ceil(M / 256)) (half without) -- about 17 MB for K = 5120,
 * whatever M. */
RFQ_API size_t rfq_linear_fused_workspace_bytes(int64_t M, int64_t K, const rfq_fallback *fb);

/* RFQ linear layer with the activation quantizer fused into the GEMM (the
 * on-the-fly residual of Sec. 4.3): Y = Q(X) W~ + phi Q(X - Q(X)) W~ with X
 * read as bf16 and quantized inside the GEMM kernel, block by block, exactly
 * as rfq_quantize_act would (MXFP4: E8M0 scale floor(log2 amax) - 2, RNE
 * saturating E2M1 codes, exact residual): one launch, no separate
 * quantizer pass.  x_bf16: device bf16 [M][K] row-major (16-byte aligned).
 * wq: MXFP4 weight [N x K] with RFQ_SCALE_MMA scales.  fb: NULL or mode
 * RFQ_FALLBACK_ALL (residual on every block) or RFQ_FALLBACK_NONE (plain
 * W4A4); RFQ_FALLBACK_AMAX returns RFQ_ERR_UNSUPPORTED.  K % 128 == 0,
 * N % 16 == 0, M >= 0.  y, out_dtype: as for rfq_linear.
 * workspace: device, rfq_linear_fused_workspace_bytes(M, K, fb) bytes,
 * 16-byte aligned, zeroed by the caller once; its first 256 bytes are the
 * GEMM workspace of rfq_linear (status word, wait limit, held start).  For
 * M > 128 the GEMM runs on CTA pairs whose epilogue warps, between output
 * tiles, quantize X in units of 8 rows x 256 columns into the rest of the
 * workspace's ring, each element once; a stage's copies wait (bounded) until
 * its rows are quantized, a block of rows is written only once every output
 * tile has loaded the block its slot held before, and the kernel leaves its
 * counters zero for the next call.  Calls that overlap on the GPU must not
 * share a workspace.  For M <= 128 each output tile quantizes its rows of X itself in shared
 * memory (one row tile, so nothing is repeated across row tiles).
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_linear_fused(const void *x_bf16, int64_t M, int64_t K, const rfq_qtensor *wq,
                                    const rfq_fallback *fb, void *y, int32_t out_dtype, void *workspace,
                                    void *stream);

/* Grouped RFQ GEMM for mixture-of-experts layers (the MoE expert
 * projections that hold most of Qwen3-VL-30B's weights, Table 2): every
 * group g (an expert) computes
 *     Y[rows of g] = X~ W~_g + phi X^ W~_g             (Algorithm 1, Eq. rfq)
 * in one launch over all groups.  xq / xr: the activations of all groups
 * stacked along rows (rfq_qtensor as for rfq_linear, rows = the stacked
 * total); group_off: device int32 [groups + 1], rows [group_off[g],
 * group_off[g+1]) belong to group g; every group start must be a multiple
 * of 128 (pad each group's rows), the offsets non-decreasing and
 * group_off[groups] <= rows.  The offsets are read on the device (a router
 * may write them): a violation is recorded in the workspace, nothing is
 * computed, and rfq_workspace_status returns RFQ_ERR_SHAPE.  wq: the
 * weights of all groups stacked, rows = groups * N (group g's W~ rows
 * [g N, (g+1) N)), N % 128 == 0.  y: device [rows][N]; every row of a
 * group (the rows padding it to the next group's start included) is
 * written, rows before group_off[0] or from group_off[groups] on are not.  Operands MXFP4, or MXFP8
 * activations with an MXFP8 or MXFP4 (32-byte aligned) W~, as for rfq_linear; all with
 * RFQ_SCALE_MMA, K % 128 == 0; phi, phi_r_s, out_dtype and workspace as
 * for rfq_linear.  1 <= groups <= 128.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_linear_grouped(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi,
                                      int32_t phi_r_s, const int32_t *group_off, int32_t groups,
                                      const rfq_qtensor *wq, int64_t N, void *y, int32_t out_dtype,
                                      void *workspace, void *stream);

/* Exact re-encoding of an MXFP4 tensor as MXFP8 (every E2M1 value is an
 * E4M3 value): dst codes [rows][k] E4M3 bytes, dst scales = src scales.
 * src: fmt MXFP4; dst: fmt MXFP8, the same rows, k and scale layout; both
 * device, caller-owned.  Used for the weight of the W4A8 baseline and of
 * the FP4-to-FP8 RFQ (rfq_quantize_act_expand writes the activation's in
 * the quantizer's own pass).
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED (other formats), RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_convert(const rfq_qtensor *src, rfq_qtensor *dst, void *stream);

/* Checked mode for inputs: the quantizers and GEMMs take finite bf16 inputs
 * (non-finite ones give unspecified codes but never a fault); a caller that
 * cannot vouch for X runs this check first.  It scans the bf16 matrix
 * x [rows][k] (device, 16-byte aligned, k % 8 == 0) and, if any element is
 * Inf or NaN, records RFQ_ERR_NONFINITE in `workspace` (the GEMM workspace,
 * rfq_linear_workspace_bytes() bytes), where rfq_workspace_status reports
 * it.  Asynchronous on `stream`; one read of x.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT, RFQ_ERR_CUDA,
 * RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_check_finite(const void *x_bf16, int64_t rows, int64_t k, void *workspace, void *stream);

/* Synchronizes `stream` and returns the device status left in a workspace by
 * earlier calls (RFQ_OK, RFQ_ERR_TIMEOUT, RFQ_ERR_SHAPE for group offsets
 * that break rfq_linear_grouped's contract, or RFQ_ERR_NONFINITE from
 * rfq_check_finite); clears it when `clear` != 0. */
RFQ_API rfq_status rfq_workspace_status(void *workspace, int32_t clear, void *stream);

/* Measurement of the ceiling the RFQ GEMM is held against: the dense
 * block-scaled FP4 tensor rate of this GPU (the kind::mxf4 MMA that carries
 * both products of Algorithm 1 / Eq. rfq), with MMAs alone.  Every SM
 * (cta_pair = 0: 128 x 256 x 64 MMAs, one CTA per SM) or every CTA pair
 * (cta_pair = 1: 256 x 256 x 64 cta_group::2 MMAs, the RFQ GEMM's form)
 * issues `iters` back-to-back MMAs from one shared-memory tile of
 * pseudo-random E2M1 codes (scales 2^0) into one TMEM accumulator; no
 * copies, scale writes or epilogue.  Time the launch on `stream` with
 * events; *flop_per_launch (host) receives its MMA work, 2 M N K per MMA
 * summed over the grid.  workspace: as for rfq_linear (a bounded final wait
 * that runs out records RFQ_ERR_TIMEOUT there).  iters in [1, 2^24].
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_fp4_mma_peak(int32_t cta_pair, int64_t iters, void *workspace, double *flop_per_launch,
                                    void *stream);

/* RFQ GEMM with the FP4-to-FP8 residual at two rates (Sec. 4.2's FP4-to-FP8
 * pathway with the Sec. 3.2.1 format; Algorithm 1, Eq. rfq):
 *     Y = X~ W~ + phi X^ W~
 * with the main product X~ W~ on the FP4 tensor path (E2M1 x E2M1) and the
 * residual product X^ W~ on the FP8 one (E4M3 x E2M1), into one fp32
 * accumulator per output tile.  xq: X~, MXFP4 [M x K]; xr: X^, MXFP8 [M x K]
 * (rfq_quantize_act with an MXFP8 residual writes both); wq: W~, MXFP4
 * [N x K]: the kernel reads its packed codes once per k-stage and expands
 * them in shared memory to the one-byte-per-code form the residual MMAs
 * read (no second copy of W~ in memory).
 * Every operand with RFQ_SCALE_MMA scales; K % 128 == 0, N % 16 == 0,
 * M >= 0 (CTA pairs at every M).  phi, phi_r_s, y, out_dtype, workspace: as
 * for rfq_linear.  rfq_linear multiplies the same RFQ with X~ and W~
 * re-encoded as E4M3 (rfq_convert), both products then at the FP8 rate.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_UNSUPPORTED, RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_linear_mixed(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi,
                                    int32_t phi_r_s, const rfq_qtensor *wq, void *y, int32_t out_dtype,
                                    void *workspace, void *stream);

/* Measurement of where the RFQ GEMM's tensor pipe idles: rfq_linear
 * (Algorithm 1, Eq. rfq) for MXFP4 operands with a residual and no phi,
 * M > 128 (the CTA-pair kernel), in a build of that kernel whose MMA-issuing
 * thread (one per CTA pair) counts, from its first wait to its final drain:
 * SM clock cycles, wall-clock nanoseconds, cycles waiting for a drained
 * accumulator, for a stage's operand copies and for a stage's scale words,
 * stages and tiles.  The sums over all pairs are added to the workspace's
 * 64-bit words 4..11 (bytes 32..95) in that order, with the number of pairs
 * in word 10: zero them before the call and read them after the stream has
 * synchronized.  Y is computed as by rfq_linear; the counters cost a few
 * instructions per stage, so time rfq_linear, not this call.
 * Errors: those of rfq_linear; RFQ_ERR_UNSUPPORTED for other operand forms. */
RFQ_API rfq_status rfq_linear_profile(const rfq_qtensor *xq, const rfq_qtensor *xr, const rfq_qtensor *wq, void *y,
                                      int32_t out_dtype, void *workspace, void *stream);

/* The debug build (librfq_debug.so, compiled with -DRFQ_DEBUG_BOUNDS): the
 * activation and weight quantizers and the CTA-pair GEMM check the index of
 * every direct global store against its buffer's extent (codes, scales, the
 * fused quantizer's ring, the grouped GEMM's row stores); an out-of-range
 * store is skipped and the source line of the first one is recorded.  This
 * call synchronizes the device and reports it: RFQ_OK (none, *line = 0) or
 * RFQ_ERR_SHAPE with *line set; clear != 0 resets the records.  The normal
 * build has no checks and returns RFQ_ERR_UNSUPPORTED.  The paper has no
 * counterpart: a debugging aid of this library.
 * Errors: RFQ_ERR_INVALID_ARG (line NULL), RFQ_ERR_CUDA. */
RFQ_API rfq_status rfq_debug_bounds(int32_t *line, int32_t clear);

/* Allocation-free variant of rfq_linear.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory, such as
 * a serving loop that must not stall the device on cudaMalloc, a plug-in
 * whose host program owns every device buffer, or a runtime with no device
 * allocator of its own.  It takes the same arguments as rfq_linear except
 * the workspace and allocates nothing: no cudaMalloc, no cudaFree, no
 * allocating library routine.
 *
 * The GEMM's workspace (its status word) lives instead in a fixed 256-byte
 * __device__ array inside the library; every GPU that loads the library
 * holds it until the process exits.  If the GEMM ever needed more workspace
 * than 256 bytes the call would return RFQ_ERR_SHAPE; every size rfq_linear
 * accepts fits today.
 *
 * The first call on each device looks up the array's device address with
 * that device current; make that first call before any stream capture.  The
 * address is kept for the life of the process: a cudaDeviceReset reloads
 * the library's device code and makes it stale, so a caller of this entry
 * point does not reset the device.  A call passes rfq_linear's argument
 * checks first (a rejected call, or one with M == 0 or N == 0, leaves the
 * array untouched), then clears the array on `stream` before the GEMM runs,
 * because all calls share it and it keeps what the last call left.  Calls
 * that overlap on the GPU (other streams, other host threads) race on the
 * array.  A
 * timeout of a bounded wait is not reported by this variant (use rfq_linear
 * with a workspace to read it); Y is then left unwritten.
 * Errors: those of rfq_linear, and RFQ_ERR_SHAPE as above. */
RFQ_API rfq_status rfq_linear_noalloc(const rfq_qtensor *xq, const rfq_qtensor *xr, const uint8_t *phi,
                                      int32_t phi_r_s, const rfq_qtensor *wq, void *y, int32_t out_dtype,
                                      void *stream);

/* Dequantization x = code value * scale (Sec. 3.2 Eq. 4; Sec. 3.3 V_i) of a
 * quantized matrix (MXFP4 or HiF4) into device out[rows][k], fp32
 * (RFQ_OUT_F32) or bf16 (RFQ_OUT_BF16).  Every HiF4 value is exact in bf16;
 * MXFP4 values are exact in bf16 except below bf16's normal range.
 * Errors: RFQ_ERR_INVALID_ARG, RFQ_ERR_SHAPE, RFQ_ERR_ALIGNMENT,
 * RFQ_ERR_CUDA, RFQ_ERR_DEVICE. */
RFQ_API rfq_status rfq_dequant(const rfq_qtensor *q, void *out, int32_t out_dtype, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* RFQ_H */
