/*
 * rfq_oracle.c -- plain, slow CPU oracle for Residual Fallback Quantization
 * (RFQ), "Activation Outliers Matter: Robust Recovery for Quantized
 * Multimodal LLMs" (arXiv 2608.26581).
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load this library.  The CUDA path shares
 * no code, header, table or helper with this file, and this file includes
 * nothing from the CUDA path.
 *
 * Everything is scalar C on fp64.  Each function names the passage of the
 * paper it follows.  The paper's GEMM notation is Z = X Y with X [P x R]
 * (activation) and Y [R x Q] (weight); here the activation is X [M x K], the
 * weight W [K x N] and the output Y [M x N] (P=M, R=K, Q=N).
 *
 * Readings taken where the paper is silent or ambiguous (each one is listed
 * in the design notes of the repository):
 *   R1  MX block scale: the OCP MX rule 2^(floor(log2 amax) - emax_elem) with
 *       emax_elem = 2 for E2M1 (Sec. 3.2 cites the OCP MX specification; the
 *       printed Eq. 3 omits the "- emax_elem" term).  The exponent is clamped
 *       to the E8M0 range [-127, 127]; amax = 0 gives the byte 0.
 *   R2  Element rounding: round to nearest, ties to even mantissa bit,
 *       saturating at +-6 (Eq. 2 says round-to-nearest only).
 *   R3  Sign of zero: a code keeps the sign bit of its input, so a negative
 *       value that rounds to zero is encoded as 0x8.
 *   R4  Packing: two 4-bit codes per byte, the lower K index in the low nibble.
 *   R5  phi: "all" (phi = 1 everywhere, Sec. 1: no threshold-based selection)
 *       or "amax" (phi(p,r) = 1 iff max |x| over the P_s x R_s tile > tau);
 *       the paper gives no formula for the indicator (Sec. 4.3).
 *   R6  HiF4 encoder (Sec. 3.3 gives only the decoder): the macro scale is the
 *       smallest UE6M2 value S with 7 S >= amax; every 4-element sub-group
 *       takes the smallest exponent t in {0,1,2} with amax_sub <= 1.75 2^t S;
 *       E1_8[g] = 1 iff a sub-group of group g needs t = 2, and
 *       E1_16[j] = max(t_j - E1_8[g], 0); elements round to nearest k/4
 *       (k = 0..7), ties to even k, saturating at k = 7.
 *   R7  HiF4 metadata word: bits [7:0] UE6M2 (E in [7:2], M in [1:0]),
 *       bits [15:8] E1_8 (bit g = group g), bits [31:16] E1_16 (bit j =
 *       sub-group j).
 *   R8  The residual pathway uses the same 4-bit format as the main one
 *       (Sec. 4.3, Eq. for the re-quantized residual); the FP4-to-FP8
 *       variant named in Sec. 4.2 re-quantizes the residual of an MXFP4 main
 *       pathway in MXFP8 E4M3 (reading R12).
 *   R11 MXFP8 E4M3 (Sec. 3.2.1): the OCP E4M3 element, Eq. 1 with 4
 *       exponent bits, 3 mantissa bits and bias 7, exponent field 0
 *       subnormal, no infinities, S.1111.111 = NaN, largest finite 448; block
 *       scale 2^(floor(log2 amax) - 8) (emax_elem = 8, as R1); elements round
 *       to nearest, ties to even mantissa, saturating at +-448; a code keeps
 *       the sign of its input (as R3); one byte per element.
 *   R12 FP8 residual pathway (Sec. 4.2 names an FP4-to-FP8 pathway without
 *       defining it): X~ = Q_MXFP4(X) and X^ = Q_MXFP8(X - X~), both with
 *       32-element blocks along K; the GEMM multiplies X^ by the same W~.
 *
 * Parity status: the MXFP4 encoder (R1-R4), the residual, phi = "all" and the
 * GEMM are pinned by the tests in tests/test_oracle_*.py against the format
 * definitions.  The HiF4 *decoder* (Sec. 3.3) and its format properties are
 * pinned; the HiF4 *encoder choice* (R6) and the phi = "amax" criterion (R5)
 * are readings of the paper with no printed value to check against:
 * parity unpinned for those two choices (their internal consistency is tested).
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stdlib.h>

#define RFQ_O_FMT_MXFP4 0
#define RFQ_O_FMT_HIF4 1
#define RFQ_O_FMT_MXFP8 2

#define RFQ_O_PHI_NONE 0
#define RFQ_O_PHI_ALL 1
#define RFQ_O_PHI_AMAX 2

/* ------------------------------------------------------------------ */
/* bf16 input                                                          */
/* ------------------------------------------------------------------ */

/* A bf16 number is the upper half of an IEEE binary32; widening is exact. */
double rfq_o_bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* ------------------------------------------------------------------ */
/* E2M1 element (MXFP4), Sec. 3.1 Eq. 1 and Sec. 3.2.2                 */
/* ------------------------------------------------------------------ */

/* Eq. 1 with E = 2 exponent bits, M = 1 mantissa bit and bias 1 (the OCP
 * E2M1 layout 1-2-1 named in Sec. 3.2.2).  Exponent field 0 is subnormal:
 * 2^(1 - bias) * (0 + m/2).  E2M1 has no Inf or NaN. */
double rfq_o_e2m1_decode(int code)
{
    int s = (code >> 3) & 1;
    int e = (code >> 1) & 3;
    int m = code & 1;
    const int bias = 1;
    double mag;
    if (e == 0)
        mag = ldexp((double)m / 2.0, 1 - bias);
    else
        mag = ldexp(1.0 + (double)m / 2.0, e - bias);
    return s ? -mag : mag;
}

/* Round y to the E2M1 grid (reading R2, R3): floating-point rounding with a
 * 1-bit mantissa and round-half-even, saturating at the largest finite
 * magnitude 6.  Returns the 4-bit code. */
int rfq_o_e2m1_encode(double y)
{
    int s = signbit(y) ? 1 : 0;
    double a = fabs(y);
    int code;
    if (a < 1.0) {
        /* subnormal binade: spacing 2^(1-bias) / 2 = 0.5 */
        double q = nearbyint(a * 2.0); /* 0, 1 or 2 halves */
        code = (int)q;                 /* 0 -> 0.0, 1 -> 0.5, 2 -> 1.0 (= code 2) */
    } else {
        int ex;
        frexp(a, &ex);        /* a = f 2^ex, f in [0.5, 1) */
        int e = ex - 1;       /* floor(log2 a) */
        if (e > 2) {
            code = 7;         /* |y| >= 8: saturate to 6 */
        } else {
            double m = ldexp(a, -e) - 1.0;     /* mantissa fraction in [0,1) */
            double q = nearbyint(m * 2.0);     /* 0, 1 or 2 */
            int ef = e + 1;                    /* biased exponent field */
            if (q >= 2.0) { ef += 1; q = 0.0; }
            if (ef > 3) { ef = 3; q = 1.0; }   /* rounded past 6: saturate */
            code = (ef << 1) | (int)q;
        }
    }
    return (s << 3) | code;
}

/* ------------------------------------------------------------------ */
/* MX block scale, Sec. 3.2 Eq. 3 (reading R1)                         */
/* ------------------------------------------------------------------ */

/* Shared exponent of one block: floor(log2 amax) - 2, clamped to the E8M0
 * range [-127, 127]; amax = 0 gives -127 (scale byte 0). */
int rfq_o_mx_scale_exp(double amax)
{
    if (!(amax > 0.0))
        return -127;
    int ex;
    frexp(amax, &ex);
    int e = (ex - 1) - 2;
    if (e < -127) e = -127;
    if (e > 127) e = 127;
    return e;
}

/* Quantize one block of n (<= 32) values (Sec. 3.2 Eqs. 3-4).  Writes n
 * codes and returns the E8M0 byte. */
static int mx_quantize_block(const double *x, int n, uint8_t *codes)
{
    double amax = 0.0;
    for (int i = 0; i < n; i++)
        if (fabs(x[i]) > amax) amax = fabs(x[i]);
    int e = rfq_o_mx_scale_exp(amax);
    for (int i = 0; i < n; i++)
        codes[i] = (uint8_t)rfq_o_e2m1_encode(ldexp(x[i], -e));
    return e + 127;
}

static void put_nibble(uint8_t *row, int64_t k, int code)
{
    if (k & 1)
        row[k >> 1] = (uint8_t)((row[k >> 1] & 0x0F) | (code << 4));
    else
        row[k >> 1] = (uint8_t)((row[k >> 1] & 0xF0) | (code & 0xF));
}

static int get_nibble(const uint8_t *row, int64_t k)
{
    return (k & 1) ? (row[k >> 1] >> 4) & 0xF : row[k >> 1] & 0xF;
}

/* MXFP4 quantization of a [rows x k] fp64 matrix along k in blocks of 32.
 * codes: [rows][k/2] bytes (reading R4); scales: [rows][k/32] E8M0 bytes. */
void rfq_o_mxfp4_quantize(const double *x, int64_t rows, int64_t k,
                          uint8_t *codes, uint8_t *scales)
{
    const int B = 32;
    for (int64_t r = 0; r < rows; r++) {
        const double *xr = x + r * k;
        uint8_t *cr = codes + r * (k / 2);
        for (int64_t j = 0; j < k / B; j++) {
            uint8_t c[32];
            scales[r * (k / B) + j] = (uint8_t)mx_quantize_block(xr + j * B, B, c);
            for (int i = 0; i < B; i++) put_nibble(cr, j * B + i, c[i]);
        }
    }
}

/* x~ = code value * 2^(byte - 127) (Sec. 3.2 Eq. 4 inverted). */
void rfq_o_mxfp4_dequant(const uint8_t *codes, const uint8_t *scales,
                         int64_t rows, int64_t k, double *out)
{
    for (int64_t r = 0; r < rows; r++)
        for (int64_t i = 0; i < k; i++) {
            int code = get_nibble(codes + r * (k / 2), i);
            int byte = scales[r * (k / 32) + i / 32];
            out[r * k + i] = ldexp(rfq_o_e2m1_decode(code), byte - 127);
        }
}

/* ------------------------------------------------------------------ */
/* E4M3 element and MXFP8, Sec. 3.1 Eq. 1 and Sec. 3.2.1 (reading R11) */
/* ------------------------------------------------------------------ */

/* Eq. 1 with E = 4 exponent bits, M = 3 mantissa bits and bias 7.  Exponent
 * field 0 is subnormal: 2^(1 - bias) (0 + m/8).  The two codes S.1111.111
 * are NaN; there is no infinity. */
double rfq_o_e4m3_decode(int code)
{
    int s = (code >> 7) & 1;
    int e = (code >> 3) & 15;
    int m = code & 7;
    const int bias = 7;
    double mag;
    if (e == 15 && m == 7)
        return NAN;
    if (e == 0)
        mag = ldexp((double)m / 8.0, 1 - bias);
    else
        mag = ldexp(1.0 + (double)m / 8.0, e - bias);
    return s ? -mag : mag;
}

/* Round y to the E4M3 grid (reading R11): a 3-bit mantissa with
 * round-half-even, subnormal spacing 2^-9, saturating at 448.  Returns the
 * 8-bit code. */
int rfq_o_e4m3_encode(double y)
{
    int s = signbit(y) ? 1 : 0;
    double a = fabs(y);
    int code;
    if (a < ldexp(1.0, -6)) {
        /* subnormal binade: spacing 2^-9; 8 steps reach the first normal */
        double q = nearbyint(ldexp(a, 9)); /* 0..8 */
        code = (int)q;                     /* q = 8 is the code of 2^-6 */
    } else {
        int ex;
        frexp(a, &ex);
        int e = ex - 1;                    /* floor(log2 a) >= -6 */
        if (e > 8) {
            code = 0x7E;                   /* |y| >= 512: saturate to 448 */
        } else {
            double m = ldexp(a, -e) - 1.0; /* fraction in [0, 1) */
            double q = nearbyint(m * 8.0); /* 0..8 */
            int ef = e + 7;
            if (q >= 8.0) { ef += 1; q = 0.0; }
            if (ef > 15 || (ef == 15 && q > 6.0)) { ef = 15; q = 6.0; } /* past 448 */
            code = (ef << 3) | (int)q;
        }
    }
    return (s << 7) | code;
}

/* Shared exponent of one MXFP8 block: floor(log2 amax) - 8 (emax of E4M3),
 * clamped to [-127, 127]; amax = 0 gives -127 (scale byte 0). */
int rfq_o_mx8_scale_exp(double amax)
{
    if (!(amax > 0.0))
        return -127;
    int ex;
    frexp(amax, &ex);
    int e = (ex - 1) - 8;
    if (e < -127) e = -127;
    if (e > 127) e = 127;
    return e;
}

/* MXFP8 quantization of [rows x k] along k in blocks of 32 (Sec. 3.2 Eqs.
 * 3-4 with the E4M3 element).  codes: [rows][k] bytes; scales: [rows][k/32]. */
void rfq_o_mxfp8_quantize(const double *x, int64_t rows, int64_t k,
                          uint8_t *codes, uint8_t *scales)
{
    const int B = 32;
    for (int64_t r = 0; r < rows; r++)
        for (int64_t j = 0; j < k / B; j++) {
            const double *xb = x + r * k + j * B;
            double amax = 0.0;
            for (int i = 0; i < B; i++)
                if (fabs(xb[i]) > amax) amax = fabs(xb[i]);
            int e = rfq_o_mx8_scale_exp(amax);
            for (int i = 0; i < B; i++)
                codes[r * k + j * B + i] = (uint8_t)rfq_o_e4m3_encode(ldexp(xb[i], -e));
            scales[r * (k / B) + j] = (uint8_t)(e + 127);
        }
}

void rfq_o_mxfp8_dequant(const uint8_t *codes, const uint8_t *scales,
                         int64_t rows, int64_t k, double *out)
{
    for (int64_t r = 0; r < rows; r++)
        for (int64_t i = 0; i < k; i++)
            out[r * k + i] = ldexp(rfq_o_e4m3_decode(codes[r * k + i]), scales[r * (k / 32) + i / 32] - 127);
}

/* ------------------------------------------------------------------ */
/* HiF4, Sec. 3.3                                                      */
/* ------------------------------------------------------------------ */

/* Unsigned E6M2 with exponent bias 48: 2^(E - 48) (1 + M/4). */
double rfq_o_ue6m2_decode(int byte)
{
    int E = (byte >> 2) & 63;
    int M = byte & 3;
    return ldexp(1.0 + (double)M / 4.0, E - 48);
}

/* S1P2 sign-magnitude element: sign, 1 integer bit, 2 fraction bits. */
double rfq_o_s1p2_decode(int code)
{
    double mag = (double)(code & 7) / 4.0;
    return (code & 8) ? -mag : mag;
}

/* Sec. 3.3: V_i = S_macro 2^(E1_8[ceil(i/8)] + E1_16[ceil(i/4)]) S1P2_i,
 * i = 1..64 (here 0-based: group i/8, sub-group i/4).  Metadata: R7. */
double rfq_o_hif4_decode(uint32_t meta, int i, int code)
{
    double S = rfq_o_ue6m2_decode((int)(meta & 0xFF));
    int e18 = (int)((meta >> 8) >> (i / 8)) & 1;
    int e116 = (int)((meta >> 16) >> (i / 4)) & 1;
    return S * ldexp(1.0, e18 + e116) * rfq_o_s1p2_decode(code);
}

/* Reading R6 for one 64-element block; returns the metadata word. */
static uint32_t hif4_quantize_block(const double *x, uint8_t *codes)
{
    double amax = 0.0;
    for (int i = 0; i < 64; i++)
        if (fabs(x[i]) > amax) amax = fabs(x[i]);
    if (amax == 0.0) {
        for (int i = 0; i < 64; i++) codes[i] = signbit(x[i]) ? 8 : 0;
        return 0;
    }
    /* macro scale: smallest UE6M2 value S with 7 S >= amax (UE6M2 values
     * increase with the byte), else the largest one */
    int sbyte = 255;
    for (int b = 0; b < 256; b++)
        if (7.0 * rfq_o_ue6m2_decode(b) >= amax) { sbyte = b; break; }
    double S = rfq_o_ue6m2_decode(sbyte);
    int t[16];
    for (int j = 0; j < 16; j++) {
        double a = 0.0;
        for (int i = 4 * j; i < 4 * j + 4; i++)
            if (fabs(x[i]) > a) a = fabs(x[i]);
        t[j] = 2;
        for (int tt = 0; tt <= 2; tt++)
            if (a <= 1.75 * ldexp(S, tt)) { t[j] = tt; break; }
    }
    uint32_t e18 = 0, e116 = 0;
    for (int g = 0; g < 8; g++) {
        int hi = (t[2 * g] == 2 || t[2 * g + 1] == 2);
        if (hi) e18 |= 1u << g;
        for (int j = 2 * g; j < 2 * g + 2; j++) {
            int v = t[j] - hi;
            if (v > 0) e116 |= 1u << j;
        }
    }
    for (int i = 0; i < 64; i++) {
        int ex = (int)((e18 >> (i / 8)) & 1) + (int)((e116 >> (i / 4)) & 1);
        double step = 0.25 * ldexp(S, ex);
        double q = nearbyint(fabs(x[i]) / step); /* ties to even k */
        int k = q > 7.0 ? 7 : (int)q;
        codes[i] = (uint8_t)((signbit(x[i]) ? 8 : 0) | k);
    }
    return (uint32_t)sbyte | (e18 << 8) | (e116 << 16);
}

/* HiF4 quantization of [rows x k] (k % 64 == 0) along k.
 * codes: [rows][k/2] bytes (R4); meta: [rows][k/64] words (R7). */
void rfq_o_hif4_quantize(const double *x, int64_t rows, int64_t k,
                         uint8_t *codes, uint32_t *meta)
{
    for (int64_t r = 0; r < rows; r++) {
        uint8_t *cr = codes + r * (k / 2);
        for (int64_t j = 0; j < k / 64; j++) {
            uint8_t c[64];
            meta[r * (k / 64) + j] = hif4_quantize_block(x + r * k + j * 64, c);
            for (int i = 0; i < 64; i++) put_nibble(cr, j * 64 + i, c[i]);
        }
    }
}

void rfq_o_hif4_dequant(const uint8_t *codes, const uint32_t *meta,
                        int64_t rows, int64_t k, double *out)
{
    for (int64_t r = 0; r < rows; r++)
        for (int64_t i = 0; i < k; i++) {
            int code = get_nibble(codes + r * (k / 2), i);
            out[r * k + i] = rfq_o_hif4_decode(meta[r * (k / 64) + i / 64], (int)(i % 64), code);
        }
}

/* ------------------------------------------------------------------ */
/* Format dispatch                                                     */
/* ------------------------------------------------------------------ */

static int64_t scale_count(int fmt, int64_t k)
{
    return fmt == RFQ_O_FMT_HIF4 ? k / 64 : k / 32;
}

static void quantize_fmt(int fmt, const double *x, int64_t rows, int64_t k,
                         uint8_t *codes, void *scales)
{
    if (fmt == RFQ_O_FMT_HIF4)
        rfq_o_hif4_quantize(x, rows, k, codes, (uint32_t *)scales);
    else if (fmt == RFQ_O_FMT_MXFP8)
        rfq_o_mxfp8_quantize(x, rows, k, codes, (uint8_t *)scales);
    else
        rfq_o_mxfp4_quantize(x, rows, k, codes, (uint8_t *)scales);
}

void rfq_o_dequant(int fmt, const uint8_t *codes, const void *scales,
                   int64_t rows, int64_t k, double *out)
{
    if (fmt == RFQ_O_FMT_HIF4)
        rfq_o_hif4_dequant(codes, (const uint32_t *)scales, rows, k, out);
    else if (fmt == RFQ_O_FMT_MXFP8)
        rfq_o_mxfp8_dequant(codes, (const uint8_t *)scales, rows, k, out);
    else
        rfq_o_mxfp4_dequant(codes, (const uint8_t *)scales, rows, k, out);
}


/* ------------------------------------------------------------------ */
/* RFQ activation decomposition, Sec. 4.3 and Algorithm 1              */
/* ------------------------------------------------------------------ */

/* Fallback indicator phi(p, r) over tiles of p_s rows x r_s columns
 * (reading R5).  phi: [ceil(M/p_s)][ceil(K/r_s)] bytes. */
void rfq_o_phi(const double *x, int64_t M, int64_t K, int mode, double tau,
               int64_t p_s, int64_t r_s, uint8_t *phi)
{
    int64_t np = (M + p_s - 1) / p_s, nr = (K + r_s - 1) / r_s;
    for (int64_t p = 0; p < np; p++)
        for (int64_t r = 0; r < nr; r++) {
            uint8_t v;
            if (mode == RFQ_O_PHI_ALL) {
                v = 1;
            } else if (mode == RFQ_O_PHI_NONE) {
                v = 0;
            } else {
                double a = 0.0;
                for (int64_t m = p * p_s; m < M && m < (p + 1) * p_s; m++)
                    for (int64_t c = r * r_s; c < K && c < (r + 1) * r_s; c++)
                        if (fabs(x[m * K + c]) > a) a = fabs(x[m * K + c]);
                v = a > tau ? 1 : 0;
            }
            phi[p * nr + r] = v;
        }
}

/* RFQ decomposition of the activation X (bf16 [M x K]):
 *   X~ = Q(X)                      (Sec. 4.3, first quantization)
 *   dX = X - X~  where phi = 1     (Sec. 4.3, residual)
 *   X^ = Q(dX)                     (Sec. 4.3, re-quantized residual, R8)
 * Blocks with phi = 0 get all-zero residual codes and scale words.
 * main/res codes: [M][K/2]; scales: [M][K/32] bytes (MXFP4) or [M][K/64]
 * words (HiF4); phi: [ceil(M/p_s)][ceil(K/r_s)], may be NULL.
 * rc/rs may be NULL when mode is RFQ_O_PHI_NONE. */
void rfq_o_quantize_act2(const uint16_t *x_bf16, int64_t M, int64_t K, int fmt,
                         int res_fmt, int mode, double tau, int64_t p_s, int64_t r_s,
                         uint8_t *mc, void *ms, uint8_t *rc, void *rs,
                         uint8_t *phi_out)
{
    double *x = (double *)malloc(sizeof(double) * M * K);
    double *xt = (double *)malloc(sizeof(double) * M * K);
    int64_t np = (M + p_s - 1) / p_s, nr = (K + r_s - 1) / r_s;
    uint8_t *phi = (uint8_t *)malloc((size_t)(np * nr));
    for (int64_t i = 0; i < M * K; i++) x[i] = rfq_o_bf16_to_double(x_bf16[i]);
    rfq_o_phi(x, M, K, mode, tau, p_s, r_s, phi);
    quantize_fmt(fmt, x, M, K, mc, ms);
    if (rc && rs) {
        rfq_o_dequant(fmt, mc, ms, M, K, xt);
        for (int64_t m = 0; m < M; m++)
            for (int64_t c = 0; c < K; c++) {
                int on = phi[(m / p_s) * nr + c / r_s];
                /* exact in fp64: both operands have few significant bits */
                xt[m * K + c] = on ? x[m * K + c] - xt[m * K + c] : 0.0;
            }
        quantize_fmt(res_fmt, xt, M, K, rc, rs);
        /* phi = 0 blocks: codes and scale words are written as zero */
        int64_t bs = res_fmt == RFQ_O_FMT_HIF4 ? 64 : 32;
        for (int64_t m = 0; m < M; m++)
            for (int64_t j = 0; j < scale_count(res_fmt, K); j++) {
                if (phi[(m / p_s) * nr + (j * bs) / r_s]) continue;
                for (int64_t c = j * bs; c < (j + 1) * bs; c++) {
                    if (res_fmt == RFQ_O_FMT_MXFP8) rc[m * K + c] = 0;
                    else put_nibble(rc + m * (K / 2), c, 0);
                }
                if (res_fmt == RFQ_O_FMT_HIF4) ((uint32_t *)rs)[m * (K / 64) + j] = 0;
                else ((uint8_t *)rs)[m * (K / 32) + j] = 0;
            }
    }
    if (phi_out) memcpy(phi_out, phi, (size_t)(np * nr));
    free(phi);
    free(xt);
    free(x);
}

/* The decomposition with one format for both pathways (R8). */
void rfq_o_quantize_act(const uint16_t *x_bf16, int64_t M, int64_t K, int fmt,
                        int mode, double tau, int64_t p_s, int64_t r_s,
                        uint8_t *mc, void *ms, uint8_t *rc, void *rs,
                        uint8_t *phi_out)
{
    rfq_o_quantize_act2(x_bf16, M, K, fmt, fmt, mode, tau, p_s, r_s, mc, ms, rc, rs, phi_out);
}

/* Weight quantization Y~ = Q(Y) (Sec. 4.3; Algorithm 1): W is bf16 [K x N]
 * row-major; blocks run along K for every column n, so the result is stored
 * K-major: codes [N][K/2], scales [N][K/32] bytes or [N][K/64] words. */
void rfq_o_quantize_weight(const uint16_t *w_bf16, int64_t K, int64_t N, int fmt,
                           uint8_t *codes, void *scales)
{
    double *wt = (double *)malloc(sizeof(double) * K * N);
    for (int64_t n = 0; n < N; n++)
        for (int64_t k = 0; k < K; k++)
            wt[n * K + k] = rfq_o_bf16_to_double(w_bf16[k * N + n]);
    quantize_fmt(fmt, wt, N, K, codes, scales);
    free(wt);
}

/* ------------------------------------------------------------------ */
/* RFQ GEMM, Algorithm 1 and Eq. (rfq)                                 */
/* ------------------------------------------------------------------ */

/* Z[m][n] = sum_k X~[m][k] Y~[k][n] + sum_k phi X^[m][k] Y~[k][n],
 * accumulated in fp64 in the order of Algorithm 1 (for each k: base term,
 * then the correction term).  The residual codes are zero where phi = 0,
 * so phi enters through them.  xr_codes may be NULL (plain W4A4).
 * W~ is K-major: codes [N][K/2].  Output Y: [M][N] doubles. */
void rfq_o_linear2(int fmt, int res_fmt, int w_fmt,
                   const uint8_t *xm_codes, const void *xm_scales,
                   const uint8_t *xr_codes, const void *xr_scales,
                   int64_t M, int64_t K, const uint8_t *w_codes,
                   const void *w_scales, int64_t N, double *Y)
{
    double *xm = (double *)malloc(sizeof(double) * M * K);
    double *xr = (double *)malloc(sizeof(double) * M * K);
    double *w = (double *)malloc(sizeof(double) * N * K);
    rfq_o_dequant(fmt, xm_codes, xm_scales, M, K, xm);
    if (xr_codes)
        rfq_o_dequant(res_fmt, xr_codes, xr_scales, M, K, xr);
    else
        memset(xr, 0, sizeof(double) * M * K);
    rfq_o_dequant(w_fmt, w_codes, w_scales, N, K, w);
    for (int64_t m = 0; m < M; m++)
        for (int64_t n = 0; n < N; n++) {
            double z = 0.0;
            for (int64_t k = 0; k < K; k++) {
                z += xm[m * K + k] * w[n * K + k];
                z += xr[m * K + k] * w[n * K + k];
            }
            Y[m * N + n] = z;
        }
    free(w);
    free(xr);
    free(xm);
}

/* The GEMM with one format for every operand. */
void rfq_o_linear(int fmt, const uint8_t *xm_codes, const void *xm_scales,
                  const uint8_t *xr_codes, const void *xr_scales,
                  int64_t M, int64_t K, const uint8_t *w_codes,
                  const void *w_scales, int64_t N, double *Y)
{
    rfq_o_linear2(fmt, fmt, fmt, xm_codes, xm_scales, xr_codes, xr_scales, M, K, w_codes, w_scales, N, Y);
}
