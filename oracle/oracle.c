/*
 * oracle.c -- plain CPU oracle for the space-filling-curve (SFC) GEMM.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file: only the tests, the smoke check and the CPU-baseline leg of
 * the benchmark use it.  It shares no code with the CUDA library.
 *
 * Two parts, each written from the paper's statement of the method:
 *
 *  1. oracle_gilbert_order -- the generalized Hilbert ("Gilbert") curve over an
 *     Mt x Nt grid of output tiles (Sec. II-B, Fig. 2; created once per shape as
 *     create_sfc_map in Listing 1).  The paper prints no curve algorithm and
 *     cites the generalized-Hilbert construction for arbitrary rectangles; this
 *     is a recursive walk written from that construction's idea:
 *       - a region is an origin plus two orthogonal axis vectors, a "major" one
 *         (the direction the walk makes progress along) and a "minor" one;
 *       - a region one cell thick is walked straight along its long side;
 *       - a region much longer than wide (2|a| > 3|b|) is cut across its major
 *         axis into two halves, the first half even-sized when possible, and
 *         both halves are walked with the same orientation;
 *       - otherwise it is cut into three: a corner block spanning the first
 *         (even-sized when possible) part of the minor axis and the first half
 *         of the major axis, walked with the two axes exchanged; the strip that
 *         spans the whole major axis over the rest of the minor axis; and the
 *         remaining corner block, walked backwards with exchanged, negated axes
 *         so the walk ends at the far end of the major axis.
 *     Output convention: out[s] = tm * Nt + tn for curve position s, the walk
 *     starts at tile (0,0).  x runs along tn (columns), y along tm (rows).
 *     Top-level orientation: the major axis is the longer grid side, except
 *     when the longer side is odd and the shorter even; then the walk runs
 *     along the even side, because a path from (0,0) to the far corner of an
 *     odd side of an odd x even grid cannot be edge-adjacent throughout (the
 *     two ends would share a chessboard colour while the cell count is even).
 *
 *  2. oracle_gemm_* -- C = A * B as its plain definition (Sec. II-A: A is M x K,
 *     B is K x N, C is M x N; Listing 1 zeroes C and accumulates every K block
 *     into it).  Inputs are bf16 bit patterns, widened exactly to double; the
 *     sum over k runs in double, i-k-j loop order, OpenMP over rows only.  The
 *     K split of the communication-avoiding variant (Sec. II-C/D) only regroups
 *     this sum, so it has no separate oracle; oracle_gemm_sub_f64 takes a k
 *     range so one layer's partial product can be formed too.
 *
 *  3. oracle_gemm_affine_f64 -- an extension beyond the paper (which zeroes C
 *     and takes B as K x N): the BLAS-style C = A B + beta * C_in + bias[j],
 *     with B given either K x N or transposed (N x K, a linear layer's weight
 *     matrix).  It is written independently of part 2: one dot product per
 *     output element (j-k loop order), then the two affine terms, in double.
 *
 *  4. oracle_decode_f8 / oracle_gemm_f8_f64 -- the same products for 8-bit
 *     float inputs (the method is independent of the data type, Sec. III):
 *     each byte is decoded to its exact value from the format's definition
 *     (e4m3: sign, 4 exponent bits with bias 7, 3 mantissa bits, no
 *     infinities, S.1111.111 is NaN; e5m2: sign, 5 exponent bits with bias 15,
 *     2 mantissa bits, IEEE-style infinities and NaNs), then summed in double.
 *
 *  oracle_round_bf16 rounds a double to the nearest bf16 (ties to even) in a
 *  single step, used to compare bf16 outputs against the fp64 reference.
 */
#include <math.h>
#include <omp.h>
#include <stdint.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* 1. generalized Hilbert curve                                               */
/* ------------------------------------------------------------------------- */

typedef struct { int x, y; } vec2;

typedef struct {
    int32_t *out;   /* output permutation            */
    int64_t  count; /* cells emitted so far          */
    int64_t  limit; /* Mt * Nt, guards the writes    */
    int      nt;    /* grid width (tiles along x=tn) */
    int      bad;   /* set if the walk left the grid */
    int      mt;
} walk_state;

static int sign_of(int v) { return (v > 0) - (v < 0); }
static int length_of(vec2 v) { int s = v.x + v.y; return s < 0 ? -s : s; }
static vec2 unit_of(vec2 v) { vec2 u = { sign_of(v.x), sign_of(v.y) }; return u; }
static vec2 add(vec2 p, vec2 q) { vec2 r = { p.x + q.x, p.y + q.y }; return r; }
static vec2 sub(vec2 p, vec2 q) { vec2 r = { p.x - q.x, p.y - q.y }; return r; }
static vec2 neg(vec2 p) { vec2 r = { -p.x, -p.y }; return r; }
static vec2 halve(vec2 p) { vec2 r = { p.x / 2, p.y / 2 }; return r; }

static void emit(walk_state *st, vec2 cell)
{
    if (cell.x < 0 || cell.y < 0 || cell.x >= st->nt || cell.y >= st->mt ||
        st->count >= st->limit) {
        st->bad = 1;
        return;
    }
    st->out[st->count++] = (int32_t)(cell.y * st->nt + cell.x);
}

/* Walk the region with corner `o`, major vector `a`, minor vector `b`. */
static void walk_region(walk_state *st, vec2 o, vec2 a, vec2 b)
{
    int la = length_of(a), lb = length_of(b);
    vec2 ua = unit_of(a), ub = unit_of(b);

    if (lb == 1) {                       /* one cell thick: straight along a */
        for (int i = 0; i < la; ++i) { vec2 c = { o.x + i * ua.x, o.y + i * ua.y }; emit(st, c); }
        return;
    }
    if (la == 1) {                       /* one cell long: straight along b */
        for (int i = 0; i < lb; ++i) { vec2 c = { o.x + i * ub.x, o.y + i * ub.y }; emit(st, c); }
        return;
    }

    vec2 a_first = halve(a);             /* first part of the major axis */
    vec2 b_first = halve(b);             /* first part of the minor axis */

    if (2 * la > 3 * lb) {
        /* long region: two halves along the major axis, same orientation */
        if ((length_of(a_first) % 2) == 1 && la > 2) a_first = add(a_first, ua);
        walk_region(st, o, a_first, b);
        walk_region(st, add(o, a_first), sub(a, a_first), b);
        return;
    }

    /* three pieces: corner block, full-width strip, returning corner block */
    if ((length_of(b_first) % 2) == 1 && lb > 2) b_first = add(b_first, ub);
    vec2 a_rest = sub(a, a_first);
    vec2 b_rest = sub(b, b_first);

    walk_region(st, o, b_first, a_first);                 /* axes exchanged  */
    walk_region(st, add(o, b_first), a, b_rest);          /* strip across    */
    vec2 far = add(add(o, sub(a, ua)), sub(b_first, ub)); /* far top corner  */
    walk_region(st, far, neg(b_first), neg(a_rest));      /* back down       */
}

/* Fills out[0 .. Mt*Nt) with out[s] = tm*Nt + tn.  Returns 0 on success,
 * -1 for a bad argument, -2 if the walk did not cover the grid exactly. */
int oracle_gilbert_order(int Mt, int Nt, int32_t *out)
{
    if (Mt <= 0 || Nt <= 0 || out == NULL) return -1;
    walk_state st = { out, 0, (int64_t)Mt * Nt, Nt, 0, Mt };
    vec2 origin = { 0, 0 };
    vec2 along_x = { Nt, 0 }, along_y = { 0, Mt };

    int x_major = (Nt >= Mt);
    int longer = x_major ? Nt : Mt, shorter = x_major ? Mt : Nt;
    if ((longer % 2) == 1 && (shorter % 2) == 0) x_major = !x_major;  /* parity rule */

    if (x_major) walk_region(&st, origin, along_x, along_y);
    else         walk_region(&st, origin, along_y, along_x);

    if (st.bad || st.count != st.limit) return -2;
    return 0;
}

/* ------------------------------------------------------------------------- */
/* 2. GEMM, plain definition in double                                        */
/* ------------------------------------------------------------------------- */

/* bf16 bit pattern -> double, exact (bf16 is the top half of an fp32). */
static double widen_bf16(uint16_t bits)
{
    uint32_t w = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

/* C[i*ldc + j] = sum_k A[i*lda + k] * B[k*ldb + j], row-major, all M x N. */
void oracle_gemm_f64(int64_t M, int64_t N, int64_t K,
                     const uint16_t *A, int64_t lda,
                     const uint16_t *B, int64_t ldb,
                     double *C, int64_t ldc)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        double *c = C + i * ldc;
        for (int64_t j = 0; j < N; ++j) c[j] = 0.0;
        for (int64_t k = 0; k < K; ++k) {
            double a = widen_bf16(A[i * lda + k]);
            const uint16_t *b = B + k * ldb;
            for (int64_t j = 0; j < N; ++j) c[j] += a * widen_bf16(b[j]);
        }
    }
}

/* out[r*ncols + c] = sum_{k0 <= k < k1} A[rows[r]][k] * B[k][cols[c]].
 * Used for sampled rows/columns of large products and for one K layer's
 * partial product of the communication-avoiding split. */
void oracle_gemm_sub_f64(const int64_t *rows, int64_t nrows,
                         const int64_t *cols, int64_t ncols,
                         int64_t k0, int64_t k1,
                         const uint16_t *A, int64_t lda,
                         const uint16_t *B, int64_t ldb,
                         double *out)
{
    #pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < nrows; ++r) {
        double *o = out + r * ncols;
        for (int64_t c = 0; c < ncols; ++c) o[c] = 0.0;
        for (int64_t k = k0; k < k1; ++k) {
            double a = widen_bf16(A[rows[r] * lda + k]);
            const uint16_t *b = B + k * ldb;
            for (int64_t c = 0; c < ncols; ++c) o[c] += a * widen_bf16(b[cols[c]]);
        }
    }
}

/* ------------------------------------------------------------------------- */
/* 3. GEMM with a transposed-B option and the beta / bias epilogue            */
/* ------------------------------------------------------------------------- */

/* C[i*ldc + j] = sum_k A[i][k] * B(k, j) + beta * C_in[i*ldcin + j] + bias[j],
 * B(k, j) = B[k*ldb + j] (b_nk == 0) or B[j*ldb + k] (b_nk == 1).  C_in and
 * bias may be NULL (terms left out). */
void oracle_gemm_affine_f64(int64_t M, int64_t N, int64_t K,
                            const uint16_t *A, int64_t lda,
                            const uint16_t *B, int64_t ldb, int b_nk,
                            double beta, const double *C_in, int64_t ldcin,
                            const double *bias,
                            double *C, int64_t ldc)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        for (int64_t j = 0; j < N; ++j) {
            double dot = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                uint16_t b = b_nk ? B[j * ldb + k] : B[k * ldb + j];
                dot += widen_bf16(A[i * lda + k]) * widen_bf16(b);
            }
            if (C_in) dot += beta * C_in[i * ldcin + j];
            if (bias) dot += bias[j];
            C[i * ldc + j] = dot;
        }
    }
}

/* ------------------------------------------------------------------------- */
/* 4. 8-bit float inputs                                                      */
/* ------------------------------------------------------------------------- */

/* Exact value of an 8-bit float; fmt 1 = e4m3, 2 = e5m2. */
double oracle_decode_f8(uint8_t code, int fmt)
{
    int sign = code >> 7;
    int ebits = fmt == 1 ? 4 : 5;
    int mbits = 7 - ebits;
    int bias = fmt == 1 ? 7 : 15;
    int e = (code >> mbits) & ((1 << ebits) - 1);
    int m = code & ((1 << mbits) - 1);
    double v;
    if (fmt == 1 && e == 15 && m == 7) return NAN;
    if (fmt == 2 && e == 31) v = (m == 0) ? INFINITY : NAN;
    else if (e == 0) v = ldexp((double)m, 1 - bias - mbits);               /* subnormal */
    else v = ldexp((double)((1 << mbits) + m), e - bias - mbits);          /* normal    */
    return sign ? -v : v;
}

/* C[i*ldc + j] = sum_k A[i][k] * B(k, j) over 8-bit float inputs of format fmt,
 * B(k, j) = B[k*ldb + j] (b_nk == 0) or B[j*ldb + k] (b_nk == 1). */
void oracle_gemm_f8_f64(int64_t M, int64_t N, int64_t K,
                        const uint8_t *A, int64_t lda,
                        const uint8_t *B, int64_t ldb, int b_nk, int fmt,
                        double *C, int64_t ldc)
{
    double table[256];
    for (int c = 0; c < 256; ++c) table[c] = oracle_decode_f8((uint8_t)c, fmt);
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < M; ++i) {
        for (int64_t j = 0; j < N; ++j) {
            double dot = 0.0;
            for (int64_t k = 0; k < K; ++k) {
                uint8_t b = b_nk ? B[j * ldb + k] : B[k * ldb + j];
                dot += table[A[i * lda + k]] * table[b];
            }
            C[i * ldc + j] = dot;
        }
    }
}

/* ------------------------------------------------------------------------- */
/* rounding helper                                                            */
/* ------------------------------------------------------------------------- */

/* Nearest bf16 to v, ties to even, in one rounding step.  Returns the bit
 * pattern.  Handles zero, subnormal results, overflow to infinity and NaN. */
uint16_t oracle_round_bf16(double v)
{
    if (isnan(v)) return 0x7FC0;
    double mag = fabs(v);
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    if (mag == 0.0) return sign;
    int e;
    frexp(mag, &e);                       /* mag = f * 2^e, f in [0.5, 1) */
    int exp_unbiased = e - 1;             /* mag in [2^(e-1), 2^e)        */
    if (exp_unbiased < -126) exp_unbiased = -126;   /* subnormal spacing */
    double quantum = ldexp(1.0, exp_unbiased - 7);  /* 8 significant bits */
    double q = mag / quantum;             /* exact: scaling by a power of 2 */
    double r = floor(q);
    double frac = q - r;
    if (frac > 0.5 || (frac == 0.5 && fmod(r, 2.0) != 0.0)) r += 1.0;
    double rounded = r * quantum;
    if (rounded >= 0x1p128) return sign | 0x7F80;   /* overflow -> inf */
    float f = (float)rounded;             /* exact: 8-bit significand */
    uint32_t w;
    memcpy(&w, &f, sizeof w);
    return sign | (uint16_t)((w >> 16) & 0x7FFF);
}

/* Element-wise oracle_round_bf16 over an array. */
void oracle_round_bf16_array(const double *v, int64_t n, uint16_t *out)
{
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = oracle_round_bf16(v[i]);
}

/* Thread count of the parallel loops above, for timing the oracle on a given
 * number of host cores (no arithmetic: every row is computed the same way). */
void oracle_set_threads(int n)
{
    if (n > 0)
        omp_set_num_threads(n);
}

int oracle_max_threads(void) { return omp_get_max_threads(); }
