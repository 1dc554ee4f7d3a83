/*
 * dptq_oracle.c -- plain, slow CPU oracle for the DynamicPTQ quantized linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent definition that the GPU
 * path is checked against.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it.  It shares no code, header, table or constant
 * generator with the CUDA library under paper_2606_12487_gb300/csrc, and the CUDA
 * library never calls it.
 *
 * What it computes (paper: "DynamicPTQ", arxiv 2606.12487):
 *   Section 2, "Low-Bit Quantization of LLMs":   Y = X W^T, the uniform b-bit
 *       quantizer Q_b(x) = s * round(x / s)            (Eq. 2, activation_quant)
 *       and its error e_b = x - Q_b(x)                 (Eq. 3, quant_error).
 *   Section 2, "Rotation-based Activation Transformation": quantize in a rotated
 *       space X R with R^T R = I                       (Eq. 4, rotation_activation)
 *       and fold R into the weight: X W^T = (XR)(WR)^T (Eq. 5, rotation_equiv).
 *   Section 4.2, "Implementation and Quantization Details": weights per-channel
 *       symmetric with RTN, activations per-token symmetric.
 *   Section 3.3, Algorithm 1 steps 1-2: weights 4-bit, activations 4 or 8 bit per
 *       layer (the mask is an input here).
 *
 * Readings where the paper is silent (each listed in the design notes):
 *   - symmetric quantizer s = absmax / (2^(b-1) - 1), no zero point (Section 4.2
 *     says "symmetric"; Eq. 1 prints the asymmetric range step);
 *   - round half to even; IEEE fp32 division y / s; clamp to [-2^(b-1), 2^(b-1)-1];
 *   - all-zero row: s = 0, every code 0;
 *   - R = blockdiag(H_B, ..., H_B, H_r) / sqrt(block), H the Sylvester Hadamard
 *     matrix in natural order, H[i][j] = (-1)^popcount(i & j); the tail block r is
 *     what is left of K after whole blocks of B: a power of two, or p 2^k with H_r the
 *     Kronecker product of Paley's H_p and the Sylvester H_(2^k) (orc_tail_factor);
 *   - scales in fp32; epilogue out = fp16_rne( fp32( fp32(acc) * s_a ) * s_w ).
 *
 * Precision: the rotation is evaluated in fp64 and rounded once to fp32.  For fp16
 * inputs the +-1 sum over a block is exact in fp64 (every fp16 is an integer
 * multiple of 2^-24 below 2^16, and 4096 of them sum below 2^52), so the only
 * roundings are the fp64 division by sqrt(block) and the final fp32 rounding.
 *
 * Build: cc -O2 -std=c11 -fPIC -shared dptq_oracle.c -o libdptq_oracle.so -lm
 * (no fast-math: the fp32 divisions and rintf must be IEEE).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* fp16 <-> fp32/fp64 by their IEEE 754 binary16 definitions                  */
/* ------------------------------------------------------------------------- */

/* binary16: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits. */
double orc_half_to_double(uint16_t h) {
    int sign = (h >> 15) & 1;
    int e = (h >> 10) & 0x1f;
    int f = h & 0x3ff;
    double v;
    if (e == 0) {
        v = ldexp((double)f, -24);                 /* subnormal: f * 2^-14 * 2^-10 */
    } else if (e == 31) {
        v = f ? NAN : INFINITY;
    } else {
        v = ldexp((double)(1024 + f), e - 25);     /* (1 + f/1024) * 2^(e-15) */
    }
    return sign ? -v : v;
}

/* Round a finite or infinite fp32 value to binary16, round-to-nearest-even,
 * overflow to +-inf, gradual underflow to subnormals. */
uint16_t orc_float_to_half(float xf) {
    double x = (double)xf;                          /* exact widening */
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (isnan(x)) return 0x7e00;
    if (isinf(a)) return sign | 0x7c00;
    if (a == 0.0) return sign;
    /* Find the binade: a = m * 2^e with 1 <= m < 2 (frexp gives 0.5 <= m < 1). */
    int e;
    (void)frexp(a, &e);
    e -= 1;                                         /* now a in [2^e, 2^(e+1)) */
    int q_exp = e < -14 ? -14 : e;                  /* subnormals share 2^-14 */
    double ulp = ldexp(1.0, q_exp - 10);            /* spacing of representable halves */
    double n = a / ulp;                             /* exact: power-of-two division */
    double r = floor(n);
    double frac = n - r;
    if (frac > 0.5 || (frac == 0.5 && fmod(r, 2.0) != 0.0)) r += 1.0;
    double v = r * ulp;                             /* rounded magnitude */
    if (v >= 65536.0) return sign | 0x7c00;         /* 65520 and up round to inf */
    if (v < ldexp(1.0, -14)) {                      /* subnormal or zero */
        return sign | (uint16_t)r;
    }
    int ve;
    (void)frexp(v, &ve);
    ve -= 1;
    uint32_t frac_bits = (uint32_t)(v / ldexp(1.0, ve - 10)) - 1024u;
    return sign | (uint16_t)((ve + 15) << 10) | (uint16_t)frac_bits;
}

/* ------------------------------------------------------------------------- */
/* Block Hadamard rotation (Section 2, Eq. 4 and Eq. 5)                        */
/* ------------------------------------------------------------------------- */

static int popcount32(uint32_t v) {
    int c = 0;
    while (v) { c += (int)(v & 1u); v >>= 1; }
    return c;
}

/* Sylvester Hadamard entry in natural order. */
int orc_hadamard_entry(int i, int j) {
    return (popcount32((uint32_t)(i & j)) & 1) ? -1 : 1;
}

static int is_pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }

static int is_prime(long v) {
    if (v < 2) return 0;
    for (long d = 2; d * d <= v; ++d)
        if (v % d == 0) return 0;
    return 1;
}

/* Quadratic character of a modulo the odd prime q: 0 for a = 0 (mod q), +1 for a
 * non-zero square, -1 otherwise (Euler's criterion, a^((q-1)/2) mod q). */
static int legendre(long a, long q) {
    long x = ((a % q) + q) % q;
    if (x == 0) return 0;
    long e = (q - 1) / 2, r = 1, b = x;
    while (e) {
        if (e & 1) r = (r * b) % q;
        b = (b * b) % q;
        e >>= 1;
    }
    return r == 1 ? 1 : -1;
}

/* Paley's first construction: for a prime q = p - 1 with q = 3 (mod 4),
 * H_p = I + S with S[0][0] = 0, S[0][j] = +1, S[i][0] = -1 and S[i][j] = chi(j - i)
 * (the Jacobsthal matrix of the quadratic character chi mod q) for i, j >= 1.  Because
 * chi(-1) = -1, S is skew-symmetric and H_p H_p^T = p I.  Entry (i, j), 0 <= i, j < p;
 * 0 when p is not such an order. */
int orc_paley_entry(int p, int i, int j) {
    if (p < 4 || p % 4 != 0 || !is_prime(p - 1)) return 0;
    if (i == j) return 1;
    if (i == 0) return 1;
    if (j == 0) return -1;
    return legendre((long)j - (long)i, p - 1);
}

/* Reading of the rotation for a tail block whose size r is not a power of two: the
 * Kronecker product H_p (x) H_(2^k) with r = p 2^k, H_p from Paley's construction, p the
 * smallest such order (odd part of r times 2^m, m >= 2, p - 1 prime) that divides r.
 * A power of two has p = 1.  Returns 0 (and leaves *p, *k unchanged) when r admits
 * neither. */
int orc_tail_factor(int r, int* p, int* k) {
    if (r <= 0) return 0;
    if (is_pow2(r)) {
        int t = 0;
        while ((1 << t) < r) ++t;
        *p = 1;
        *k = t;
        return 1;
    }
    int tz = 0;
    while (((r >> tz) & 1) == 0) ++tz;
    const int odd = r >> tz;
    for (int m = 2; m <= tz; ++m) {
        const long cand = (long)odd << m;
        if (is_prime(cand - 1)) {
            *p = (int)cand;
            *k = tz - m;
            return 1;
        }
    }
    return 0;
}

/* Entry (i, j) of the tail block's Hadamard matrix H_p (x) H_(2^k) (r = p 2^k):
 * H_p[i >> k][j >> k] * H_(2^k)[i & (2^k - 1)][j & (2^k - 1)]. */
int orc_tail_entry(int r, int i, int j) {
    int p, k;
    if (!orc_tail_factor(r, &p, &k)) return 0;
    if (p == 1) return orc_hadamard_entry(i, j);
    const int mask = (1 << k) - 1;
    return orc_paley_entry(p, i >> k, j >> k) * orc_hadamard_entry(i & mask, j & mask);
}

/* Block layout of R along K: q whole blocks of size B then one tail of size r.
 * Returns 0 when K does not split into blocks of B plus a tail that is a power of two
 * or a Paley order times a power of two (orc_tail_factor). */
int orc_block_layout(int K, int B, int* q, int* r) {
    if (K <= 0 || !is_pow2(B)) return 0;
    *q = K / B;
    *r = K % B;
    int p, k;
    if (*r != 0 && !orc_tail_factor(*r, &p, &k)) return 0;
    return 1;
}

/* The tail block's matrix H_r as a table, tab[j * r + k] = orc_tail_entry(r, j, k), when
 * the tail r = K mod B is not a power of two (its entries then cost a primality test and
 * a Legendre symbol each); NULL otherwise, and the entries are taken one by one. */
static signed char* tail_table(int K, int B) {
    int q, r, p, k;
    if (!orc_block_layout(K, B, &q, &r) || r == 0 || is_pow2(r) || !orc_tail_factor(r, &p, &k)) return NULL;
    signed char* tab = (signed char*)malloc((size_t)r * (size_t)r);
    if (!tab) return NULL;
    for (int j = 0; j < r; ++j)
        for (int c = 0; c < r; ++c) tab[(size_t)j * r + c] = (signed char)orc_tail_entry(r, j, c);
    return tab;
}

/* y[k] = sum_j x[j] R[j][k] for one row of length K, in fp64.
 * R = blockdiag(H_B/sqrt(B), ..., H_r/sqrt(r)), the tail's H_r from orc_tail_entry
 * (read from tab when given).  Returns 0 on a bad layout. */
static int rotate_row(const double* x, double* y, int K, int B, const signed char* tab) {
    int q, r;
    if (!orc_block_layout(K, B, &q, &r)) return 0;
    int nblk = q + (r ? 1 : 0);
    for (int b = 0; b < nblk; ++b) {
        int k0 = b * B;
        int n = (b < q) ? B : r;
        double norm = sqrt((double)n);
        for (int k = 0; k < n; ++k) {
            double acc = 0.0;
            for (int j = 0; j < n; ++j) {
                const int h = b < q ? orc_hadamard_entry(j, k)
                                    : (tab ? tab[(size_t)j * n + k] : orc_tail_entry(n, j, k));
                acc += x[k0 + j] * (double)h;
            }
            y[k0 + k] = acc / norm;
        }
    }
    return 1;
}

int orc_rotate_row_f64(const double* x, double* y, int K, int B) {
    signed char* tab = tail_table(K, B);
    const int ok = rotate_row(x, y, K, B, tab);
    free(tab);
    return ok;
}

/* Rotate an fp16 matrix x[M][K] (row-major, raw binary16 bits) into fp32 y[M][K]:
 * evaluate in fp64, round once to fp32.
 * signs (may be NULL): the randomized Hadamard of QuaRot (Section 1; Section 4.2),
 * R' = D R with D = diag(signs), signs[k] in {+1, -1}: x is multiplied elementwise by
 * the signs before the block Hadamard.  D is orthogonal, so R'^T R' = I still holds
 * (Eq. 4), and folding the same R' into the weights keeps X W^T (Eq. 5). */
int orc_rotate_f16_signed(const uint16_t* x, float* y, int M, int K, int B, const int8_t* signs) {
    int q, r;
    if (!orc_block_layout(K, B, &q, &r)) return 0;
    double* xr = (double*)malloc(sizeof(double) * (size_t)K);
    double* yr = (double*)malloc(sizeof(double) * (size_t)K);
    if (!xr || !yr) { free(xr); free(yr); return 0; }
    signed char* tab = tail_table(K, B);
    for (int m = 0; m < M; ++m) {
        for (int k = 0; k < K; ++k) {
            xr[k] = orc_half_to_double(x[(size_t)m * K + k]);
            if (signs && signs[k] < 0) xr[k] = -xr[k];
        }
        rotate_row(xr, yr, K, B, tab);
        for (int k = 0; k < K; ++k) y[(size_t)m * K + k] = (float)yr[k];
    }
    free(tab);
    free(xr);
    free(yr);
    return 1;
}

int orc_rotate_f16(const uint16_t* x, float* y, int M, int K, int B) {
    return orc_rotate_f16_signed(x, y, M, K, B, NULL);
}

/* ------------------------------------------------------------------------- */
/* Symmetric quantizer (Section 2 Eq. 2; Section 4.2 "symmetric")              */
/* ------------------------------------------------------------------------- */

/* One row: s = max|y| / qmax (fp32 division), c = clamp(rint(y / s)).
 * bits in {4, 8}.  Returns the scale; writes K codes. */
float orc_quant_row(const float* y, int K, int bits, int8_t* codes) {
    int qmax = (1 << (bits - 1)) - 1;
    int qmin = -(1 << (bits - 1));
    float amax = 0.0f;
    for (int k = 0; k < K; ++k) {
        float a = fabsf(y[k]);
        if (a > amax) amax = a;
    }
    float s = amax / (float)qmax;
    for (int k = 0; k < K; ++k) {
        int c = 0;
        if (amax > 0.0f) {
            float t = y[k] / s;                     /* IEEE fp32 division */
            float rt = rintf(t);                    /* round half to even */
            c = (int)rt;
            if (c > qmax) c = qmax;
            if (c < qmin) c = qmin;
        }
        codes[k] = (int8_t)c;
    }
    return s;
}

int orc_quant_rows(const float* y, int M, int K, int bits, int8_t* codes, float* scales) {
    if (bits != 4 && bits != 8) return 0;
    for (int m = 0; m < M; ++m)
        scales[m] = orc_quant_row(y + (size_t)m * K, K, bits, codes + (size_t)m * K);
    return 1;
}

/* Online activation path: rotate (Eq. 4) then per-token quantize (Eq. 2).
 * signs: NULL, or the randomized Hadamard's diagonal (see orc_rotate_f16_signed). */
int orc_rotate_quant_act_signed(const uint16_t* x, int M, int K, int B, int bits, const int8_t* signs,
                                int8_t* codes, float* scales) {
    if (bits != 4 && bits != 8) return 0;
    float* y = (float*)malloc(sizeof(float) * (size_t)M * K);
    if (!y) return 0;
    int ok = orc_rotate_f16_signed(x, y, M, K, B, signs);
    if (ok) orc_quant_rows(y, M, K, bits, codes, scales);
    free(y);
    return ok;
}

int orc_rotate_quant_act(const uint16_t* x, int M, int K, int B, int bits,
                         int8_t* codes, float* scales) {
    return orc_rotate_quant_act_signed(x, M, K, B, bits, NULL, codes, scales);
}

/* Offline weight path (Eq. 5 fold, Section 4.2 RTN per-channel symmetric int4):
 * W'[n] = W[n] R, s_w[n] = max|W'[n]| / 7, q = clamp(rint(W'/s_w), -8, 7). */
int orc_pack_weights_signed(const uint16_t* W, int N, int K, int B, const int8_t* signs, int8_t* q, float* sw) {
    return orc_rotate_quant_act_signed(W, N, K, B, 4, signs, q, sw);
}

int orc_pack_weights(const uint16_t* W, int N, int K, int B, int8_t* q, float* sw) {
    return orc_pack_weights_signed(W, N, K, B, NULL, q, sw);
}

/* ------------------------------------------------------------------------- */
/* Integer GEMM and the scale epilogue (Section 2: Y = X W^T)                  */
/* ------------------------------------------------------------------------- */

/* acc[m][n] = sum_k a[m][k] * w[n][k], evaluated in int64.  Returns 0 if any sum
 * leaves the int32 range (the GPU accumulates in 32 bits). */
int orc_gemm_i32(const int8_t* a, const int8_t* w, int M, int N, int K, int32_t* acc) {
    int ok = 1;
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            int64_t s = 0;
            for (int k = 0; k < K; ++k)
                s += (int64_t)a[(size_t)m * K + k] * (int64_t)w[(size_t)n * K + k];
            if (s > INT32_MAX || s < INT32_MIN) ok = 0;
            acc[(size_t)m * N + n] = (int32_t)s;
        }
    }
    return ok;
}

/* out[m][n] = fp16_rne( fp32( fp32(acc) * s_a[m] ) * s_w[n] ), every product a
 * single fp32 rounding (dequantization s * c of Eq. 2 on both operands). */
void orc_epilogue(const int32_t* acc, const float* sa, const float* sw, int M, int N,
                  uint16_t* out) {
    for (int m = 0; m < M; ++m) {
        for (int n = 0; n < N; ++n) {
            float a = (float)acc[(size_t)m * N + n];
            float t = a * sa[m];
            float v = t * sw[n];
            out[(size_t)m * N + n] = orc_float_to_half(v);
        }
    }
}

/* The whole quantized linear layer for one activation matrix:
 * rotate + quantize x, integer GEMM against packed weights q (int4 codes in int8),
 * scale epilogue.  acc may be NULL.  Returns 0 on a bad shape or int32 overflow. */
int orc_qlinear_signed(const uint16_t* x, int M, int K, int B, int bits, const int8_t* signs,
                       const int8_t* q, const float* sw, int N,
                       uint16_t* out, int32_t* acc_out, int8_t* codes_out, float* sa_out) {
    int8_t* codes = codes_out ? codes_out : (int8_t*)malloc((size_t)M * K);
    float* sa = sa_out ? sa_out : (float*)malloc(sizeof(float) * (size_t)M);
    int32_t* acc = acc_out ? acc_out : (int32_t*)malloc(sizeof(int32_t) * (size_t)M * N);
    int ok = codes && sa && acc;
    if (ok) ok = orc_rotate_quant_act_signed(x, M, K, B, bits, signs, codes, sa);
    if (ok) ok = orc_gemm_i32(codes, q, M, N, K, acc);
    if (ok) orc_epilogue(acc, sa, sw, M, N, out);
    if (!codes_out) free(codes);
    if (!sa_out) free(sa);
    if (!acc_out) free(acc);
    return ok;
}

int orc_qlinear(const uint16_t* x, int M, int K, int B, int bits,
                const int8_t* q, const float* sw, int N,
                uint16_t* out, int32_t* acc_out, int8_t* codes_out, float* sa_out) {
    return orc_qlinear_signed(x, M, K, B, bits, NULL, q, sw, N, out, acc_out, codes_out, sa_out);
}

/* ------------------------------------------------------------------------- */
/* KV-cache quantization (Section 4.2: group-wise, group size 128, 4-bit)       */
/* ------------------------------------------------------------------------- */

/* Group-wise symmetric 4-bit codes of an fp16 matrix x[rows][cols]: each row is cut
 * into groups of `group` consecutive columns, and each group is quantized on its own
 * with the quantizer of Eq. 2 (s = max|x| / 7, c = clamp(rint(x / s), -8, 7), an
 * all-zero group gets s = 0).  The paper says group-wise with group 128 and does not
 * say symmetric or asymmetric; symmetric is this oracle's reading.  codes int8
 * [rows][cols], scales fp32 [rows][cols / group].  Returns 0 unless group divides
 * cols. */
int orc_kv4_quantize(const uint16_t* x, int rows, int cols, int group, int8_t* codes, float* scales) {
    if (group <= 0 || cols % group != 0) return 0;
    float* v = (float*)malloc(sizeof(float) * (size_t)group);
    if (!v) return 0;
    int ng = cols / group;
    for (int m = 0; m < rows; ++m) {
        for (int g = 0; g < ng; ++g) {
            size_t base = (size_t)m * cols + (size_t)g * group;
            for (int i = 0; i < group; ++i) v[i] = (float)orc_half_to_double(x[base + i]);
            scales[(size_t)m * ng + g] = orc_quant_row(v, group, 4, codes + base);
        }
    }
    free(v);
    return 1;
}

/* ------------------------------------------------------------------------- */
/* Sensitive-layer policy (Section 3.3, Eq. 20; Algorithm 1 step 2)             */
/* ------------------------------------------------------------------------- */

/* bits[l] = 8 if JR_l > tau_jr and SNR_l < tau_snr (the sensitive set of Eq. 20),
 * else 4.  The paper gives no threshold values; they are inputs. */
void orc_policy_mask(const double* jr, const double* snr, int L, double tau_jr, double tau_snr,
                     uint8_t* bits) {
    for (int l = 0; l < L; ++l) bits[l] = (jr[l] > tau_jr && snr[l] < tau_snr) ? 8 : 4;
}

/* ------------------------------------------------------------------------- */
/* Public code formats                                                         */
/* ------------------------------------------------------------------------- */

/* 4-bit codes two to a byte: byte k/2 holds code k (even) in its low nibble and
 * code k+1 in its high nibble, each as 4-bit two's complement.  K even. */
void orc_pack_nibbles(const int8_t* codes, int rows, int K, uint8_t* packed) {
    for (int m = 0; m < rows; ++m) {
        for (int k = 0; k < K; k += 2) {
            uint8_t lo = (uint8_t)(codes[(size_t)m * K + k] & 0x0f);
            uint8_t hi = (uint8_t)(codes[(size_t)m * K + k + 1] & 0x0f);
            packed[(size_t)m * (K / 2) + k / 2] = (uint8_t)(lo | (hi << 4));
        }
    }
}

void orc_unpack_nibbles(const uint8_t* packed, int rows, int K, int8_t* codes) {
    for (int m = 0; m < rows; ++m) {
        for (int k = 0; k < K; k += 2) {
            uint8_t b = packed[(size_t)m * (K / 2) + k / 2];
            int lo = b & 0x0f, hi = (b >> 4) & 0x0f;
            codes[(size_t)m * K + k] = (int8_t)(lo >= 8 ? lo - 16 : lo);
            codes[(size_t)m * K + k + 1] = (int8_t)(hi >= 8 ? hi - 16 : hi);
        }
    }
}

/* ------------------------------------------------------------------------- */
/* Residual-stream statistics (Section 3.1, Eqs. 8-11), for the sensitivity    */
/* policy that produces the per-layer bit mask.                                */
/* ------------------------------------------------------------------------- */

/* JR_l = mean_t ||dx_t|| / (||x_t|| + eps)                       (Eqs. 8-9)
 * SNR_l = mean_t 10 log10( ||x_t||^2 / (||xhat_t - x_t||^2 + eps) )  (Eqs. 10-11)
 * with xhat_t = Q_b(x_t + dx_t) - dx_t, Q_b the per-token symmetric quantizer of
 * Eq. 2 applied to the updated state (Eq. 7), evaluated in fp64 apart from Q_b,
 * which follows the fp32 quantizer above.  x, dx are fp32 [T][d]. */
int orc_residual_stats(const float* x, const float* dx, int T, int d, int bits, double eps,
                       double* jr_out, double* snr_out) {
    float* upd = (float*)malloc(sizeof(float) * (size_t)d);
    int8_t* c = (int8_t*)malloc((size_t)d);
    if (!upd || !c) { free(upd); free(c); return 0; }
    double jr = 0.0, snr = 0.0;
    for (int t = 0; t < T; ++t) {
        const float* xt = x + (size_t)t * d;
        const float* dt = dx + (size_t)t * d;
        double nx2 = 0.0, nd2 = 0.0;
        for (int i = 0; i < d; ++i) {
            nx2 += (double)xt[i] * xt[i];
            nd2 += (double)dt[i] * dt[i];
            upd[i] = xt[i] + dt[i];
        }
        jr += sqrt(nd2) / (sqrt(nx2) + eps);
        float s = orc_quant_row(upd, d, bits, c);
        double err2 = 0.0;
        for (int i = 0; i < d; ++i) {
            double xhat = (double)s * c[i] - (double)dt[i];   /* Eq. 10 */
            double e = xhat - (double)xt[i];
            err2 += e * e;
        }
        snr += 10.0 * log10(nx2 / (err2 + eps));
    }
    *jr_out = jr / T;
    *snr_out = snr / T;
    free(upd);
    free(c);
    return 1;
}
