/*
 * wq_oracle.c -- CPU oracle for the W4/W2-GateUp decode MLP path.
 *
 * TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and the
 * cpu_baseline / reference legs of bench.py may load or call this library.
 * The product path (the CUDA library under paper_2606_04238_gb300/) never
 * calls it, and the two share no code, header, table or helper.
 *
 * Everything here is the plain definition, written out with no blocking,
 * fusion or reordering:
 *
 *   - Stage-1 quantization (Sec. 4.1; W4/W2-GateUp configuration, Sec. 3.3):
 *     asymmetric min-max round-to-nearest per group of `group` consecutive
 *     input features of one output row, done in IEEE fp32 exactly as the
 *     packed format defines it, so that codes, scales and zeros can be
 *     compared bit for bit.
 *   - The tiled storage format of those codes / scales / zeros (a byte
 *     layout; its definition is the packing loop below).
 *   - LoRA forward Y = W X + alpha B A X (Eq. 1), with W the dequantized
 *     matrix, evaluated in fp64.
 *   - The gated MLP h = SiLU(gate(x)) * up(x), y = x + down(h) (Sec. 3.3),
 *     optionally preceded by a unit-weight RMSNorm of the MLP input.
 *   - The down layer of the BF16/W2-GateUp configuration (bf16 weights,
 *     Sec. 6.1), and the merged matrix deq(W) + alpha B A of an adapter
 *     folded into the quantized weights (Sec. 4.2).
 *
 * bf16 rounding happens only where the CUDA path stores a bf16 tensor: the
 * hidden activation h and the layer output y.  The RMSNorm-normalized input
 * is never stored, so it is used unrounded.  Between those points the
 * arithmetic is fp64.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_OK 0
#define ORC_ERR_ARG (-1)

/* ------------------------------------------------------------------ */
/* IEEE 754 conversions, written from the binary16 / bfloat16 formats. */
/* ------------------------------------------------------------------ */

/* fp32 -> binary16, round to nearest, ties to even. */
uint16_t orc_f32_to_f16(float f)
{
    uint32_t bits;
    memcpy(&bits, &f, 4);
    uint16_t sign = (uint16_t)((bits >> 16) & 0x8000u);
    if (isnan(f)) return (uint16_t)(sign | 0x7E00u);
    double a = fabs((double)f);
    if (isinf(f)) return (uint16_t)(sign | 0x7C00u);
    if (a == 0.0) return sign;
    int e;
    frexp(a, &e);               /* a in [2^(e-1), 2^e) */
    int E = e - 1;
    if (E < -14) E = -14;       /* subnormal binade: spacing 2^-24 */
    double quantum = ldexp(1.0, E - 10);
    double r = rint(a / quantum) * quantum;   /* exact scaling, ties-even */
    if (r > 65504.0) return (uint16_t)(sign | 0x7C00u);
    if (r < ldexp(1.0, -14)) {
        return (uint16_t)(sign | (uint16_t)(r / ldexp(1.0, -24)));
    }
    frexp(r, &e);
    E = e - 1;
    uint16_t ex = (uint16_t)(E + 15);
    uint16_t mant = (uint16_t)((r / ldexp(1.0, E) - 1.0) * 1024.0);
    return (uint16_t)(sign | (ex << 10) | mant);
}

/* binary16 -> fp64 (exact). */
double orc_f16_to_f64(uint16_t h)
{
    int sign = (h >> 15) & 1;
    int ex = (h >> 10) & 31;
    int mant = h & 1023;
    double v;
    if (ex == 0) v = ldexp((double)mant, -24);
    else if (ex == 31) v = mant ? NAN : INFINITY;
    else v = ldexp(1.0 + mant / 1024.0, ex - 15);
    return sign ? -v : v;
}

/* fp64 -> bfloat16, round to nearest, ties to even. */
uint16_t orc_f64_to_bf16(double v)
{
    if (isnan(v)) return 0x7FC0u;
    uint16_t sign = signbit(v) ? 0x8000u : 0;
    double a = fabs(v);
    if (isinf(a)) return (uint16_t)(sign | 0x7F80u);
    if (a == 0.0) return sign;
    int e;
    frexp(a, &e);
    int E = e - 1;
    if (E < -126) E = -126;     /* subnormal binade: spacing 2^-133 */
    double quantum = ldexp(1.0, E - 7);
    double r = rint(a / quantum) * quantum;
    if (r >= ldexp(1.0, 128)) return (uint16_t)(sign | 0x7F80u);
    float rf = (float)r;        /* exact: r has at most 8 significant bits */
    uint32_t bits;
    memcpy(&bits, &rf, 4);
    return (uint16_t)(sign | (uint16_t)(bits >> 16));
}

/* bfloat16 -> fp64 (exact). */
double orc_bf16_to_f64(uint16_t b)
{
    uint32_t bits = (uint32_t)b << 16;
    float f;
    memcpy(&f, &bits, 4);
    return (double)f;
}

/* ------------------------------------------------------------------ */
/* Stage-1 quantization (Sec. 4.1): asymmetric min-max RTN per group.  */
/* ------------------------------------------------------------------ */
/*
 * For output row n and group j (input features j*group .. j*group+group-1):
 *   mn, mx   = min, max of the group's fp32 weights
 *   s        = fp16(( mx - mn ) / qmax)          IEEE fp32 division, then RN
 *              (s = 1.0 when that rounds to zero: a constant group)
 *   z        = clamp(rint(-mn / s), 0, qmax)      stored as fp16 (an integer)
 *   q[n,k]   = clamp(rint(w[n,k] / s) + z, 0, qmax)
 * qmax = 2^bits - 1.  rint is round-half-to-even.  Every division is an IEEE
 * fp32 division by the stored (fp16) scale.
 * Returns the number of non-finite weights seen (0 for a clean matrix), or a
 * negative error code.
 */
int orc_quantize(const float *w, int n, int k, int group, int bits,
                 uint8_t *q, uint16_t *s_out, uint16_t *z_out)
{
    if (n < 0 || k < 0 || group <= 0 || k % group != 0) return ORC_ERR_ARG;
    if (bits < 2 || bits > 4) return ORC_ERR_ARG;   /* INT2, INT3 (App. B), INT4 */
    const float qmax = (float)((1 << bits) - 1);
    const int ng = k / group;
    int nonfinite = 0;
    for (int r = 0; r < n; ++r) {
        for (int j = 0; j < ng; ++j) {
            const float *wg = w + (size_t)r * k + (size_t)j * group;
            float mn = INFINITY, mx = -INFINITY;
            for (int i = 0; i < group; ++i) {
                if (!isfinite(wg[i])) nonfinite++;
                mn = fminf(mn, wg[i]);
                mx = fmaxf(mx, wg[i]);
            }
            volatile float range = mx - mn;
            volatile float s32 = range / qmax;
            uint16_t s16 = orc_f32_to_f16(s32);
            if (orc_f16_to_f64(s16) == 0.0) s16 = 0x3C00u; /* 1.0 */
            float sf = (float)orc_f16_to_f64(s16);
            volatile float negmn_over_s = -mn / sf;
            float zf = fminf(fmaxf(rintf(negmn_over_s), 0.0f), qmax) + 0.0f;
            s_out[(size_t)r * ng + j] = s16;
            z_out[(size_t)r * ng + j] = orc_f32_to_f16(zf);
            for (int i = 0; i < group; ++i) {
                volatile float ratio = wg[i] / sf;
                float qf = fminf(fmaxf(rintf(ratio) + zf, 0.0f), qmax);
                q[(size_t)r * k + (size_t)j * group + i] = (uint8_t)qf;
            }
        }
    }
    return nonfinite;
}

/* ------------------------------------------------------------------ */
/* Packed storage format.                                              */
/* ------------------------------------------------------------------ */
/*
 * Rows are padded to a multiple of 16 and input features to a multiple of
 * 128; padded codes are 0 and padded scales and zeros are 0, so padding adds
 * nothing to any dot product.
 *
 * codes: uint32 words, one block of 16 rows x 128 features after another,
 * blocks ordered row-tile major: block (rt, kb) starts at word
 * (rt * KB + kb) * words_per_block, KB = K_pad / 128.  Within a block, a code
 * for local row i (0..15) and local feature c (0..127) lives in
 *   lane  = (i % 8) * 4 + (c % 8) / 2
 *   half  = c % 2                      (bit 16 of the word selects it)
 * and, for 2-bit codes (128 words per block):
 *   word  = lane * 4 + c / 32
 *   bit   = 16*half + 8*(i / 8) + 2*( 2*((c % 32) / 16) + (c % 16) / 8 )
 * and, for 4-bit codes (256 words per block, two 64-feature halves):
 *   word  = (c / 64) * 128 + lane * 4 + (c % 64) / 16
 *   bit   = 16*half + 8*(i / 8) + 4*((c % 16) / 8)
 * and, for 3-bit codes (App. B; 192 words per block, 3 bits a weight), two
 * bit planes: q % 4 in words 0..127 exactly as a 2-bit code, and q / 4 in
 * words 128..191:
 *   word  = 128 + lane * 2 + (c / 32) / 2
 *   bit   = 16*half + 8*((c / 32) % 2) + 2*( 2*((c % 32) / 16) + (c % 16) / 8 ) + i / 8
 *
 * meta: uint16 (binary16) values, 32 per (row tile, group): for row tile rt
 * and group j (NG = K_pad / group groups per row) the 32 values at
 * (rt * NG + j) * 32 are, for e = 0..7,
 *   [4e+0] = s[row 16rt+e]   [4e+1] = s[row 16rt+e+8]
 *   [4e+2] = z[row 16rt+e]   [4e+3] = z[row 16rt+e+8]
 */
static int orc_words_per_block(int bits) { return bits == 2 ? 128 : bits == 3 ? 192 : 256; }

int orc_tile_pack(const uint8_t *q, const uint16_t *s, const uint16_t *z,
                  int n, int k, int group, int bits,
                  uint32_t *codes, uint16_t *meta)
{
    if (bits < 2 || bits > 4 || group <= 0 || k % group != 0 || 128 % group != 0)
        return ORC_ERR_ARG;
    const int RT = (n + 15) / 16, KB = (k + 127) / 128;
    const int Kp = KB * 128, NG = Kp / group, ngk = k / group;
    const int wpb = orc_words_per_block(bits);
    memset(codes, 0, sizeof(uint32_t) * (size_t)RT * KB * wpb);
    memset(meta, 0, sizeof(uint16_t) * (size_t)RT * NG * 32);
    for (int r = 0; r < n; ++r) {
        const int rt = r / 16, i = r % 16;
        for (int col = 0; col < k; ++col) {
            const int kb = col / 128, c = col % 128;
            const uint32_t code = q[(size_t)r * k + col];
            const int lane = (i % 8) * 4 + (c % 8) / 2;
            const int half = c % 2;
            int word, bit;
            if (bits == 4) {
                word = (c / 64) * 128 + lane * 4 + (c % 64) / 16;
                bit = 16 * half + 8 * (i / 8) + 4 * ((c % 16) / 8);
            } else {
                word = lane * 4 + c / 32;
                bit = 16 * half + 8 * (i / 8) + 2 * (2 * ((c % 32) / 16) + (c % 16) / 8);
            }
            uint32_t *blk = codes + ((size_t)rt * KB + kb) * wpb;
            if (bits == 3) {
                const int cls = 2 * ((c % 32) / 16) + (c % 16) / 8;
                blk[word] |= (code & 3u) << bit;
                blk[128 + lane * 2 + (c / 32) / 2] |=
                    (code >> 2) << (16 * half + 8 * ((c / 32) % 2) + 2 * cls + i / 8);
            } else {
                blk[word] |= code << bit;
            }
        }
        for (int j = 0; j < ngk; ++j) {
            const size_t base = ((size_t)rt * NG + j) * 32;
            const int e = i % 8, hi = i / 8;
            meta[base + 4 * e + 0 + hi] = s[(size_t)r * ngk + j];
            meta[base + 4 * e + 2 + hi] = z[(size_t)r * ngk + j];
        }
    }
    return ORC_OK;
}

int orc_tile_unpack(const uint32_t *codes, const uint16_t *meta,
                    int n, int k, int group, int bits,
                    uint8_t *q, uint16_t *s, uint16_t *z)
{
    if (bits < 2 || bits > 4 || group <= 0 || k % group != 0 || 128 % group != 0)
        return ORC_ERR_ARG;
    const int KB = (k + 127) / 128;
    const int Kp = KB * 128, NG = Kp / group, ngk = k / group;
    const int wpb = orc_words_per_block(bits);
    const uint32_t mask = (1u << bits) - 1u;
    for (int r = 0; r < n; ++r) {
        const int rt = r / 16, i = r % 16;
        for (int col = 0; col < k; ++col) {
            const int kb = col / 128, c = col % 128;
            const int lane = (i % 8) * 4 + (c % 8) / 2;
            const int half = c % 2;
            int word, bit;
            if (bits == 4) {
                word = (c / 64) * 128 + lane * 4 + (c % 64) / 16;
                bit = 16 * half + 8 * (i / 8) + 4 * ((c % 16) / 8);
            } else {
                word = lane * 4 + c / 32;
                bit = 16 * half + 8 * (i / 8) + 2 * (2 * ((c % 32) / 16) + (c % 16) / 8);
            }
            const uint32_t *blk = codes + ((size_t)rt * KB + kb) * wpb;
            if (bits == 3) {
                const int cls = 2 * ((c % 32) / 16) + (c % 16) / 8;
                const uint32_t hi = (blk[128 + lane * 2 + (c / 32) / 2] >>
                                     (16 * half + 8 * ((c / 32) % 2) + 2 * cls + i / 8)) & 1u;
                q[(size_t)r * k + col] = (uint8_t)(((blk[word] >> bit) & 3u) | (hi << 2));
            } else {
                q[(size_t)r * k + col] = (uint8_t)((blk[word] >> bit) & mask);
            }
        }
        for (int j = 0; j < ngk; ++j) {
            const size_t base = ((size_t)rt * NG + j) * 32;
            const int e = i % 8, hi = i / 8;
            s[(size_t)r * ngk + j] = meta[base + 4 * e + 0 + hi];
            z[(size_t)r * ngk + j] = meta[base + 4 * e + 2 + hi];
        }
    }
    return ORC_OK;
}

/* deq(W)[n,k] = s[n, k/group] * (q[n,k] - z[n, k/group]), in fp64. */
int orc_dequant(const uint8_t *q, const uint16_t *s, const uint16_t *z,
                int n, int k, int group, double *w)
{
    if (group <= 0 || k % group != 0) return ORC_ERR_ARG;
    const int ng = k / group;
    for (int r = 0; r < n; ++r)
        for (int col = 0; col < k; ++col) {
            const size_t gi = (size_t)r * ng + col / group;
            w[(size_t)r * k + col] =
                orc_f16_to_f64(s[gi]) * ((double)q[(size_t)r * k + col] - orc_f16_to_f64(z[gi]));
        }
    return ORC_OK;
}

/*
 * Merging the adapter into the quantized matrix (Sec. 4.2: once trained, the
 * adapters may be merged into the quantized weights instead of being kept as
 * a separate module; Sec. 7, step 5 of the deployment pipeline).  By Eq. 1
 * the merged matrix is W + alpha B A, with W the dequantized matrix:
 *   w_out[n,k] = fp32( s[n,j] (q[n,k] - z[n,j]) + alpha * sum_rho B[n,rho] A[rho,k] )
 * with j = k / group, B bf16 [n, r], A bf16 [r, k].  The sum runs over rho
 * in ascending order in fp64 (every product of two bf16 values is exact in
 * fp64), alpha multiplies it in fp64, and the result is rounded to fp32 once.
 * The merged matrix is then quantized again with orc_quantize at the same
 * bits and group (the paper names no other quantizer for this step).
 */
int orc_merge_lora(const uint8_t *q, const uint16_t *s, const uint16_t *z,
                   int n, int k, int group,
                   const uint16_t *lora_b, const uint16_t *lora_a, int r,
                   double lora_scale, float *w_out)
{
    if (n < 0 || k < 0 || group <= 0 || k % group != 0 || r < 0) return ORC_ERR_ARG;
    const int ng = k / group;
    for (int row = 0; row < n; ++row)
        for (int col = 0; col < k; ++col) {
            const size_t gi = (size_t)row * ng + col / group;
            const double w = orc_f16_to_f64(s[gi]) *
                             ((double)q[(size_t)row * k + col] - orc_f16_to_f64(z[gi]));
            double ba = 0.0;
            for (int rho = 0; rho < r; ++rho)
                ba += orc_bf16_to_f64(lora_b[(size_t)row * r + rho]) *
                      orc_bf16_to_f64(lora_a[(size_t)rho * k + col]);
            w_out[(size_t)row * k + col] = (float)(w + lora_scale * ba);
        }
    return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* Forward pass.                                                       */
/* ------------------------------------------------------------------ */

/*
 * Unit-weight RMSNorm scale of each token: rs[t] = 1 / sqrt(mean_c x[t,c]^2 + eps).
 * The normalized input x[t,c] * rs[t] is used unrounded by orc_gateup (it is
 * never stored, so it has no bf16 rounding point).
 */
int orc_rms_scale(const uint16_t *x, int m, int d, double eps, double *rs)
{
    if (m < 0 || d <= 0) return ORC_ERR_ARG;
    for (int t = 0; t < m; ++t) {
        double ss = 0.0;
        for (int c = 0; c < d; ++c) {
            double v = orc_bf16_to_f64(x[(size_t)t * d + c]);
            ss += v * v;
        }
        rs[t] = 1.0 / sqrt(ss / d + eps);
    }
    return ORC_OK;
}

/* One quantized row dotted with one activation row: sum_k x[k] * s(q - z). */
static double orc_qdot_f64(const uint8_t *qrow, const uint16_t *srow, const uint16_t *zrow,
                           int k, int group, const double *xrow)
{
    double acc = 0.0;
    for (int col = 0; col < k; ++col) {
        const int j = col / group;
        const double w = orc_f16_to_f64(srow[j]) * ((double)qrow[col] - orc_f16_to_f64(zrow[j]));
        acc += xrow[col] * w;
    }
    return acc;
}

/* The same with a bf16 activation row. */
static double orc_qdot(const uint8_t *qrow, const uint16_t *srow, const uint16_t *zrow,
                       int k, int group, const uint16_t *xrow)
{
    double acc = 0.0;
    for (int col = 0; col < k; ++col) {
        const int j = col / group;
        const double w = orc_f16_to_f64(srow[j]) * ((double)qrow[col] - orc_f16_to_f64(zrow[j]));
        acc += orc_bf16_to_f64(xrow[col]) * w;
    }
    return acc;
}

/*
 * Gate/up half of the gated MLP with unmerged LoRA on both projections
 * (Eq. 1 applied to gate and to up, then SiLU(gate) * up):
 *   xin      = prenorm ? x * rs (RMSNorm, unrounded, rs of orc_rms_scale) : x
 *   t_g      = xin . A_g^T,  t_u = xin . A_u^T        (A = lora_a rows 0..r-1 / r..2r-1)
 *   g[m,n]   = sum_k xin[m,k] deq(Wg)[n,k] + lora_scale * sum_p t_g[m,p] B_g[n,p]
 *   u[m,n]   = likewise with Wu, A_u, B_u
 *   h[m,n]   = g / (1 + exp(-g)) * u
 * x: [m, d] bf16.  Wg, Wu: [inter, d] codes + [inter, d/group] scales/zeros.
 * lora_a: [2r, d] bf16, lora_bg / lora_bu: [inter, r] bf16 (r = 0: no LoRA).
 * h_f64: [m, inter] (optional), h_bf16: [m, inter] bf16 (optional).
 */
int orc_gateup(const uint16_t *x, int m, int d, int inter,
               const uint8_t *qg, const uint16_t *sg, const uint16_t *zg,
               const uint8_t *qu, const uint16_t *su, const uint16_t *zu, int group,
               const uint16_t *lora_a, const uint16_t *lora_bg, const uint16_t *lora_bu,
               int r, double lora_scale, int prenorm, double eps,
               double *h_f64, uint16_t *h_bf16)
{
    if (m < 0 || d <= 0 || inter <= 0 || group <= 0 || d % group != 0 || r < 0) return ORC_ERR_ARG;
    const int ng = d / group;
    double *xin = (double *)malloc(sizeof(double) * ((size_t)m * d + 1));
    double *rs = (double *)malloc(sizeof(double) * ((size_t)m + 1));
    double *t = (double *)malloc(sizeof(double) * ((size_t)m * 2 * r + 1));
    if (!xin || !rs || !t) { free(xin); free(rs); free(t); return ORC_ERR_ARG; }
    for (int tk = 0; tk < m; ++tk) rs[tk] = 1.0;
    if (prenorm) orc_rms_scale(x, m, d, eps, rs);
    for (int tk = 0; tk < m; ++tk)
        for (int c = 0; c < d; ++c)
            xin[(size_t)tk * d + c] = orc_bf16_to_f64(x[(size_t)tk * d + c]) * rs[tk];
    for (int tk = 0; tk < m; ++tk)
        for (int p = 0; p < 2 * r; ++p) {
            double acc = 0.0;
            for (int c = 0; c < d; ++c)
                acc += xin[(size_t)tk * d + c] * orc_bf16_to_f64(lora_a[(size_t)p * d + c]);
            t[(size_t)tk * 2 * r + p] = acc;
        }
#pragma omp parallel for schedule(static)
    for (int n = 0; n < inter; ++n) {
        for (int tk = 0; tk < m; ++tk) {
            const double *xr = xin + (size_t)tk * d;
            double g = orc_qdot_f64(qg + (size_t)n * d, sg + (size_t)n * ng, zg + (size_t)n * ng, d, group, xr);
            double u = orc_qdot_f64(qu + (size_t)n * d, su + (size_t)n * ng, zu + (size_t)n * ng, d, group, xr);
            double lg = 0.0, lu = 0.0;
            for (int p = 0; p < r; ++p) {
                lg += t[(size_t)tk * 2 * r + p] * orc_bf16_to_f64(lora_bg[(size_t)n * r + p]);
                lu += t[(size_t)tk * 2 * r + r + p] * orc_bf16_to_f64(lora_bu[(size_t)n * r + p]);
            }
            g += lora_scale * lg;
            u += lora_scale * lu;
            const double h = g / (1.0 + exp(-g)) * u;
            if (h_f64) h_f64[(size_t)tk * inter + n] = h;
            if (h_bf16) h_bf16[(size_t)tk * inter + n] = orc_f64_to_bf16(h);
        }
    }
    free(xin);
    free(rs);
    free(t);
    return ORC_OK;
}

/*
 * Down projection with residual (Sec. 3.3: down stays at 4 bits):
 *   y[m,c] = residual[m,c] + sum_n h[m,n] deq(Wd)[c,n]
 * h: [m, inter] bf16.  Wd: [d, inter] codes, [d, inter/group] scales/zeros.
 * residual: [m, d] bf16 or NULL.  y_f64 / y_bf16 optional outputs.
 */
int orc_down(const uint16_t *h, int m, int inter, int d,
             const uint8_t *qd, const uint16_t *sd, const uint16_t *zd, int group,
             const uint16_t *residual, double *y_f64, uint16_t *y_bf16)
{
    if (m < 0 || d <= 0 || inter <= 0 || group <= 0 || inter % group != 0) return ORC_ERR_ARG;
    const int ng = inter / group;
#pragma omp parallel for schedule(static)
    for (int c = 0; c < d; ++c) {
        for (int tk = 0; tk < m; ++tk) {
            double y = orc_qdot(qd + (size_t)c * inter, sd + (size_t)c * ng, zd + (size_t)c * ng,
                                inter, group, h + (size_t)tk * inter);
            if (residual) y += orc_bf16_to_f64(residual[(size_t)tk * d + c]);
            if (y_f64) y_f64[(size_t)tk * d + c] = y;
            if (y_bf16) y_bf16[(size_t)tk * d + c] = orc_f64_to_bf16(y);
        }
    }
    return ORC_OK;
}

/*
 * bf16 down projection with residual: the down layer of the BF16/W2-GateUp
 * configuration of the accuracy experiments (Sec. 6.1 keeps every layer but
 * gate/up in BF16; Sec. 7 names it beside the deployed W4/W2-GateUp form):
 *   y[m,c] = residual[m,c] + sum_n h[m,n] Wd[c,n]
 * h: [m, inter] bf16.  Wd: [d, inter] bf16 row-major.  residual: [m, d] bf16
 * or NULL.  fp64 sum over n in ascending order; y_f64 / y_bf16 optional.
 */
int orc_down_bf16(const uint16_t *h, int m, int inter, int d, const uint16_t *wd,
                  const uint16_t *residual, double *y_f64, uint16_t *y_bf16)
{
    if (m < 0 || d <= 0 || inter <= 0) return ORC_ERR_ARG;
#pragma omp parallel for schedule(static)
    for (int c = 0; c < d; ++c) {
        for (int tk = 0; tk < m; ++tk) {
            double y = 0.0;
            for (int n = 0; n < inter; ++n)
                y += orc_bf16_to_f64(h[(size_t)tk * inter + n]) * orc_bf16_to_f64(wd[(size_t)c * inter + n]);
            if (residual) y += orc_bf16_to_f64(residual[(size_t)tk * d + c]);
            if (y_f64) y_f64[(size_t)tk * d + c] = y;
            if (y_bf16) y_bf16[(size_t)tk * d + c] = orc_f64_to_bf16(y);
        }
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------ */
/* Decode-step attention (the rest of a decoder layer; the paper's     */
/* throughput analysis, Sec. 5, counts its KV-cache reads among the     */
/* operators whose cost does not depend on the weight precision).       */
/* ------------------------------------------------------------------ */

/*
 * Rotary position embedding of heads of dimension hd (even) at position pos,
 * pairing element i with element i + hd/2 ("rotate half" convention):
 *   a = pos * theta^(-2i/hd),
 *   x'[i]        = x[i] cos a - x[i + hd/2] sin a
 *   x'[i + hd/2] = x[i + hd/2] cos a + x[i] sin a,     i < hd/2.
 * x: fp64 [n_heads, hd], rotated in place.
 */
int orc_rope(double *x, int n_heads, int hd, long pos, double theta)
{
    if (n_heads < 0 || hd <= 0 || hd % 2 != 0 || theta <= 0.0) return ORC_ERR_ARG;
    const int half = hd / 2;
    for (int h = 0; h < n_heads; ++h) {
        double *v = x + (size_t)h * hd;
        for (int i = 0; i < half; ++i) {
            const double a = (double)pos * pow(theta, -2.0 * i / hd);
            const double c = cos(a), s = sin(a);
            const double x0 = v[i], x1 = v[i + half];
            v[i] = x0 * c - x1 * s;
            v[i + half] = x1 * c + x0 * s;
        }
    }
    return ORC_OK;
}

/*
 * One decode step of grouped-query attention over a bf16 KV cache: for each
 * sequence b and query head h (kv head g = h / (n_heads / n_kv)),
 *   s[j] = (q[b,h] . K[b,g,j]) / sqrt(hd),   j < len[b],
 *   p    = softmax(s),   o[b,h] = sum_j p[j] V[b,g,j].
 * q: fp64 [B, n_heads, hd].  K, V: bf16 [B, n_kv, max_len, hd].  len: [B],
 * 1 <= len[b] <= max_len.  o: fp64 [B, n_heads, hd].  The softmax subtracts
 * max s before exponentiating (the same value in exact arithmetic).
 */
int orc_attn_decode(const double *q, const uint16_t *k_cache, const uint16_t *v_cache, const int *len,
                    int batch, int n_heads, int n_kv, int hd, int max_len, double *o)
{
    if (batch < 0 || n_heads <= 0 || n_kv <= 0 || n_heads % n_kv != 0 || hd <= 0 || max_len <= 0)
        return ORC_ERR_ARG;
    for (int b = 0; b < batch; ++b)
        if (len[b] < 1 || len[b] > max_len) return ORC_ERR_ARG;
    const int rep = n_heads / n_kv;
    double *s = (double *)malloc(sizeof(double) * (size_t)max_len);
    if (!s) return ORC_ERR_ARG;
    for (int b = 0; b < batch; ++b)
        for (int h = 0; h < n_heads; ++h) {
            const int g = h / rep;
            const double *qh = q + ((size_t)b * n_heads + h) * hd;
            const uint16_t *kb = k_cache + ((size_t)b * n_kv + g) * max_len * hd;
            const uint16_t *vb = v_cache + ((size_t)b * n_kv + g) * max_len * hd;
            double mx = -INFINITY;
            for (int j = 0; j < len[b]; ++j) {
                double dot = 0.0;
                for (int e = 0; e < hd; ++e) dot += qh[e] * orc_bf16_to_f64(kb[(size_t)j * hd + e]);
                s[j] = dot / sqrt((double)hd);
                if (s[j] > mx) mx = s[j];
            }
            double den = 0.0;
            for (int j = 0; j < len[b]; ++j) {
                s[j] = exp(s[j] - mx);
                den += s[j];
            }
            double *oh = o + ((size_t)b * n_heads + h) * hd;
            for (int e = 0; e < hd; ++e) {
                double acc = 0.0;
                for (int j = 0; j < len[b]; ++j) acc += s[j] * orc_bf16_to_f64(vb[(size_t)j * hd + e]);
                oh[e] = acc / den;
            }
        }
    free(s);
    return ORC_OK;
}

/*
 * Projection of unrounded fp64 inputs through a quantized matrix:
 *   out[t, n] = sum_k x[t, k] deq(W)[n, k],   x: fp64 [m, k], W: [n, k].
 */
int orc_qproj(const double *x, int m, int k, const uint8_t *q, const uint16_t *s, const uint16_t *z,
              int n, int group, double *out)
{
    if (m < 0 || k <= 0 || n <= 0 || group <= 0 || k % group != 0) return ORC_ERR_ARG;
    const int ng = k / group;
#pragma omp parallel for schedule(static)
    for (int r = 0; r < n; ++r)
        for (int t = 0; t < m; ++t)
            out[(size_t)t * n + r] = orc_qdot_f64(q + (size_t)r * k, s + (size_t)r * ng, z + (size_t)r * ng,
                                                  k, group, x + (size_t)t * k);
    return ORC_OK;
}

/* Threads used by the OpenMP loops above (1 without OpenMP). */
int orc_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void orc_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Array forms of the conversions, for the tests' pins. */
void orc_f32_to_f16_array(const float *in, size_t n, uint16_t *out)
{
    for (size_t i = 0; i < n; ++i) out[i] = orc_f32_to_f16(in[i]);
}

void orc_f16_to_f64_array(const uint16_t *in, size_t n, double *out)
{
    for (size_t i = 0; i < n; ++i) out[i] = orc_f16_to_f64(in[i]);
}

void orc_f64_to_bf16_array(const double *in, size_t n, uint16_t *out)
{
    for (size_t i = 0; i < n; ++i) out[i] = orc_f64_to_bf16(in[i]);
}

void orc_bf16_to_f64_array(const uint16_t *in, size_t n, double *out)
{
    for (size_t i = 0; i < n; ++i) out[i] = orc_bf16_to_f64(in[i]);
}
