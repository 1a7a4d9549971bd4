/*
 * mnmt_oracle.c -- plain, slow CPU oracle of the full-INT8 encoder-decoder
 * translation path of MobileNMT (arXiv 2306.04235).
 *
 * TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg load this library.  It shares no code, header or constant
 * generator with the CUDA library: it parses the documented "MNMT v1" blob
 * itself and computes every step with scalar loops, in the paper's order.
 *
 * Build: gcc -std=c11 -O2 -ffp-contract=off -fPIC -shared -pthread -lm.
 * -ffp-contract=off is part of the definition: every a*b+c below is two IEEE
 * fp32 roundings unless written as fmaf().
 *
 * What each function follows:
 *   q8 ................ symmetric uniform quantiser (App. B, Eq. 3/4 with the
 *                       zero point fixed at 0; per-channel weights, per-tensor
 *                       activations; round half to even, clamp [-127, 127])
 *   linear ............ int8 x int8 -> int32 GEMM of every quantised linear
 *                       (Sec. 3.3 "FFN and Attention Quantizers", Fig. 5;
 *                       biases and residuals stay full precision)
 *   layer_norm ........ LayerNorm before each sublayer (App. A, App. D
 *                       "normalization before layers"); post-LN as an option
 *   attend ............ Eq. 1/2 (scaled dot-product attention) per head,
 *                       softmax kept in full precision, V and the context
 *                       quantised (Fig. 5b)
 *   residual .......... learnable weight gamma_i on the residual branch
 *                       (Sec. 3.3, Fig. 5: X -> gamma_i -> add)
 *   ffn ............... Eq. 3, Y = ReLU(X W1 + b1) W2 + b2
 *   embed ............. shared source/target embedding (App. D), optional
 *                       factorisation V*E + E*H (Sec. 2.1 "Scaling E")
 *   greedy / beam ..... greedy search (App. D) and beam search (Table 6 row
 *                       "+Greedy Search" implies beam was the default)
 *   4-bit weights ..... row-wise low-bit quantisation of the attention and
 *                       FFN linears (Sec. 3.3 "lower-bit quantization ...
 *                       row-wise"; the embedding stays 8-bit; Table
 *                       "quantizing weights to lower bits", 4-8-8): per
 *                       output row either a symmetric scale (codes -7..7) or
 *                       the min-max scale and offset of App. B Eq. scale /
 *                       Eq. quant (codes 0..15, offset r_m = the row minimum)
 *
 * Where the paper is silent (rounding ties, LN epsilon and arithmetic,
 * softmax arithmetic, exp/log, beam details) the reading implemented here is
 * the fixed-point, order-free one: LN sums and softmax weights are exact
 * integers, so any summation order gives the same bits.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_EINVAL (-1)
#define OR_ENOMEM (-2)
#define OR_EFORMAT (-5)
#define OR_EOVERFLOW (-6)

/* ------------------------------------------------------------------------ */
/* model description parsed from the blob                                   */
/* ------------------------------------------------------------------------ */
typedef struct {
    int n_enc, n_dec, d, H, F, V, E, pre_ln, tied, max_pos, pad, bos, eos;
} ocfg;

/* A linear: int8 codes w [n][k] (bits 8), or 4-bit codes packed two per byte
 * in wp (bits 4; see lin_code), with per-row scale s, bias b and, for the
 * min-max form (asym), per-row offset m. */
typedef struct { const int8_t *w; const uint8_t *wp; const float *s, *b, *m; int n, k, bits, asym; } olin;
typedef struct { const float *g, *b; } oln;
typedef struct { oln ln; float s_in, s_q, s_k, s_v, s_ctx, gamma; olin qkv, o; } oself;
typedef struct { oln ln; float s_in, s_q, s_k, s_v, s_ctx, gamma; olin q, kv, o; } ocross;
typedef struct { oln ln; float s_in, s_h, gamma; olin w1, w2; } offn;

typedef struct {
    ocfg c;
    int wq;
    const int8_t *emb_q;
    const float *emb_s;
    int factorised;
    olin proj;
    float emb_scale, s_enc, s_dout;
    const float *pe;
    oself enc_self[64];
    offn enc_ffn[64];
    oln enc_final;
    oself dec_self[64];
    ocross dec_cross[64];
    offn dec_ffn[64];
    oln dec_final;
    olin out;
} omodel;

typedef struct { const uint8_t *base; size_t off, size; int bad; } cursor;

static const void *take(cursor *cu, size_t bytes) {
    if (cu->bad || cu->off + bytes > cu->size) { cu->bad = 1; return NULL; }
    const void *p = cu->base + cu->off;
    cu->off += bytes;
    cu->off = (cu->off + 15) & ~(size_t)15; /* every array starts 16-byte aligned */
    if (cu->off > cu->size) cu->off = cu->size;
    return p;
}

/* weight format of the blob's linears: 8 = int8 symmetric per row, 4 =
 * int4 symmetric per row, 4 | WQ_ASYM = int4 min-max per row */
#define WQ_ASYM 0x100
static olin take_lin_q(cursor *cu, int n, int k, int wq) {
    olin l;
    memset(&l, 0, sizeof(l));
    l.n = n; l.k = k;
    l.bits = wq & 0xFF;
    l.asym = (wq & WQ_ASYM) != 0;
    if (l.bits == 4) {
        l.wp = (const uint8_t *)take(cu, (size_t)n * k / 2);
    } else {
        l.w = (const int8_t *)take(cu, (size_t)n * k);
    }
    l.s = (const float *)take(cu, (size_t)n * 4);
    if (l.asym) l.m = (const float *)take(cu, (size_t)n * 4);
    l.b = (const float *)take(cu, (size_t)n * 4);
    return l;
}

static oln take_ln(cursor *cu, int d) {
    oln l;
    l.g = (const float *)take(cu, (size_t)d * 4);
    l.b = (const float *)take(cu, (size_t)d * 4);
    return l;
}

static int parse(const void *blob, size_t bytes, omodel *m) {
    memset(m, 0, sizeof(*m));
    if (bytes < 64) return OR_EFORMAT;
    const uint8_t *p = (const uint8_t *)blob;
    if (memcmp(p, "MNMT", 4) != 0) return OR_EFORMAT;
    uint32_t ver;
    memcpy(&ver, p + 4, 4);
    if (ver != 1 && ver != 2) return OR_EFORMAT;
    int32_t h[13];
    memcpy(h, p + 8, sizeof(h));
    int32_t wq = 8; /* version 2 names the linears' weight format at byte 60 */
    if (ver == 2) memcpy(&wq, p + 60, 4);
    if (wq != 8 && wq != 4 && wq != (4 | WQ_ASYM)) return OR_EFORMAT;
    m->wq = wq;
    ocfg *c = &m->c;
    c->n_enc = h[0]; c->n_dec = h[1]; c->d = h[2]; c->H = h[3]; c->F = h[4]; c->V = h[5];
    c->E = h[6]; c->pre_ln = h[7]; c->tied = h[8]; c->max_pos = h[9];
    c->pad = h[10]; c->bos = h[11]; c->eos = h[12];
    if (c->n_enc < 1 || c->n_enc > 64 || c->n_dec < 1 || c->n_dec > 64) return OR_EFORMAT;
    if (c->d < 16 || c->d > 2048 || c->H < 1 || c->d % c->H || c->F < 1 || c->V < 4 || c->E < 1 || c->E > c->d)
        return OR_EFORMAT;
    if (c->tied && c->E != c->d) return OR_EFORMAT;
    if (c->max_pos < 1) return OR_EFORMAT;
    int d = c->d, F = c->F, V = c->V, E = c->E;
    if (wq != 8 && (d % 32 || F % 32)) return OR_EFORMAT; /* 32-code chunks */
    cursor cu = {p, 64, bytes, 0};
    m->emb_q = (const int8_t *)take(&cu, (size_t)V * E);
    m->emb_s = (const float *)take(&cu, (size_t)V * 4);
    m->factorised = (E != d);
    /* the embedding (its table, factorised projection and an untied output
     * projection: the "E" of W-E-A) stays 8-bit whatever the linears' format */
    if (m->factorised) m->proj = take_lin_q(&cu, d, E, 8);
    const float *gl = (const float *)take(&cu, 16);
    m->pe = (const float *)take(&cu, (size_t)c->max_pos * d * 4);
    for (int l = 0; l < c->n_enc; l++) {
        oself *a = &m->enc_self[l];
        a->ln = take_ln(&cu, d);
        const float *s = (const float *)take(&cu, 32);
        a->qkv = take_lin_q(&cu, 3 * d, d, wq);
        a->o = take_lin_q(&cu, d, d, wq);
        if (s) { a->s_in = s[0]; a->s_q = s[1]; a->s_k = s[2]; a->s_v = s[3]; a->s_ctx = s[4]; a->gamma = s[5]; }
        offn *f = &m->enc_ffn[l];
        f->ln = take_ln(&cu, d);
        s = (const float *)take(&cu, 16);
        f->w1 = take_lin_q(&cu, F, d, wq);
        f->w2 = take_lin_q(&cu, d, F, wq);
        if (s) { f->s_in = s[0]; f->s_h = s[1]; f->gamma = s[2]; }
    }
    if (c->pre_ln) m->enc_final = take_ln(&cu, d);
    for (int l = 0; l < c->n_dec; l++) {
        oself *a = &m->dec_self[l];
        a->ln = take_ln(&cu, d);
        const float *s = (const float *)take(&cu, 32);
        a->qkv = take_lin_q(&cu, 3 * d, d, wq);
        a->o = take_lin_q(&cu, d, d, wq);
        if (s) { a->s_in = s[0]; a->s_q = s[1]; a->s_k = s[2]; a->s_v = s[3]; a->s_ctx = s[4]; a->gamma = s[5]; }
        ocross *x = &m->dec_cross[l];
        x->ln = take_ln(&cu, d);
        s = (const float *)take(&cu, 32);
        x->q = take_lin_q(&cu, d, d, wq);
        x->kv = take_lin_q(&cu, 2 * d, d, wq);
        x->o = take_lin_q(&cu, d, d, wq);
        if (s) { x->s_in = s[0]; x->s_q = s[1]; x->s_k = s[2]; x->s_v = s[3]; x->s_ctx = s[4]; x->gamma = s[5]; }
        offn *f = &m->dec_ffn[l];
        f->ln = take_ln(&cu, d);
        s = (const float *)take(&cu, 16);
        f->w1 = take_lin_q(&cu, F, d, wq);
        f->w2 = take_lin_q(&cu, d, F, wq);
        if (s) { f->s_in = s[0]; f->s_h = s[1]; f->gamma = s[2]; }
    }
    if (c->pre_ln) m->dec_final = take_ln(&cu, d);
    m->out.n = V; m->out.k = d;
    if (c->tied) {
        /* the output projection is the 8-bit embedding table (the "E" of W-E-A) */
        m->out.bits = 8;
        m->out.w = m->emb_q;
        m->out.s = m->emb_s;
    } else {
        m->out = take_lin_q(&cu, V, d, 8);
    }
    if (c->tied) m->out.b = (const float *)take(&cu, (size_t)V * 4);
    if (cu.bad || cu.off != bytes) return OR_EFORMAT;
    m->emb_scale = gl[0]; m->s_enc = gl[1]; m->s_dout = gl[2];
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* scalar building blocks                                                    */
/* ------------------------------------------------------------------------ */

/* Symmetric 8-bit quantiser (App. B, Eq. 3/4 with r_m = 0): code of x at
 * scale s given inv = fl(1/s); round to nearest, ties to even; clamp to the
 * symmetric range [-127, 127]. */
static int8_t q8(float x, float inv) {
    float t = x * inv;
    t = rintf(t);
    if (t > 127.0f) t = 127.0f;
    if (t < -127.0f) t = -127.0f;
    return (int8_t)t;
}

/* int32 dot product of two int8 vectors: the integer GEMM of Sec. 4.1. */
static int32_t dot_i8(const int8_t *a, const int8_t *w, int k) {
    int32_t s = 0;
    for (int i = 0; i < k; i++) s += (int32_t)a[i] * (int32_t)w[i];
    return s;
}

/* Dequantise then add the full-precision bias (Fig. 5: matmul output red,
 * bias add black): y = fl(fl(acc * fl(s_x * s_w[n])) + b[n]). */
static float dequant_bias(int32_t acc, float s_x, float s_w, float b) {
    float sc = s_x * s_w;
    float t = (float)acc * sc;
    return t + b;
}

/* The 4-bit code of weight (n, k): the codes of a row are packed in chunks of
 * 32 codes held in 16 bytes, code j of a chunk in the low nibble of byte j
 * (j < 16) or the high nibble of byte j - 16.  Symmetric rows store v + 8 for
 * a code v in [-7, 7]; min-max rows store u in [0, 15]. */
static int lin_code(const olin *L, int n, int k) {
    const uint8_t byte = L->wp[(size_t)n * L->k / 2 + (size_t)(k / 32) * 16 + (k % 32) % 16];
    return (k % 32) < 16 ? (byte & 15) : (byte >> 4);
}

/* Output n of a quantised linear on the int8 row a at activation scale s_x.
 *   8-bit and 4-bit symmetric rows (codes v): the dequant-then-bias of
 *     dequant_bias on the exact integer sum of a_k v_nk.
 *   4-bit min-max rows, W_nk = s_n u_nk + r_n (App. B Eq. quant with the row
 *     minimum r_n as offset): x W_n = s_x (s_n sum a_k u_nk + r_n sum a_k)
 *     exactly, so with the two integer sums A_u and A_1,
 *     y = fl(fl(fl(A_u fl(s_x s_n)) + fl(A_1 fl(s_x r_n))) + b_n). */
static float lin_out(const olin *L, int n, const int8_t *a, float s_x) {
    if (L->bits == 8) return dequant_bias(dot_i8(a, L->w + (size_t)n * L->k, L->k), s_x, L->s[n], L->b[n]);
    int32_t acc = 0, a1 = 0;
    for (int k = 0; k < L->k; k++) {
        int u = lin_code(L, n, k);
        acc += (int32_t)a[k] * (L->asym ? u : u - 8);
        a1 += a[k];
    }
    if (!L->asym) return dequant_bias(acc, s_x, L->s[n], L->b[n]);
    float sc = s_x * L->s[n];
    float mc = s_x * L->m[n];
    float t = (float)acc * sc;
    float o = (float)a1 * mc;
    float y = t + o;
    return y + L->b[n];
}

/* Quantised linear on one row: y[n] for n in [0, N). */
static void linear_row(const int8_t *a, float s_x, const olin *L, float *y) {
    for (int n = 0; n < L->n; n++) y[n] = lin_out(L, n, a, s_x);
}

/* Nearest float (ties to even) to the exact value s 2^e / d, |s| < 2^63,
 * 1 <= d <= 2048.  For a power-of-two d the long double quotient (64-bit
 * significand on x86, 113-bit on Arm) is exact.  Otherwise s 2^e / d is
 * either a midpoint between two floats (then the quotient, an odd multiple of
 * a power of two with at most 26 significant bits, is exact in long double
 * too) or at least 2^-36 (relative) away from every midpoint (its distance
 * to M 2^E is a nonzero multiple of 2^E / d, and M < 2^25, d < 2^11), while
 * the long double quotient is within 2^-64 of it: either way the one rounding
 * to float is the correct rounding of the exact value, subnormals included. */
static float rn32_scaled(int64_t s, int e, int d) {
    return (float)(ldexpl((long double)s, e) / (long double)d);
}

/* Nearest float (ties to even) to the exact quotient n / z of integers with
 * |n| < 2^62 and 1 <= z < 2^35.  If n/z is not itself a midpoint M 2^E between
 * two floats (M odd, < 2^26), it lies at least 2^-60 (relative) away from
 * every midpoint, while the long double quotient is within 2^-64 of n/z; so
 * the long double quotient rounds to float exactly as n/z does (and a
 * midpoint quotient is computed exactly, ties going to even). */
static float rn32_quotient(int64_t n, int64_t z) {
    return (float)((long double)n / (long double)z);
}

/* LayerNorm (App. A / App. D).  The paper fixes neither epsilon nor the
 * arithmetic; this reading makes the mean and the (biased, divide-by-d)
 * variance exact fixed-point sums, so their value does not depend on the
 * summation order, each rounded once to fp32.  Each sum is taken on a grid
 * set by the row's own largest magnitude (an order-free maximum): with
 * 2^ea > max|r_i| every term r_i 2^(52-ea) is below 2^52, and with
 * 2^eb > max|c_i| every c_i^2 2^(52-2eb) is below 2^52, so d <= 2048 terms
 * cannot overflow int64 and every term keeps its leading 24+ bits.
 * rstd = 1 / sqrt(var + 1e-5) in IEEE fp32.  |r_i| >= 2^32 is rejected. */
static int ln_stats(const float *r, int d, float *mu_out, float *var_out) {
    float amax = 0.0f;
    for (int i = 0; i < d; i++) {
        float v = fabsf(r[i]);
        if (!(v < 0x1p32f)) return OR_EOVERFLOW;
        if (v > amax) amax = v;
    }
    int ea = 0;
    if (amax > 0.0f) frexpf(amax, &ea);
    int64_t s1 = 0;
    for (int i = 0; i < d; i++) s1 += llrint(ldexp((double)r[i], 52 - ea));
    float mu = rn32_scaled(s1, ea - 52, d);
    float bmax = 0.0f;
    for (int i = 0; i < d; i++) {
        float v = fabsf(r[i] - mu);
        if (v > bmax) bmax = v;
    }
    int eb = 0;
    if (bmax > 0.0f) frexpf(bmax, &eb);
    int64_t s2 = 0;
    for (int i = 0; i < d; i++) {
        float c = r[i] - mu;
        float c2 = c * c;
        s2 += llrint(ldexp((double)c2, 52 - 2 * eb));
    }
    float var = rn32_scaled(s2, 2 * eb - 52, d);
    *mu_out = mu;
    *var_out = var;
    return OR_OK;
}

static int layer_norm(const float *r, int d, const oln *ln, float *out) {
    float mu, var;
    int st = ln_stats(r, d, &mu, &var);
    if (st) return st;
    float rstd = 1.0f / sqrtf(var + 1e-5f);
    for (int i = 0; i < d; i++) {
        float c = r[i] - mu;
        float t = c * rstd;
        t = t * ln->g[i];
        out[i] = t + ln->b[i];
    }
    return OR_OK;
}

/* e^x for x <= 0, written from the mathematics: Cody-Waite reduction
 * x = n ln2 + r with ln2 split into a 16-bit head and a tail, then the
 * degree-7 Taylor polynomial of e^r by Horner's rule in fused multiply-adds,
 * scaled by 2^n through the exponent field.  Returns 0 below -87 (under the
 * smallest normal float). */
static float exp_own(float x) {
    if (x < -87.0f) return 0.0f;
    float n = rintf(x * 0x1.715476p+0f);
    float r = fmaf(-n, 0x1.62e4p-1f, x);
    r = fmaf(-n, 0x1.7f7d1cp-20f, r);
    float p = 0x1.a01a02p-13f;          /* 1/7! */
    p = fmaf(p, r, 0x1.6c16c2p-10f);    /* 1/6! */
    p = fmaf(p, r, 0x1.111112p-7f);     /* 1/5! */
    p = fmaf(p, r, 0x1.555556p-5f);     /* 1/4! */
    p = fmaf(p, r, 0x1.555556p-3f);     /* 1/3! */
    p = fmaf(p, r, 0.5f);               /* 1/2! */
    p = fmaf(p, r, 1.0f);
    p = fmaf(p, r, 1.0f);
    int ni = (int)n;                    /* in [-126, 0] */
    uint32_t bits = (uint32_t)(ni + 127) << 23;
    float two_n;
    memcpy(&two_n, &bits, 4);
    return p * two_n;
}

/* natural log in double for z >= 1, from the mathematics: z = f 2^k with
 * f in [sqrt(1/2), sqrt(2)), ln f = 2 atanh(s), s = (f-1)/(f+1), by the odd
 * series in s up to s^23 (|s| <= 0.1716, so the tail is below 1e-18). */
static double log_own(double z) {
    int k;
    double f = frexp(z, &k);
    if (f < 0x1.6a09e667f3bcdp-1) { f = f * 2.0; k = k - 1; }
    double s = (f - 1.0) / (f + 1.0);
    double s2 = s * s;
    double q = 0x1.642c8590b2164p-5;    /* 1/23 */
    q = q * s2 + 0x1.8618618618618p-5;  /* 1/21 */
    q = q * s2 + 0x1.af286bca1af28p-5;  /* 1/19 */
    q = q * s2 + 0x1.e1e1e1e1e1e1ep-5;  /* 1/17 */
    q = q * s2 + 0x1.1111111111111p-4;  /* 1/15 */
    q = q * s2 + 0x1.3b13b13b13b14p-4;  /* 1/13 */
    q = q * s2 + 0x1.745d1745d1746p-4;  /* 1/11 */
    q = q * s2 + 0x1.c71c71c71c71cp-4;  /* 1/9 */
    q = q * s2 + 0x1.2492492492492p-3;  /* 1/7 */
    q = q * s2 + 0x1.999999999999ap-3;  /* 1/5 */
    q = q * s2 + 0x1.5555555555555p-2;  /* 1/3 */
    q = q * s2 + 1.0;
    return (2.0 * s) * q + (double)k * 0x1.62e42fefa39efp-1;
}

/* One attention head (Eq. 1/2).  Scores are int32 dot products of int8 q and
 * keys, scaled by sigma = fl32(s_q s_k / sqrt(d_h)); the softmax stays in full
 * precision as fixed-point weights E_j = rne(exp(s_j - max) * 2^24); the
 * context is the nearest float to the exact integer sum of E_j v_j over the
 * exact sum of E_j, in units of V's codes, then requantised with
 * rho = fl(s_v / s_ctx). */
static void attend(const int8_t *q, const int8_t *const *keys, const int8_t *const *vals,
                   int n, int dh, float sigma, float rho, int8_t *out, float *sbuf,
                   int64_t *nbuf) {
    float m = -INFINITY;
    for (int j = 0; j < n; j++) {
        sbuf[j] = (float)dot_i8(q, keys[j], dh) * sigma;
        if (sbuf[j] > m) m = sbuf[j];
    }
    int64_t Z = 0;
    for (int e = 0; e < dh; e++) nbuf[e] = 0;
    for (int j = 0; j < n; j++) {
        float ex = exp_own(sbuf[j] - m);
        int64_t Ej = (int64_t)rintf(ex * 16777216.0f);
        Z += Ej;
        for (int e = 0; e < dh; e++) nbuf[e] += Ej * (int64_t)vals[j][e];
    }
    for (int e = 0; e < dh; e++) {
        float ctx = rn32_quotient(nbuf[e], Z);
        out[e] = q8(ctx, rho);
    }
}

static float sigma_of(float s_q, float s_k, int dh) {
    return (float)((double)s_q * (double)s_k / sqrt((double)dh));
}

/* Embedding of one token at one position (shared src/tgt table, App. D):
 * x = fl(fl(dequant(Eq[id]) * sqrt(d)) + PE[pos]); with factorisation the
 * E-dim int8 row feeds the E->d linear directly, its per-row scale folded
 * into the dequantisation (Sec. 2.1 "Scaling E"). */
static void embed(const omodel *m, int id, int pos, float *x) {
    const ocfg *c = &m->c;
    const int8_t *row = m->emb_q + (size_t)id * c->E;
    const float *pe = m->pe + (size_t)pos * c->d;
    if (!m->factorised) {
        for (int i = 0; i < c->d; i++) {
            float t = (float)row[i] * m->emb_s[id];
            t = t * m->emb_scale;
            x[i] = t + pe[i];
        }
    } else {
        for (int n = 0; n < c->d; n++) {
            float y = lin_out(&m->proj, n, row, m->emb_s[id]);
            float t = y * m->emb_scale;
            x[n] = t + pe[n];
        }
    }
}

/* residual with the learnable weight on the residual branch:
 * r = fl(fl(gamma * r) + y) */
static void residual(float *r, const float *y, float gamma, int d) {
    for (int i = 0; i < d; i++) {
        float t = gamma * r[i];
        r[i] = t + y[i];
    }
}

/* Sublayer input: q8(LN(r)) before the sublayer (pre-LN) or q8(r) (post-LN). */
static int sub_input(const omodel *m, const float *r, const oln *ln, float s_in, int8_t *a,
                     float *tmp) {
    int d = m->c.d;
    float inv = 1.0f / s_in;
    if (m->c.pre_ln) {
        int st = layer_norm(r, d, ln, tmp);
        if (st) return st;
        for (int i = 0; i < d; i++) a[i] = q8(tmp[i], inv);
    } else {
        for (int i = 0; i < d; i++) a[i] = q8(r[i], inv);
    }
    return OR_OK;
}

/* After the residual add: post-LN normalises the stream in place. */
static int sub_output(const omodel *m, float *r, const oln *ln, float *tmp) {
    if (m->c.pre_ln) return OR_OK;
    int st = layer_norm(r, m->c.d, ln, tmp);
    if (st) return st;
    memcpy(r, tmp, sizeof(float) * m->c.d);
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* encoder                                                                   */
/* ------------------------------------------------------------------------ */
typedef struct {
    int S;              /* padded rows */
    int len;            /* valid rows */
    int8_t *enc_q;      /* [S][d]  quantised encoder output (scale s_enc) */
    int8_t *ck, *cv;    /* [n_dec][S][d]  cross-attention keys / values */
} oenc;

static int encode_one(const omodel *m, const int32_t *src, int len, int S, oenc *out) {
    const ocfg *c = &m->c;
    int d = c->d, dh = d / c->H, F = c->F;
    if (len < 1 || len > S || S > c->max_pos) return OR_EINVAL;
    float *r = malloc(sizeof(float) * S * d);
    int8_t *a = malloc((size_t)S * (d > F ? d : F) + 64);
    int8_t *qkv = malloc((size_t)S * 3 * d);
    int8_t *ctx = malloc((size_t)S * d);
    float *y = malloc(sizeof(float) * (3 * d > F ? 3 * d : F));
    float *tmp = malloc(sizeof(float) * d);
    float *sbuf = malloc(sizeof(float) * S);
    int64_t *nbuf = malloc(sizeof(int64_t) * dh);
    const int8_t **kp = malloc(sizeof(void *) * S), **vp = malloc(sizeof(void *) * S);
    int st = OR_OK;
    if (!r || !a || !qkv || !ctx || !y || !tmp || !sbuf || !nbuf || !kp || !vp) { st = OR_ENOMEM; goto done; }
    for (int s = 0; s < S; s++) {
        int id = src[s];
        if (id < 0 || id >= c->V) { st = OR_EINVAL; goto done; }
        embed(m, id, s, r + (size_t)s * d);
    }
    for (int l = 0; l < c->n_enc; l++) {
        const oself *A = &m->enc_self[l];
        float iq = 1.0f / A->s_q, ik = 1.0f / A->s_k, iv = 1.0f / A->s_v;
        for (int s = 0; s < S; s++) {
            if ((st = sub_input(m, r + (size_t)s * d, &A->ln, A->s_in, a, tmp))) goto done;
            linear_row(a, A->s_in, &A->qkv, y);
            for (int n = 0; n < d; n++) {
                qkv[(size_t)s * 3 * d + n] = q8(y[n], iq);
                qkv[(size_t)s * 3 * d + d + n] = q8(y[d + n], ik);
                qkv[(size_t)s * 3 * d + 2 * d + n] = q8(y[2 * d + n], iv);
            }
        }
        float sigma = sigma_of(A->s_q, A->s_k, dh), rho = A->s_v / A->s_ctx;
        for (int s = 0; s < S; s++)
            for (int h = 0; h < c->H; h++) {
                for (int j = 0; j < len; j++) { /* key padding mask: j < len */
                    kp[j] = qkv + (size_t)j * 3 * d + d + h * dh;
                    vp[j] = qkv + (size_t)j * 3 * d + 2 * d + h * dh;
                }
                attend(qkv + (size_t)s * 3 * d + h * dh, kp, vp, len, dh, sigma, rho,
                       ctx + (size_t)s * d + h * dh, sbuf, nbuf);
            }
        for (int s = 0; s < S; s++) {
            linear_row(ctx + (size_t)s * d, A->s_ctx, &A->o, y);
            residual(r + (size_t)s * d, y, A->gamma, d);
            if ((st = sub_output(m, r + (size_t)s * d, &A->ln, tmp))) goto done;
        }
        const offn *Fb = &m->enc_ffn[l];
        float ih = 1.0f / Fb->s_h;
        for (int s = 0; s < S; s++) {
            if ((st = sub_input(m, r + (size_t)s * d, &Fb->ln, Fb->s_in, a, tmp))) goto done;
            linear_row(a, Fb->s_in, &Fb->w1, y);
            for (int n = 0; n < F; n++) a[n] = q8(y[n] > 0.0f ? y[n] : 0.0f, ih);
            linear_row(a, Fb->s_h, &Fb->w2, y);
            residual(r + (size_t)s * d, y, Fb->gamma, d);
            if ((st = sub_output(m, r + (size_t)s * d, &Fb->ln, tmp))) goto done;
        }
    }
    {
        float ie = 1.0f / m->s_enc;
        for (int s = 0; s < S; s++) {
            const float *src_row = r + (size_t)s * d;
            if (c->pre_ln) {
                if ((st = layer_norm(src_row, d, &m->enc_final, tmp))) goto done;
                src_row = tmp;
            }
            for (int i = 0; i < d; i++) out->enc_q[(size_t)s * d + i] = q8(src_row[i], ie);
        }
        for (int l = 0; l < c->n_dec; l++) {
            const ocross *X = &m->dec_cross[l];
            float ik = 1.0f / X->s_k, iv = 1.0f / X->s_v;
            for (int s = 0; s < S; s++) {
                linear_row(out->enc_q + (size_t)s * d, m->s_enc, &X->kv, y);
                for (int n = 0; n < d; n++) {
                    out->ck[((size_t)l * S + s) * d + n] = q8(y[n], ik);
                    out->cv[((size_t)l * S + s) * d + n] = q8(y[d + n], iv);
                }
            }
        }
    }
done:
    free(r); free(a); free(qkv); free(ctx); free(y); free(tmp); free(sbuf); free(nbuf);
    free((void *)kp); free((void *)vp);
    return st;
}

/* ------------------------------------------------------------------------ */
/* decoder: one incremental step of one hypothesis                           */
/* ------------------------------------------------------------------------ */
typedef struct {
    int T;            /* capacity (positions) */
    int8_t *k, *v;    /* [n_dec][T][d] self-attention cache of this hypothesis */
} ocache;

typedef struct {
    float *r, *y, *tmp, *sbuf;
    int8_t *a, *q, *ctx;
    int64_t *nbuf;
    const int8_t **kp, **vp;
} oscratch;

static int scratch_init(oscratch *w, const ocfg *c, int nkeys) {
    int d = c->d, F = c->F, big = 3 * d > F ? 3 * d : F;
    w->r = malloc(sizeof(float) * d);
    w->y = malloc(sizeof(float) * (big > c->V ? big : c->V));
    w->tmp = malloc(sizeof(float) * d);
    w->sbuf = malloc(sizeof(float) * nkeys);
    w->a = malloc((size_t)big);
    w->q = malloc((size_t)d);
    w->ctx = malloc((size_t)d);
    w->nbuf = malloc(sizeof(int64_t) * (d / c->H));
    w->kp = malloc(sizeof(void *) * nkeys);
    w->vp = malloc(sizeof(void *) * nkeys);
    if (!w->r || !w->y || !w->tmp || !w->sbuf || !w->a || !w->q || !w->ctx || !w->nbuf || !w->kp || !w->vp)
        return OR_ENOMEM;
    return OR_OK;
}

static void scratch_free(oscratch *w) {
    free(w->r); free(w->y); free(w->tmp); free(w->sbuf); free(w->a); free(w->q); free(w->ctx);
    free(w->nbuf); free((void *)w->kp); free((void *)w->vp);
}

/* Runs the decoder for token `tok` at position t, appending K/V at t to the
 * hypothesis's cache, and writes the vocabulary logits (fp32, [V]) into
 * logits.  If dec_q is non-NULL it receives the quantised decoder output. */
static int decode_step(const omodel *m, const oenc *enc, ocache *cache, int tok, int t,
                       oscratch *w, float *logits, int8_t *dec_q) {
    const ocfg *c = &m->c;
    int d = c->d, dh = d / c->H, F = c->F;
    int st;
    if (t >= cache->T || t >= c->max_pos || tok < 0 || tok >= c->V) return OR_EINVAL;
    embed(m, tok, t, w->r);
    for (int l = 0; l < c->n_dec; l++) {
        /* self-attention over positions 0..t (causal by construction) */
        const oself *A = &m->dec_self[l];
        if ((st = sub_input(m, w->r, &A->ln, A->s_in, w->a, w->tmp))) return st;
        linear_row(w->a, A->s_in, &A->qkv, w->y);
        float iq = 1.0f / A->s_q, ik = 1.0f / A->s_k, iv = 1.0f / A->s_v;
        int8_t *kt = cache->k + ((size_t)l * cache->T + t) * d;
        int8_t *vt = cache->v + ((size_t)l * cache->T + t) * d;
        for (int n = 0; n < d; n++) {
            w->q[n] = q8(w->y[n], iq);
            kt[n] = q8(w->y[d + n], ik);
            vt[n] = q8(w->y[2 * d + n], iv);
        }
        float sigma = sigma_of(A->s_q, A->s_k, dh), rho = A->s_v / A->s_ctx;
        for (int h = 0; h < c->H; h++) {
            for (int j = 0; j <= t; j++) {
                w->kp[j] = cache->k + ((size_t)l * cache->T + j) * d + h * dh;
                w->vp[j] = cache->v + ((size_t)l * cache->T + j) * d + h * dh;
            }
            attend(w->q + h * dh, w->kp, w->vp, t + 1, dh, sigma, rho, w->ctx + h * dh, w->sbuf,
                   w->nbuf);
        }
        linear_row(w->ctx, A->s_ctx, &A->o, w->y);
        residual(w->r, w->y, A->gamma, d);
        if ((st = sub_output(m, w->r, &A->ln, w->tmp))) return st;

        /* cross-attention over the source keys j < len */
        const ocross *X = &m->dec_cross[l];
        if ((st = sub_input(m, w->r, &X->ln, X->s_in, w->a, w->tmp))) return st;
        linear_row(w->a, X->s_in, &X->q, w->y);
        float iqx = 1.0f / X->s_q;
        for (int n = 0; n < d; n++) w->q[n] = q8(w->y[n], iqx);
        float sx = sigma_of(X->s_q, X->s_k, dh), rx = X->s_v / X->s_ctx;
        for (int h = 0; h < c->H; h++) {
            for (int j = 0; j < enc->len; j++) {
                w->kp[j] = enc->ck + ((size_t)l * enc->S + j) * d + h * dh;
                w->vp[j] = enc->cv + ((size_t)l * enc->S + j) * d + h * dh;
            }
            attend(w->q + h * dh, w->kp, w->vp, enc->len, dh, sx, rx, w->ctx + h * dh, w->sbuf,
                   w->nbuf);
        }
        linear_row(w->ctx, X->s_ctx, &X->o, w->y);
        residual(w->r, w->y, X->gamma, d);
        if ((st = sub_output(m, w->r, &X->ln, w->tmp))) return st;

        /* FFN */
        const offn *Fb = &m->dec_ffn[l];
        if ((st = sub_input(m, w->r, &Fb->ln, Fb->s_in, w->a, w->tmp))) return st;
        linear_row(w->a, Fb->s_in, &Fb->w1, w->y);
        float ih = 1.0f / Fb->s_h;
        for (int n = 0; n < F; n++) w->a[n] = q8(w->y[n] > 0.0f ? w->y[n] : 0.0f, ih);
        linear_row(w->a, Fb->s_h, &Fb->w2, w->y);
        residual(w->r, w->y, Fb->gamma, d);
        if ((st = sub_output(m, w->r, &Fb->ln, w->tmp))) return st;
    }
    const float *o = w->r;
    if (c->pre_ln) {
        if ((st = layer_norm(w->r, d, &m->dec_final, w->tmp))) return st;
        o = w->tmp;
    }
    float io = 1.0f / m->s_dout;
    for (int i = 0; i < d; i++) w->a[i] = q8(o[i], io);
    if (dec_q) memcpy(dec_q, w->a, (size_t)d);
    linear_row(w->a, m->s_dout, &m->out, logits);
    return OR_OK;
}

/* ------------------------------------------------------------------------ */
/* search                                                                    */
/* ------------------------------------------------------------------------ */

/* Normaliser of the beam search's log-softmax over one logit row (App. D
 * decodes with log-probabilities; their arithmetic is unstated): m = max_n l[n]
 * (order-free), fixed-point weights E_n = rne(exp(fl(l[n] - m)) 2^24) summed
 * exactly as Z = sum E_n, and lambda = fl32(ln Z - 24 ln 2), i.e. the natural
 * log of the sum of exp(l[n] - m) on the 2^-24 grid.  Returns Z. */
static int64_t log_softmax_norm(const float *l, int V, float *m_out, float *lam_out) {
    float mx = l[0];
    for (int n = 1; n < V; n++) if (l[n] > mx) mx = l[n];
    int64_t Z = 0;
    for (int n = 0; n < V; n++) Z += (int64_t)rintf(exp_own(l[n] - mx) * 16777216.0f);
    *m_out = mx;
    *lam_out = (float)(log_own((double)Z) - 0x1.0a2b23f3bab73p+4); /* 24 ln 2 */
    return Z;
}

/* greedy: argmax, ties to the lowest id */
static int argmax_f(const float *l, int V) {
    int best = 0;
    for (int n = 1; n < V; n++)
        if (l[n] > l[best]) best = n;
    return best;
}

static int oenc_alloc(oenc *e, const ocfg *c, int S, int len) {
    e->S = S; e->len = len;
    e->enc_q = malloc((size_t)S * c->d);
    e->ck = malloc((size_t)c->n_dec * S * c->d);
    e->cv = malloc((size_t)c->n_dec * S * c->d);
    return (e->enc_q && e->ck && e->cv) ? OR_OK : OR_ENOMEM;
}

static void oenc_free(oenc *e) { free(e->enc_q); free(e->ck); free(e->cv); }

static int cache_alloc(ocache *k, const ocfg *c, int T) {
    k->T = T;
    k->k = calloc((size_t)c->n_dec * T * c->d, 1);
    k->v = calloc((size_t)c->n_dec * T * c->d, 1);
    return (k->k && k->v) ? OR_OK : OR_ENOMEM;
}

static void cache_free(ocache *k) { free(k->k); free(k->v); }

static int greedy_one(const omodel *m, const oenc *enc, int max_len, int32_t *out_ids,
                      int32_t *out_len) {
    const ocfg *c = &m->c;
    ocache cache = {0, NULL, NULL};
    oscratch w;
    memset(&w, 0, sizeof(w));
    float *logits = malloc(sizeof(float) * c->V);
    int st = cache_alloc(&cache, c, max_len);
    if (!st) st = scratch_init(&w, c, max_len > enc->S ? max_len : enc->S);
    if (!logits) st = OR_ENOMEM;
    int tok = c->bos, n_out = 0;
    for (int t = 0; t < max_len; t++) out_ids[t] = c->pad;
    for (int t = 0; !st && t < max_len; t++) {
        st = decode_step(m, enc, &cache, tok, t, &w, logits, NULL);
        if (st) break;
        int y = argmax_f(logits, c->V);
        out_ids[t] = y;
        n_out = t + 1;
        if (y == c->eos) break;
        tok = y;
    }
    *out_len = n_out;
    scratch_free(&w);
    cache_free(&cache);
    free(logits);
    return st;
}

typedef struct { float score; int64_t idx; } ocand;

/* candidate a ranks before b: higher score first, then lower flat index */
static int cand_before(const ocand *a, const ocand *b) {
    if (a->score > b->score) return 1;
    if (a->score < b->score) return 0;
    return a->idx < b->idx;
}

/* keep the k best candidates seen so far, sorted best first */
static void push_cand(ocand *top, int *nt, int k, ocand cd) {
    if (*nt == k && !cand_before(&cd, &top[k - 1])) return;
    int pos = *nt < k ? *nt : k - 1; /* when full, the last one is dropped */
    while (pos > 0 && cand_before(&cd, &top[pos - 1])) { top[pos] = top[pos - 1]; pos--; }
    top[pos] = cd;
    if (*nt < k) (*nt)++;
}

/* Beam search over k hypotheses (reading of the paper's unstated beam: no
 * length penalty, finished hypotheses carry their score forward as a single
 * PAD candidate, ranking by (score desc, flat index asc), output beam 0).
 * Each hypothesis owns a full copy of its self-attention cache. */
static int beam_one(const omodel *m, const oenc *enc, int k, int max_len, int32_t *out_ids,
                    int32_t *out_len, float *out_score) {
    const ocfg *c = &m->c;
    int V = c->V, st = OR_OK;
    size_t cache_bytes = (size_t)c->n_dec * max_len * c->d;
    ocache *cache = calloc(k, sizeof(ocache)), *next = calloc(k, sizeof(ocache));
    int *tok = calloc(k, sizeof(int)), *fin = calloc(k, sizeof(int)), *nfin = calloc(k, sizeof(int));
    int *ntok = calloc(k, sizeof(int));
    float *cum = calloc(k, sizeof(float)), *ncum = calloc(k, sizeof(float));
    int32_t *hist = calloc((size_t)k * max_len, sizeof(int32_t));
    int32_t *nhist = calloc((size_t)k * max_len, sizeof(int32_t));
    float *logits = malloc(sizeof(float) * V);
    ocand *top = malloc(sizeof(ocand) * k);
    oscratch w;
    memset(&w, 0, sizeof(w));
    if (!cache || !next || !tok || !fin || !nfin || !ntok || !cum || !ncum || !hist || !nhist ||
        !logits || !top) {
        st = OR_ENOMEM;
        goto done;
    }
    if ((st = scratch_init(&w, c, max_len > enc->S ? max_len : enc->S))) goto done;
    for (int i = 0; i < k && !st; i++) {
        st = cache_alloc(&cache[i], c, max_len);
        if (!st) st = cache_alloc(&next[i], c, max_len);
    }
    if (st) goto done_w;
    for (int i = 0; i < k; i++) {
        tok[i] = c->bos;
        cum[i] = i == 0 ? 0.0f : -INFINITY; /* only beam 0 is live at the start */
        fin[i] = 0;
    }
    for (int i = 0; i < k * max_len; i++) hist[i] = c->pad;
    int steps = 0;
    for (int t = 0; t < max_len; t++) {
        int nt = 0; /* number of candidates kept in top[] */
        for (int i = 0; i < k; i++) {
            if (fin[i]) { /* a finished hypothesis offers itself once, unchanged */
                ocand cd = {cum[i], (int64_t)i * V + c->pad};
                push_cand(top, &nt, k, cd);
                continue;
            }
            if ((st = decode_step(m, enc, &cache[i], tok[i], t, &w, logits, NULL))) goto done_w;
            float mx, lam;
            log_softmax_norm(logits, V, &mx, &lam);
            for (int n = 0; n < V; n++) {
                float lp = (logits[n] - mx) - lam;
                ocand cd = {cum[i] + lp, (int64_t)i * V + n};
                push_cand(top, &nt, k, cd);
            }
        }
        /* new hypotheses: parent p, token n; copy the parent's cache and history */
        for (int i = 0; i < k; i++) {
            int p = (int)(top[i].idx / V), n = (int)(top[i].idx % V);
            memcpy(next[i].k, cache[p].k, cache_bytes);
            memcpy(next[i].v, cache[p].v, cache_bytes);
            memcpy(nhist + (size_t)i * max_len, hist + (size_t)p * max_len, sizeof(int32_t) * max_len);
            nhist[(size_t)i * max_len + t] = n;
            ncum[i] = top[i].score;
            nfin[i] = fin[p] || n == c->eos;
            ntok[i] = n;
        }
        for (int i = 0; i < k; i++) {
            ocache tmpc = cache[i]; cache[i] = next[i]; next[i] = tmpc;
            cum[i] = ncum[i]; fin[i] = nfin[i]; tok[i] = ntok[i];
        }
        int32_t *th = hist; hist = nhist; nhist = th;
        steps = t + 1;
        int all = 1;
        for (int i = 0; i < k; i++) all &= fin[i];
        if (all) break;
    }
    {
        int n_out = steps;
        for (int t = 0; t < max_len; t++) out_ids[t] = t < steps ? hist[t] : c->pad;
        for (int t = 0; t < steps; t++)
            if (hist[t] == c->eos) { n_out = t + 1; break; }
        for (int t = n_out; t < max_len; t++) out_ids[t] = c->pad;
        *out_len = n_out;
        *out_score = cum[0];
    }
done_w:
    for (int i = 0; i < k; i++) {
        if (cache) cache_free(&cache[i]);
        if (next) cache_free(&next[i]);
    }
    scratch_free(&w);
done:
    free(cache); free(next); free(tok); free(fin); free(nfin); free(ntok); free(cum); free(ncum);
    free(hist); free(nhist); free(logits); free(top);
    return st;
}

/* ------------------------------------------------------------------------ */
/* exported entry points (ctypes)                                            */
/* ------------------------------------------------------------------------ */

int oracle_check_blob(const void *blob, size_t bytes, int32_t *cfg_out) {
    omodel *mm = malloc(sizeof(omodel));
    if (!mm) return OR_ENOMEM;
    int st = parse(blob, bytes, mm);
    if (!st && cfg_out) {
        const ocfg *c = &mm->c;
        int32_t v[13] = {c->n_enc, c->n_dec, c->d, c->H, c->F, c->V, c->E, c->pre_ln, c->tied,
                         c->max_pos, c->pad, c->bos, c->eos};
        memcpy(cfg_out, v, sizeof(v));
    }
    free(mm);
    return st;
}

float oracle_q8(float x, float inv) { return (float)q8(x, inv); }

/* Row-wise quantisation of a float64 matrix W [N][K] to `bits` bits (App. B
 * Eq. scale / Eq. quant; Sec. 3.3 per-row "row-wise" scales for low bits).
 *   symmetric (asym = 0): s_n = fl32(max_k |W_nk| / (2^(bits-1) - 1)), code
 *     v = clamp(rne(W_nk / s_n), -(2^(bits-1) - 1), 2^(bits-1) - 1): Eq. quant
 *     with the range [-max|W_n|, max|W_n|] and zero offset.
 *   min-max (asym = 1): r_n = fl32(min_k W_nk), s_n = fl32((max_k W_nk - r_n) /
 *     (2^bits - 1)), code u = clamp(rne((W_nk - r_n) / s_n), 0, 2^bits - 1);
 *     the dequantised weight is s_n u + r_n.
 * codes [N][K] receive v or u; s [N], m [N] (r_n; 0 when symmetric).  A row
 * of zeros (or a constant row, min-max) gets scale 1. */
int oracle_quantise_rows(const double *W, int N, int K, int bits, int asym, int32_t *codes, float *s,
                         float *m) {
    if (bits < 2 || bits > 8 || N < 1 || K < 1) return OR_EINVAL;
    for (int n = 0; n < N; n++) {
        const double *w = W + (size_t)n * K;
        double lo = w[0], hi = w[0], amax = 0.0;
        for (int k = 0; k < K; k++) {
            if (w[k] < lo) lo = w[k];
            if (w[k] > hi) hi = w[k];
            if (fabs(w[k]) > amax) amax = fabs(w[k]);
        }
        if (!asym) {
            int qmax = (1 << (bits - 1)) - 1;
            float sn = amax > 0.0 ? (float)(amax / qmax) : 1.0f;
            s[n] = sn;
            m[n] = 0.0f;
            for (int k = 0; k < K; k++) {
                double t = rint(w[k] / (double)sn);
                if (t > qmax) t = qmax;
                if (t < -qmax) t = -qmax;
                codes[(size_t)n * K + k] = (int32_t)t;
            }
        } else {
            int qmax = (1 << bits) - 1;
            float rn = (float)lo;
            float sn = hi > (double)rn ? (float)((hi - (double)rn) / qmax) : 1.0f;
            if (sn == 0.0f) sn = 1.0f;
            s[n] = sn;
            m[n] = rn;
            for (int k = 0; k < K; k++) {
                double t = rint((w[k] - (double)rn) / (double)sn);
                if (t > qmax) t = qmax;
                if (t < 0) t = 0;
                codes[(size_t)n * K + k] = (int32_t)t;
            }
        }
    }
    return OR_OK;
}

/* A 4-bit quantised linear on M int8 rows (kernel-level parity): Wp [N][K/2]
 * packed as in the blob (lin_code), s / m / b [N] (m only if asym); mode as
 * oracle_linear. */
int oracle_linear_w4(const int8_t *A, const uint8_t *Wp, const float *s_w, const float *m_w, const float *b,
                     float s_x, const float *inv_out, float gamma, int M, int N, int K, int asym, int mode,
                     int8_t *out_q, float *out_f) {
    if (K % 32) return OR_EINVAL;
    olin L;
    memset(&L, 0, sizeof(L));
    L.wp = Wp; L.s = s_w; L.m = m_w; L.b = b; L.n = N; L.k = K; L.bits = 4; L.asym = asym;
    for (int mm = 0; mm < M; mm++) {
        for (int n = 0; n < N; n++) {
            float y = lin_out(&L, n, A + (size_t)mm * K, s_x);
            size_t o = (size_t)mm * N + n;
            if (mode == 0) out_q[o] = q8(y, inv_out[n]);
            else if (mode == 1) out_q[o] = q8(y > 0.0f ? y : 0.0f, inv_out[n]);
            else if (mode == 2) { float t = gamma * out_f[o]; out_f[o] = t + y; }
            else out_f[o] = y;
        }
    }
    return OR_OK;
}

/* ---- fake quantisation (QAT forward / backward; App. B "PTQ and QAT") ----
 * The quantiser of Eq. quant inserted into a float model, with a learnable
 * scale s (and, min-max form, offset r_m):
 *   symmetric, n bits: q = clamp(rne(fl(x fl(1/s))), -(2^(n-1)-1), 2^(n-1)-1),
 *                      y = fl(q s)
 *   min-max,   n bits: q = clamp(rne(fl(fl(x - r_m) fl(1/s))), 0, 2^n - 1),
 *                      y = fl(fl(q s) + r_m)
 * Backward (straight-through estimator for x; the scale and offset gradients
 * of the same expression, rounding held fixed): with t = the unrounded code
 * above and `in` = qmin <= t <= qmax,
 *   dy/dx = in,  dy/ds = in ? q - t : q,  dy/dr_m = in ? 0 : 1. */
static void fq_range(int bits, int minmax, int *qmin, int *qmax) {
    if (minmax) { *qmin = 0; *qmax = (1 << bits) - 1; }
    else { *qmax = (1 << (bits - 1)) - 1; *qmin = -*qmax; }
}

int oracle_fake_quant(const float *x, int n, float s, float r_m, int bits, int minmax, float *y, int32_t *codes) {
    if (bits < 2 || bits > 8 || !(s > 0.0f)) return OR_EINVAL;
    int qmin, qmax;
    fq_range(bits, minmax, &qmin, &qmax);
    float inv = 1.0f / s;
    for (int i = 0; i < n; i++) {
        float t = minmax ? (x[i] - r_m) * inv : x[i] * inv;
        float q = rintf(t);
        if (q < qmin) q = (float)qmin;
        if (q > qmax) q = (float)qmax;
        if (codes) codes[i] = (int32_t)q;
        if (y) {
            float v = q * s;
            y[i] = minmax ? v + r_m : v;
        }
    }
    return OR_OK;
}

int oracle_fake_quant_backward(const float *x, const float *g, int n, float s, float r_m, int bits, int minmax,
                               float *gx, double *gs, double *gr) {
    if (bits < 2 || bits > 8 || !(s > 0.0f)) return OR_EINVAL;
    int qmin, qmax;
    fq_range(bits, minmax, &qmin, &qmax);
    float inv = 1.0f / s;
    double as = 0.0, ar = 0.0;
    for (int i = 0; i < n; i++) {
        float t = minmax ? (x[i] - r_m) * inv : x[i] * inv;
        int in = t >= (float)qmin && t <= (float)qmax;
        float q = rintf(t);
        if (q < qmin) q = (float)qmin;
        if (q > qmax) q = (float)qmax;
        gx[i] = in ? g[i] : 0.0f;
        as += (double)g[i] * (in ? (double)q - (double)t : (double)q);
        if (!in) ar += (double)g[i];
    }
    *gs = as;
    if (gr) *gr = minmax ? ar : 0.0;
    return OR_OK;
}

/* QAT forward of one linear: X [M][K] float fake-quantised per tensor to
 * 8-bit codes at scale s_x, W [N][K] float fake-quantised per row to `wbits`
 * symmetric codes at scales s_w[n]; y = the quantised linear of the codes
 * (dequantise with fl(s_x s_w[n]), add the bias), i.e. X_q W_q^T + b with the
 * products exact. */
int oracle_fake_quant_linear(const float *X, const float *W, float s_x, const float *s_w, const float *b, int M,
                             int N, int K, int wbits, float *y) {
    if (wbits < 2 || wbits > 8 || !(s_x > 0.0f)) return OR_EINVAL;
    int32_t *qx = malloc(sizeof(int32_t) * (size_t)M * K), *qw = malloc(sizeof(int32_t) * (size_t)N * K);
    if (!qx || !qw) { free(qx); free(qw); return OR_ENOMEM; }
    int st = oracle_fake_quant(X, M * K, s_x, 0.0f, 8, 0, NULL, qx);
    for (int n = 0; !st && n < N; n++) st = oracle_fake_quant(W + (size_t)n * K, K, s_w[n], 0.0f, wbits, 0, NULL, qw + (size_t)n * K);
    for (int m = 0; !st && m < M; m++)
        for (int n = 0; n < N; n++) {
            int32_t acc = 0;
            for (int k = 0; k < K; k++) acc += qx[(size_t)m * K + k] * qw[(size_t)n * K + k];
            y[(size_t)m * N + n] = dequant_bias(acc, s_x, s_w[n], b[n]);
        }
    free(qx); free(qw);
    return st;
}

/* The LayerNorm's mean and biased variance of M rows of length d. */
int oracle_ln_stats(const float *r, int M, int d, float *mu, float *var) {
    for (int m = 0; m < M; m++) {
        int st = ln_stats(r + (size_t)m * d, d, mu + m, var + m);
        if (st) return st;
    }
    return OR_OK;
}
float oracle_exp(float x) { return exp_own(x); }
double oracle_log(double z) { return log_own(z); }

/* C[m][n] = sum_k A[m][k] W[n][k] (int32) */
void oracle_gemm_i32(const int8_t *A, const int8_t *W, int M, int N, int K, int32_t *C) {
    for (int m = 0; m < M; m++)
        for (int n = 0; n < N; n++) C[(size_t)m * N + n] = dot_i8(A + (size_t)m * K, W + (size_t)n * K, K);
}

/* Quantised linear with one of the fused epilogues:
 *   mode 0: int8 out = q8(y, inv_out[n])          (E1)
 *   mode 1: int8 out = q8(max(y, 0), inv_out[n])  (E2, ReLU)
 *   mode 2: fp32 resid[m][n] = fl(fl(gamma * resid) + y)   (E3, residual)
 *   mode 3: fp32 out = y                          (logits)
 * with y = fl(fl(acc * fl(s_x * s_w[n])) + b[n]). */
int oracle_linear(const int8_t *A, const int8_t *W, const float *s_w, const float *b, float s_x,
                  const float *inv_out, float gamma, int M, int N, int K, int mode, int8_t *out_q,
                  float *out_f) {
    for (int m = 0; m < M; m++)
        for (int n = 0; n < N; n++) {
            float y = dequant_bias(dot_i8(A + (size_t)m * K, W + (size_t)n * K, K), s_x, s_w[n], b[n]);
            size_t o = (size_t)m * N + n;
            if (mode == 0) out_q[o] = q8(y, inv_out[n]);
            else if (mode == 1) out_q[o] = q8(y > 0.0f ? y : 0.0f, inv_out[n]);
            else if (mode == 2) { float t = gamma * out_f[o]; out_f[o] = t + y; }
            else if (mode == 3) out_f[o] = y;
            else return OR_EINVAL;
        }
    return OR_OK;
}

/* LayerNorm of M rows, optional fp32 output and int8 output q8(LN(r), inv). */
int oracle_layernorm(const float *r, const float *g, const float *b, int M, int d, float inv,
                     float *out_f, int8_t *out_q) {
    oln ln = {g, b};
    float *tmp = malloc(sizeof(float) * d);
    if (!tmp) return OR_ENOMEM;
    for (int m = 0; m < M; m++) {
        int st = layer_norm(r + (size_t)m * d, d, &ln, tmp);
        if (st) { free(tmp); return st; }
        for (int i = 0; i < d; i++) {
            if (out_f) out_f[(size_t)m * d + i] = tmp[i];
            if (out_q) out_q[(size_t)m * d + i] = q8(tmp[i], inv);
        }
    }
    free(tmp);
    return OR_OK;
}

/* Incremental (decode) attention of R query rows over per-row caches:
 * q [R][H][dh], cache K/V [R][H][T][dh], row r attends keys 0..n_keys[r]-1. */
int oracle_attention_decode(const int8_t *q, const int8_t *Kc, const int8_t *Vc, const int32_t *n_keys,
                            int R, int H, int dh, int T, float sigma, float rho, int8_t *ctx) {
    float *sbuf = malloc(sizeof(float) * T);
    int64_t *nbuf = malloc(sizeof(int64_t) * dh);
    const int8_t **kp = malloc(sizeof(void *) * T), **vp = malloc(sizeof(void *) * T);
    if (!sbuf || !nbuf || !kp || !vp) return OR_ENOMEM;
    for (int r = 0; r < R; r++)
        for (int h = 0; h < H; h++) {
            int n = n_keys[r];
            if (n < 1 || n > T) { free(sbuf); free(nbuf); free((void *)kp); free((void *)vp); return OR_EINVAL; }
            for (int j = 0; j < n; j++) {
                kp[j] = Kc + (((size_t)r * H + h) * T + j) * dh;
                vp[j] = Vc + (((size_t)r * H + h) * T + j) * dh;
            }
            attend(q + ((size_t)r * H + h) * dh, kp, vp, n, dh, sigma, rho, ctx + ((size_t)r * H + h) * dh,
                   sbuf, nbuf);
        }
    free(sbuf); free(nbuf); free((void *)kp); free((void *)vp);
    return OR_OK;
}

/* Attention diagnostics of one head: fp32 softmax weights P_j = E_j / Z. */
int oracle_attention_probs(const int8_t *q, const int8_t *K, int n, int dh, float sigma, float *P) {
    float *s = malloc(sizeof(float) * n);
    if (!s) return OR_ENOMEM;
    float m = -INFINITY;
    for (int j = 0; j < n; j++) {
        s[j] = (float)dot_i8(q, K + (size_t)j * dh, dh) * sigma;
        if (s[j] > m) m = s[j];
    }
    int64_t Z = 0;
    for (int j = 0; j < n; j++) Z += (int64_t)rintf(exp_own(s[j] - m) * 16777216.0f);
    for (int j = 0; j < n; j++)
        P[j] = rn32_quotient((int64_t)rintf(exp_own(s[j] - m) * 16777216.0f), Z);
    free(s);
    return OR_OK;
}

float oracle_sigma(float s_q, float s_k, int dh) { return sigma_of(s_q, s_k, dh); }

/* Encoder of one sentence: quantised output [S][d] and cross K/V [n_dec][S][d]. */
int oracle_encode(const void *blob, size_t bytes, const int32_t *src, int len, int S, int8_t *enc_q,
                  int8_t *ck, int8_t *cv) {
    omodel *m = malloc(sizeof(omodel));
    if (!m) return OR_ENOMEM;
    int st = parse(blob, bytes, m);
    if (!st) {
        oenc e = {S, len, enc_q, ck, cv};
        st = encode_one(m, src, len, S, &e);
    }
    free(m);
    return st;
}

/* Teacher-forced greedy trace of one sentence: for t in [0, T) feeds tgt[t]
 * (tgt[0] is normally BOS) and writes the step's logits [T][V] and the
 * quantised decoder output [T][d]; if self_k/self_v are given they receive
 * the final self-attention cache [n_dec][T][d]. */
int oracle_decode_trace(const void *blob, size_t bytes, const int32_t *src, int len, int S,
                        const int32_t *tgt, int T, float *logits, int8_t *dec_q, int8_t *self_k,
                        int8_t *self_v) {
    omodel *m = malloc(sizeof(omodel));
    if (!m) return OR_ENOMEM;
    int st = parse(blob, bytes, m);
    if (st) { free(m); return st; }
    const ocfg *c = &m->c;
    oenc e;
    ocache cache = {0, NULL, NULL};
    oscratch w;
    memset(&w, 0, sizeof(w));
    st = oenc_alloc(&e, c, S, len);
    if (!st) st = encode_one(m, src, len, S, &e);
    if (!st) st = cache_alloc(&cache, c, T);
    if (!st) st = scratch_init(&w, c, T > S ? T : S);
    for (int t = 0; !st && t < T; t++)
        st = decode_step(m, &e, &cache, tgt[t], t, &w, logits + (size_t)t * c->V,
                         dec_q ? dec_q + (size_t)t * c->d : NULL);
    if (!st && self_k) memcpy(self_k, cache.k, (size_t)c->n_dec * T * c->d);
    if (!st && self_v) memcpy(self_v, cache.v, (size_t)c->n_dec * T * c->d);
    scratch_free(&w);
    cache_free(&cache);
    oenc_free(&e);
    free(m);
    return st;
}

/* Teacher-forced decoder computed layer by layer over the whole target
 * prefix at once, with an explicit causal mask (keys j <= i for query i).
 * A second, independently structured path: it must give the same logits as
 * the incremental decode_step. */
int oracle_decode_forced(const void *blob, size_t bytes, const int32_t *src, int len, int S,
                         const int32_t *tgt, int T, float *logits) {
    omodel *m = malloc(sizeof(omodel));
    if (!m) return OR_ENOMEM;
    int st = parse(blob, bytes, m);
    if (st) { free(m); return st; }
    const ocfg *c = &m->c;
    int d = c->d, dh = d / c->H, F = c->F, big = 3 * d > F ? 3 * d : F;
    oenc e;
    st = oenc_alloc(&e, c, S, len);
    if (!st) st = encode_one(m, src, len, S, &e);
    float *r = malloc(sizeof(float) * T * d), *y = malloc(sizeof(float) * big);
    float *tmp = malloc(sizeof(float) * d), *sbuf = malloc(sizeof(float) * (T > S ? T : S));
    int8_t *a = malloc((size_t)big), *Q = malloc((size_t)T * d), *K = malloc((size_t)T * d);
    int8_t *Vv = malloc((size_t)T * d), *C = malloc((size_t)T * d);
    int64_t *nbuf = malloc(sizeof(int64_t) * dh);
    int nk = T > S ? T : S;
    const int8_t **kp = malloc(sizeof(void *) * nk), **vp = malloc(sizeof(void *) * nk);
    if (!r || !y || !tmp || !sbuf || !a || !Q || !K || !Vv || !C || !nbuf || !kp || !vp) st = OR_ENOMEM;
    for (int i = 0; !st && i < T; i++) embed(m, tgt[i], i, r + (size_t)i * d);
    for (int l = 0; !st && l < c->n_dec; l++) {
        const oself *A = &m->dec_self[l];
        float iq = 1.0f / A->s_q, ik = 1.0f / A->s_k, iv = 1.0f / A->s_v;
        for (int i = 0; !st && i < T; i++) {
            st = sub_input(m, r + (size_t)i * d, &A->ln, A->s_in, a, tmp);
            linear_row(a, A->s_in, &A->qkv, y);
            for (int n = 0; n < d; n++) {
                Q[(size_t)i * d + n] = q8(y[n], iq);
                K[(size_t)i * d + n] = q8(y[d + n], ik);
                Vv[(size_t)i * d + n] = q8(y[2 * d + n], iv);
            }
        }
        float sigma = sigma_of(A->s_q, A->s_k, dh), rho = A->s_v / A->s_ctx;
        for (int i = 0; i < T; i++)
            for (int h = 0; h < c->H; h++) {
                int n = 0;
                for (int j = 0; j < T; j++) {
                    if (j > i) continue; /* causal mask */
                    kp[n] = K + (size_t)j * d + h * dh;
                    vp[n] = Vv + (size_t)j * d + h * dh;
                    n++;
                }
                attend(Q + (size_t)i * d + h * dh, kp, vp, n, dh, sigma, rho, C + (size_t)i * d + h * dh,
                       sbuf, nbuf);
            }
        for (int i = 0; !st && i < T; i++) {
            linear_row(C + (size_t)i * d, A->s_ctx, &A->o, y);
            residual(r + (size_t)i * d, y, A->gamma, d);
            st = sub_output(m, r + (size_t)i * d, &A->ln, tmp);
        }
        const ocross *X = &m->dec_cross[l];
        float iqx = 1.0f / X->s_q;
        float sx = sigma_of(X->s_q, X->s_k, dh), rx = X->s_v / X->s_ctx;
        for (int i = 0; !st && i < T; i++) {
            st = sub_input(m, r + (size_t)i * d, &X->ln, X->s_in, a, tmp);
            linear_row(a, X->s_in, &X->q, y);
            for (int n = 0; n < d; n++) Q[(size_t)i * d + n] = q8(y[n], iqx);
            for (int h = 0; h < c->H; h++) {
                for (int j = 0; j < len; j++) {
                    kp[j] = e.ck + ((size_t)l * S + j) * d + h * dh;
                    vp[j] = e.cv + ((size_t)l * S + j) * d + h * dh;
                }
                attend(Q + (size_t)i * d + h * dh, kp, vp, len, dh, sx, rx, C + (size_t)i * d + h * dh,
                       sbuf, nbuf);
            }
            linear_row(C + (size_t)i * d, X->s_ctx, &X->o, y);
            residual(r + (size_t)i * d, y, X->gamma, d);
            if (!st) st = sub_output(m, r + (size_t)i * d, &X->ln, tmp);
        }
        const offn *Fb = &m->dec_ffn[l];
        float ih = 1.0f / Fb->s_h;
        for (int i = 0; !st && i < T; i++) {
            st = sub_input(m, r + (size_t)i * d, &Fb->ln, Fb->s_in, a, tmp);
            linear_row(a, Fb->s_in, &Fb->w1, y);
            for (int n = 0; n < F; n++) a[n] = q8(y[n] > 0.0f ? y[n] : 0.0f, ih);
            linear_row(a, Fb->s_h, &Fb->w2, y);
            residual(r + (size_t)i * d, y, Fb->gamma, d);
            if (!st) st = sub_output(m, r + (size_t)i * d, &Fb->ln, tmp);
        }
    }
    float io = 1.0f / m->s_dout;
    for (int i = 0; !st && i < T; i++) {
        const float *o = r + (size_t)i * d;
        if (c->pre_ln) {
            st = layer_norm(o, d, &m->dec_final, tmp);
            o = tmp;
        }
        for (int n = 0; n < d; n++) a[n] = q8(o[n], io);
        linear_row(a, m->s_dout, &m->out, logits + (size_t)i * c->V);
    }
    free(r); free(y); free(tmp); free(sbuf); free(a); free(Q); free(K); free(Vv); free(C); free(nbuf);
    free((void *)kp); free((void *)vp);
    oenc_free(&e);
    free(m);
    return st;
}

/* Embedding rows (fp32 [n][d]) for ids at positions pos. */
int oracle_embed(const void *blob, size_t bytes, const int32_t *ids, const int32_t *pos, int n,
                 float *x) {
    omodel *m = malloc(sizeof(omodel));
    if (!m) return OR_ENOMEM;
    int st = parse(blob, bytes, m);
    for (int i = 0; !st && i < n; i++) {
        if (ids[i] < 0 || ids[i] >= m->c.V || pos[i] < 0 || pos[i] >= m->c.max_pos) { st = OR_EINVAL; break; }
        embed(m, ids[i], pos[i], x + (size_t)i * m->c.d);
    }
    free(m);
    return st;
}

/* Beam-search log-probabilities of one logit row: lp[n] = fl(fl(l - m) - lambda),
 * with m and lambda from log_softmax_norm (the function beam_one uses). */
int oracle_log_softmax(const float *l, int V, float *lp) {
    float mx, lam;
    log_softmax_norm(l, V, &mx, &lam);
    for (int n = 0; n < V; n++) lp[n] = (l[n] - mx) - lam;
    return OR_OK;
}

/* The normaliser alone: *m = max_n l[n], *lam = lambda, *Z = the fixed-point sum. */
int oracle_log_softmax_norm(const float *l, int V, float *m, float *lam, int64_t *Z) {
    int64_t z = log_softmax_norm(l, V, m, lam);
    if (Z) *Z = z;
    return OR_OK;
}

/* ---------------------------- translation ------------------------------- */
typedef struct {
    const omodel *m;
    const int32_t *src, *lens;
    int B, S, beam, max_len;
    int32_t *out_ids, *out_lens;
    float *out_scores;
    int next;              /* next sentence to take */
    int status;
    pthread_mutex_t mu;
} ojob;

static int translate_sentence(const omodel *m, const int32_t *src, int len, int S, int beam,
                              int max_len, int32_t *ids, int32_t *olen, float *score) {
    oenc e;
    int st = oenc_alloc(&e, &m->c, S, len);
    if (!st) st = encode_one(m, src, len, S, &e);
    if (!st) {
        if (beam == 1) { /* beam < 0 requests the beam search with width -beam */
            st = greedy_one(m, &e, max_len, ids, olen);
            *score = 0.0f;
        } else {
            st = beam_one(m, &e, beam < 0 ? -beam : beam, max_len, ids, olen, score);
        }
    }
    oenc_free(&e);
    return st;
}

static void *worker(void *arg) {
    ojob *j = (ojob *)arg;
    for (;;) {
        pthread_mutex_lock(&j->mu);
        int b = j->next++;
        pthread_mutex_unlock(&j->mu);
        if (b >= j->B) break;
        int st = translate_sentence(j->m, j->src + (size_t)b * j->S, j->lens[b], j->S, j->beam,
                                    j->max_len, j->out_ids + (size_t)b * j->max_len, j->out_lens + b,
                                    j->out_scores + b);
        if (st) {
            pthread_mutex_lock(&j->mu);
            if (!j->status) j->status = st;
            pthread_mutex_unlock(&j->mu);
        }
    }
    return NULL;
}

/* Translate B sentences (src [B][S] right-padded, lens [B]); out_ids
 * [B][max_len] PAD-filled, out_lens [B] (tokens up to and including EOS),
 * out_scores [B] (beam: final cumulative log-probability of the best
 * hypothesis; greedy: 0).  beam = 1 is greedy search; beam = -k runs the
 * beam search with width k even for k = 1.  Sentences run in parallel on n_threads threads,
 * each sentence single-threaded. */
int oracle_translate(const void *blob, size_t bytes, const int32_t *src, const int32_t *lens, int B,
                     int S, int beam, int max_len, int n_threads, int32_t *out_ids, int32_t *out_lens,
                     float *out_scores) {
    omodel *m = malloc(sizeof(omodel));
    if (!m) return OR_ENOMEM;
    int st = parse(blob, bytes, m);
    if (st) { free(m); return st; }
    if (B < 1 || S < 1 || beam == 0 || beam > 4096 || beam < -4096 || max_len < 1 ||
        max_len > m->c.max_pos || S > m->c.max_pos) {
        free(m);
        return OR_EINVAL;
    }
    ojob j;
    j.m = m; j.src = src; j.lens = lens; j.B = B; j.S = S; j.beam = beam; j.max_len = max_len;
    j.out_ids = out_ids; j.out_lens = out_lens; j.out_scores = out_scores; j.next = 0; j.status = 0;
    pthread_mutex_init(&j.mu, NULL);
    if (n_threads < 1) n_threads = 1;
    if (n_threads > B) n_threads = B;
    pthread_t *th = malloc(sizeof(pthread_t) * n_threads);
    int started = 0;
    for (int i = 1; th && i < n_threads; i++)
        if (pthread_create(&th[started], NULL, worker, &j) == 0) started++;
    /* the calling thread works too */
    worker(&j);
    for (int i = 0; i < started; i++) pthread_join(th[i], NULL);
    free(th);
    pthread_mutex_destroy(&j.mu);
    free(m);
    return j.status;
}
