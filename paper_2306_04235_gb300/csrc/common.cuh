// common.cuh -- device arithmetic shared by the sm_103a kernels of libmnmt.
//
// Every float operation here is written with explicit round-to-nearest
// intrinsics and the library is compiled with --fmad=false, so each a*b+c is
// two IEEE roundings exactly as the method's arithmetic is defined (the int8
// quantiser of App. B with zero point 0, the full-precision epilogues of Fig. 5,
// the fixed-point LayerNorm and softmax sums).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/mnmt.h"

#define MNMT_DEV __device__ __forceinline__

// ---------------------------------------------------------------------------
// programmatic dependent launch: every kernel of the library is launched
// allowed to start before its predecessor in the stream has finished; it lets
// its own successor launch at once, then waits for the predecessor (and the
// memory it wrote) before it reads anything.  Every kernel waits, so waiting
// for the predecessor also covers everything before it.
// ---------------------------------------------------------------------------
MNMT_DEV void pdl_allow_next() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }
MNMT_DEV void pdl_grid_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }

// ---------------------------------------------------------------------------
// quantiser: q8(x, inv) = clamp(round_half_even(fl(x * inv)), -127, 127)
// ---------------------------------------------------------------------------
MNMT_DEV int8_t q8(float x, float inv) {
    float t = rintf(__fmul_rn(x, inv));
    t = fminf(fmaxf(t, -127.0f), 127.0f);
    return (int8_t)__float2int_rz(t);
}

// dequantise + bias: y = fl(fl(acc * fl(s_x * s_w)) + b)
MNMT_DEV float dequant_bias(int32_t acc, float s_x, float s_w, float b) {
    float sc = __fmul_rn(s_x, s_w);
    return __fadd_rn(__fmul_rn(__int2float_rn(acc), sc), b);
}

// ---------------------------------------------------------------------------
// round_half_even(v * 2^shift) as int64, with integer operations only.  Equal
// to llrint(ldexp((double)v, shift)) whenever |v| 2^shift < 2^62.
// ---------------------------------------------------------------------------
MNMT_DEV long long fx_scale(float v, int shift) {
    uint32_t bits = __float_as_uint(v);
    uint32_t ex = (bits >> 23) & 0xFFu;
    // fast path: v normal and y = v 2^shift a normal float below 2^62 -- the
    // scaling is then exact.  |y| >= 2^23 is an integer, its significand
    // shifted left; |y| < 2^23 rounds half to even into 32 bits (the 64-bit
    // float-to-integer conversion runs at a small fraction of this rate)
    if (ex != 0 && (int)ex + shift >= 1 && (int)ex + shift <= 127 + 61) {
        const int ey = (int)ex + shift;  // biased exponent of y
        if (ey >= 127 + 23) {
            const long long q = (long long)((bits & 0x7FFFFFu) | 0x800000u) << (ey - 150);
            return (bits >> 31) ? -q : q;
        }
        return (long long)__float2int_rn(__uint_as_float(bits + ((uint32_t)shift << 23)));
    }
    uint32_t man = bits & 0x7FFFFFu;
    int e;
    if (ex == 0) {
        e = -126 - 23;  // subnormal: value = man * 2^-149
    } else {
        man |= 0x800000u;
        e = (int)ex - 127 - 23;  // value = man * 2^e
    }
    int s = e + shift;
    long long q;
    if (s >= 0) {
        q = (long long)man << s;
    } else if (s < -25) {
        q = 0;  // man < 2^24: the value is below 1/2
    } else {
        int r = -s;
        uint32_t qq = man >> r;
        uint32_t rem = man & ((1u << r) - 1u);
        uint32_t half = 1u << (r - 1);
        if (rem > half || (rem == half && (qq & 1u))) qq++;
        q = (long long)qq;
    }
    return (bits >> 31) ? -q : q;
}

// exponent e with 2^(e-1) <= |v| < 2^e (0 for v == 0), as frexpf, read from the
// bits: normal v of biased exponent E gives E - 126; a subnormal with an
// n-bit significand gives n - 149
MNMT_DEV int exp_bound(float v) {
    const uint32_t a = __float_as_uint(v) & 0x7FFFFFFFu;
    const int E = (int)(a >> 23);
    if (E != 0) return E - 126;
    return a == 0 ? 0 : (32 - __clz((int)a)) - 149;
}

// ---------------------------------------------------------------------------
// e^x for x <= 0: Cody-Waite reduction with ln2 split into a 16-bit head and
// a tail, degree-7 Taylor polynomial of e^r by Horner in fused multiply-adds,
// scaled by 2^n through the exponent field; 0 below -87.
// ---------------------------------------------------------------------------
MNMT_DEV float exp_own(float x) {
    if (x < -87.0f) return 0.0f;
    // n = rne(x log2(e)) in [-126, 0] by adding 1.5 2^23 (ulp 1 there: the sum
    // rounds the fraction half to even and its low bits hold n)
    const float t = __fadd_rn(__fmul_rn(x, 0x1.715476p+0f), 12582912.0f);
    const float n = __fsub_rn(t, 12582912.0f);
    float r = __fmaf_rn(-n, 0x1.62e4p-1f, x);
    r = __fmaf_rn(-n, 0x1.7f7d1cp-20f, r);
    float p = 0x1.a01a02p-13f;
    p = __fmaf_rn(p, r, 0x1.6c16c2p-10f);
    p = __fmaf_rn(p, r, 0x1.111112p-7f);
    p = __fmaf_rn(p, r, 0x1.555556p-5f);
    p = __fmaf_rn(p, r, 0x1.555556p-3f);
    p = __fmaf_rn(p, r, 0.5f);
    p = __fmaf_rn(p, r, 1.0f);
    p = __fmaf_rn(p, r, 1.0f);
    const int ni = (int)(__float_as_uint(t) - 0x4B400000u);
    float two_n = __uint_as_float((uint32_t)(ni + 127) << 23);
    return __fmul_rn(p, two_n);
}

// softmax weight on the 2^-24 grid: rne(exp(x) * 2^24), x <= 0
MNMT_DEV int32_t softmax_weight(float x) {
    return __float2int_rn(__fmul_rn(exp_own(x), 16777216.0f));
}

// natural log in double for z >= 1: z = f 2^k, f in [sqrt(1/2), sqrt(2)),
// ln f = 2 atanh(s), s = (f - 1)/(f + 1), odd series up to s^23.
MNMT_DEV double log_own(double z) {
    int k;
    double f = frexp(z, &k);
    if (f < 0x1.6a09e667f3bcdp-1) {
        f = __dmul_rn(f, 2.0);
        k = k - 1;
    }
    double s = __ddiv_rn(__dadd_rn(f, -1.0), __dadd_rn(f, 1.0));
    double s2 = __dmul_rn(s, s);
    double q = 0x1.642c8590b2164p-5;
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.8618618618618p-5);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.af286bca1af28p-5);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.e1e1e1e1e1e1ep-5);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.1111111111111p-4);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.3b13b13b13b14p-4);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.745d1745d1746p-4);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.c71c71c71c71cp-4);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.2492492492492p-3);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.999999999999ap-3);
    q = __dadd_rn(__dmul_rn(q, s2), 0x1.5555555555555p-2);
    q = __dadd_rn(__dmul_rn(q, s2), 1.0);
    return __dadd_rn(__dmul_rn(__dmul_rn(2.0, s), q), __dmul_rn((double)k, 0x1.62e42fefa39efp-1));
}

// ---------------------------------------------------------------------------
// Ordering keys: a float and an index packed so that unsigned max picks the
// larger float, and between equal floats the lower index (-0 counts as +0).
// ---------------------------------------------------------------------------
MNMT_DEV uint32_t ordered_bits(float f) {
    uint32_t u = __float_as_uint(__fadd_rn(f, 0.0f));  // -0 + 0 = +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
MNMT_DEV float from_ordered_bits(uint32_t o) {
    uint32_t u = (o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o;
    return __uint_as_float(u);
}
MNMT_DEV unsigned long long pack_key(float f, uint32_t idx) {
    return ((unsigned long long)ordered_bits(f) << 32) | (unsigned long long)(0xFFFFFFFFu - idx);
}
MNMT_DEV uint32_t key_index(unsigned long long k) { return 0xFFFFFFFFu - (uint32_t)(k & 0xFFFFFFFFull); }
MNMT_DEV float key_value(unsigned long long k) { return from_ordered_bits((uint32_t)(k >> 32)); }

// ---------------------------------------------------------------------------
// warp reductions
// ---------------------------------------------------------------------------
MNMT_DEV float warp_max_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    return v;
}
MNMT_DEV long long warp_sum_ll(long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}
MNMT_DEV int warp_sum_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}
MNMT_DEV unsigned long long warp_max_u64(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xFFFFFFFFu, v, o);
        v = w > v ? w : v;
    }
    return v;
}

// dp4a over 16 bytes held as int4
MNMT_DEV int dot16(int4 a, int4 b, int acc) {
    acc = __dp4a(a.x, b.x, acc);
    acc = __dp4a(a.y, b.y, acc);
    acc = __dp4a(a.z, b.z, acc);
    acc = __dp4a(a.w, b.w, acc);
    return acc;
}

// ---------------------------------------------------------------------------
// Exact roundings to fp32 with integer operations only (no double precision,
// which is slow on this part).
// ---------------------------------------------------------------------------
// nearest float (ties to even) to S * 2^e, subnormals included
MNMT_DEV float rn32_pow2(long long S, int e) {
    if (S == 0) return 0.0f;
    {
        // fast path: the integer rounds to float once (half to even); scaling
        // by 2^e is exact while the result stays a normal float
        const float f = __ll2float_rn(S);
        const uint32_t fb = __float_as_uint(f);
        const int fe = (int)((fb >> 23) & 0xFFu) + e;
        if (fe >= 1 && fe <= 254) return __uint_as_float(fb + ((uint32_t)e << 23));
    }
    const unsigned long long a = S < 0 ? 0ull - (unsigned long long)S : (unsigned long long)S;
    const int nb = 64 - __clzll(a);  // significant bits of a
    const int E = nb - 1 + e;        // floor(log2 |value|)
    const int p = E >= -126 ? 24 : 150 + E;  // bits the float keeps
    const int shift = nb - p;
    unsigned long long q;
    if (shift <= 0) {
        q = a << (-shift);
    } else if (shift > 64) {
        q = 0;
    } else {
        q = shift == 64 ? 0ull : (a >> shift);
        const unsigned long long rem = shift == 64 ? a : (a & ((1ull << shift) - 1ull));
        const unsigned long long half = 1ull << (shift - 1);
        if (rem > half || (rem == half && (q & 1ull))) q++;
    }
    uint32_t bits;
    if (E >= -126) {
        int EE = E;
        if (q == (1ull << 24)) {
            q >>= 1;
            EE++;
        }
        bits = EE > 127 ? 0x7F800000u : (((uint32_t)(EE + 127) << 23) | (uint32_t)(q - (1ull << 23)));
    } else {
        bits = (uint32_t)q;  // subnormal, or the smallest normal after a carry
    }
    if (S < 0) bits |= 0x80000000u;
    return __uint_as_float(bits);
}

// nearest float (ties to even) to S * 2^e / d for 1 <= d <= 2048 and
// |S| < 2^63: the LayerNorm's mean and variance, S an exact fixed-point sum of
// d terms.  With d = z 2^k (z odd) and z = 1 this is rn32_pow2.  Otherwise
// |S| is shifted so the integer quotient q = floor(|S| 2^t / z) keeps at least
// 50 significant bits; the float keeps at most 24 of them, so the remainder
// only decides whether the value lies exactly on q or strictly above it, which
// one appended sticky bit (2q + [r != 0]) tells rn32_pow2 without moving the
// value across a rounding boundary.
MNMT_DEV float rn32_scaled_div(long long S, int e, int d) {
    const int k = __ffs(d) - 1;
    const unsigned z = (unsigned)d >> k;
    if (z == 1u) return rn32_pow2(S, e - k);
    if (S == 0) return 0.0f;
    const unsigned long long a = S < 0 ? 0ull - (unsigned long long)S : (unsigned long long)S;
    const int nb = 64 - __clzll(a);
    const int t = nb < 62 ? 62 - nb : 0;
    const unsigned long long num = a << t;
    const unsigned long long q = num / z, r = num - q * z;
    const float f = rn32_pow2((long long)(2ull * q + (r != 0ull ? 1ull : 0ull)), e - k - t - 1);
    return S < 0 ? -f : f;
}

// sign of a - X * 2^E for a < 2^62, X < 2^63
MNMT_DEV int cmp_scaled(unsigned long long a, unsigned long long X, int E) {
    if (E >= 0) {
        if (X == 0) return a > 0 ? 1 : 0;
        if (64 - __clzll(X) + E > 62) return -1;  // X 2^E >= 2^62 > a
        const unsigned long long v = X << E;
        return a > v ? 1 : (a < v ? -1 : 0);
    }
    const int s = -E;
    const unsigned long long qx = s >= 64 ? 0ull : (X >> s);
    const unsigned long long rx = s >= 64 ? X : (X & ((1ull << s) - 1ull));
    if (a > qx) return 1;
    if (a < qx) return -1;
    return rx ? -1 : 0;
}

// nearest float (ties to even) to the exact quotient n / z, |n| < 2^41, 1 <= z < 2^35
MNMT_DEV float rn32_div(long long n, long long z) {
    if (n == 0) return 0.0f;
    const unsigned long long a = n < 0 ? 0ull - (unsigned long long)n : (unsigned long long)n;
    float q = __fdiv_rn(__ull2float_rn(a), __ll2float_rn(z));  // within a few ulp of a / z
    for (int it = 0; it < 8; it++) {
        const uint32_t qb = __float_as_uint(q);
        const unsigned long long mq = (qb & 0x7FFFFFu) | 0x800000u;  // q = mq 2^eq (normal: a/z > 2^-35)
        const int eq = (int)((qb >> 23) & 0xFFu) - 150;
        // midpoint above: (2 mq + 1) 2^(eq-1); below: (2 mq - 1) 2^(eq-1), or (2^25 - 1) 2^(eq-2) at a power of two
        const int up = cmp_scaled(a, (unsigned long long)z * (2ull * mq + 1ull), eq - 1);
        if (up > 0 || (up == 0 && (mq & 1ull))) {
            q = __uint_as_float(qb + 1u);
            continue;
        }
        const bool pow2 = mq == 0x800000ull;
        const int dn = pow2 ? cmp_scaled(a, (unsigned long long)z * ((1ull << 25) - 1ull), eq - 2)
                            : cmp_scaled(a, (unsigned long long)z * (2ull * mq - 1ull), eq - 1);
        if (dn < 0 || (dn == 0 && (mq & 1ull))) {
            q = __uint_as_float(qb - 1u);
            continue;
        }
        break;
    }
    return n < 0 ? -q : q;
}

// q8(nearest float to n / z, rho): the quantised attention context of Eq. 2.
// The approximate quotient fl(fl(n) / fl(z)) is within 2^-22 (relative) of
// the exact rounded one -- three roundings of 2^-24 each, plus the exact
// quotient's own -- which is at most 4 ulp, 8 across a binade boundary;
// fl(x * rho), the rounding and the clamp are monotone in x, so when both ends
// of the +-8-ulp bracket give the same code, so does the exact quotient.  Only
// a bracket that straddles a rounding boundary needs the exact quotient.
template <typename ExactDiv>
MNMT_DEV int8_t q8_quotient(long long n, long long z, float rho, ExactDiv exact) {
    if (n == 0) return q8(0.0f, rho);
    const unsigned long long a = n < 0 ? 0ull - (unsigned long long)n : (unsigned long long)n;
    const uint32_t qb = __float_as_uint(__fdiv_rn(__ull2float_rn(a), __ll2float_rn(z)));
    const float sgn = n < 0 ? -1.0f : 1.0f;
    const int8_t lo = q8(__fmul_rn(sgn, __uint_as_float(qb - 8u)), rho);
    const int8_t hi = q8(__fmul_rn(sgn, __uint_as_float(qb + 8u)), rho);
    if (lo == hi) return lo;
    return q8(exact(n, z), rho);
}

// ---------------------------------------------------------------------------
// LayerNorm (App. A / App. D) of one row by one warp.  Mean and biased
// variance are exact fixed-point sums: the row's largest magnitude (an
// order-free maximum) sets a power-of-two grid on which every term is an
// integer below 2^52, summed in int64, so any reduction order gives the same
// bits; each sum / d is rounded once to fp32 (rn32_scaled_div); rstd =
// 1 / sqrt(var + 1e-5) in IEEE fp32; returns false if |x| >= 2^32.
// warp LayerNorm over a row held as VPL values per lane (element u*32 + lane)
// ---------------------------------------------------------------------------
// exact warp sum of int64 values with |v| < 2^58 per lane: three 20-bit
// pieces summed by single-instruction warp reductions
MNMT_DEV long long warp_sum_exact(long long v) {
    int p0 = (int)(v & 0xFFFFF), p1 = (int)((v >> 20) & 0xFFFFF), p2 = (int)(v >> 40);
    p0 = __reduce_add_sync(0xFFFFFFFFu, p0);
    p1 = __reduce_add_sync(0xFFFFFFFFu, p1);
    p2 = __reduce_add_sync(0xFFFFFFFFu, p2);
    return (long long)p0 + (long long)p1 * (1LL << 20) + (long long)p2 * (1LL << 40);
}

// LayerNorm of one row held by a warp (x[u] = element u*32 + lane); gv / bv
// are the matching gamma / beta values, loaded by the caller
template <int VPL>
MNMT_DEV bool warp_layernorm_v(const float (&x)[VPL], int d, const float (&gv)[VPL], const float (&bv)[VPL],
                               float (&out)[VPL], int lane) {
    unsigned amax_bits = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) amax_bits = max(amax_bits, __float_as_uint(x[u]) & 0x7FFFFFFFu);
    const float amax = __uint_as_float(__reduce_max_sync(0xFFFFFFFFu, amax_bits));
    if (!(amax < 0x1p32f)) return false;
    const int ea = exp_bound(amax);
    long long s1 = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) s1 += fx_scale(x[u], 52 - ea);
    s1 = warp_sum_exact(s1);
    const float mu = rn32_scaled_div(s1, ea - 52, d);
    float c[VPL];
    unsigned bmax_bits = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++) {
        c[u] = __fsub_rn(x[u], mu);
        if (u * 32 + lane < d) bmax_bits = max(bmax_bits, __float_as_uint(c[u]) & 0x7FFFFFFFu);
    }
    const int eb = exp_bound(__uint_as_float(__reduce_max_sync(0xFFFFFFFFu, bmax_bits)));
    long long s2 = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) s2 += fx_scale(__fmul_rn(c[u], c[u]), 52 - 2 * eb);
    s2 = warp_sum_exact(s2);
    const float var = rn32_scaled_div(s2, 2 * eb - 52, d);
    const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, 1e-5f)));
#pragma unroll
    for (int u = 0; u < VPL; u++) out[u] = __fadd_rn(__fmul_rn(__fmul_rn(c[u], rstd), gv[u]), bv[u]);
    return true;
}

template <int VPL>
MNMT_DEV bool warp_layernorm(const float (&x)[VPL], int d, const float *__restrict__ g,
                             const float *__restrict__ b, float (&out)[VPL], int lane) {
    unsigned amax_bits = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) amax_bits = max(amax_bits, __float_as_uint(x[u]) & 0x7FFFFFFFu);
    const float amax = __uint_as_float(__reduce_max_sync(0xFFFFFFFFu, amax_bits));
    if (!(amax < 0x1p32f)) return false;
    const int ea = exp_bound(amax);
    long long s1 = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) s1 += fx_scale(x[u], 52 - ea);
    s1 = warp_sum_exact(s1);
    const float mu = rn32_scaled_div(s1, ea - 52, d);
    float c[VPL];
    unsigned bmax_bits = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++) {
        c[u] = __fsub_rn(x[u], mu);
        if (u * 32 + lane < d) bmax_bits = max(bmax_bits, __float_as_uint(c[u]) & 0x7FFFFFFFu);
    }
    const int eb = exp_bound(__uint_as_float(__reduce_max_sync(0xFFFFFFFFu, bmax_bits)));
    long long s2 = 0;
#pragma unroll
    for (int u = 0; u < VPL; u++)
        if (u * 32 + lane < d) s2 += fx_scale(__fmul_rn(c[u], c[u]), 52 - 2 * eb);
    s2 = warp_sum_exact(s2);
    const float var = rn32_scaled_div(s2, 2 * eb - 52, d);
    const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, 1e-5f)));
#pragma unroll
    for (int u = 0; u < VPL; u++) {
        int i = u * 32 + lane;
        if (i < d) out[u] = __fadd_rn(__fmul_rn(__fmul_rn(c[u], rstd), g[i]), b[i]);
    }
    return true;
}

MNMT_DEV bool warp_layernorm16(const float (&x)[16], int d, const float *g, const float *b, float (&out)[16],
                               int lane) {
    return warp_layernorm<16>(x, d, g, b, out, lane);
}

// device-side status word: first error wins
MNMT_DEV void set_status(int *status, int code) {
    if (status) atomicCAS(status, 0, code);
}
