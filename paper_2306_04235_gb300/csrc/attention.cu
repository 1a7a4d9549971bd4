// attention.cu -- scaled dot-product attention of the INT8 encoder-decoder
// (App. A, Eq. 1/2) per head, with the quantisation points of Fig. 5b: int8 Q,
// K, V and context; the softmax in full precision.
//
// Per head and query row: scores acc_j = q . k_j (exact int32, dp4a),
// s_j = fl(acc_j * sigma), m = max_j s_j, weights E_j = rne(exp(fl(s_j - m)) 2^24)
// (an integer in [0, 2^24]), context N_e = sum_j E_j v_j[e] and Z = sum_j E_j as
// exact integer sums (so any summation order gives the same bits), then
// ctx_e = q8(nearest fp32 to N_e / Z, rho).  N_e is accumulated in two int32 halves,
// E_j = Eh 2^12 + El, which cannot overflow for up to 1024 keys.
//
// Kernels:
//   attn_decode  one warp per (row, head): the incremental step of the decoder
//                over the self-attention cache (keys 0..t, through the beam
//                ancestry table when hypotheses were reordered) or over the
//                cross-attention keys of the row's sentence.  Bound by the
//                cache bytes it streams.
//   attn_encoder one block per (sentence, head, chunk of 4..32 queries): K and V of
//                the head staged in shared memory, keys masked past the
//                source length.
//   attn_encoder_mma  the same on the int8 tensor cores (mma.sync, exact int32)
//                for d_h = 64 and up to 256 keys: scores as one product, the
//                weights split into bytes for the context products.
#include <type_traits>

#include "common.cuh"
#include "internal.h"

namespace mnmt {

constexpr int DEC_MAX_KEYS = 1024;

// 32-bit word k of a 4-, 8- or 16-byte vector held in registers
MNMT_DEV uint32_t vec_word(uint32_t v, int) { return v; }
MNMT_DEV uint32_t vec_word(const uint2 &v, int k) { return k ? v.y : v.x; }
MNMT_DEV uint32_t vec_word(const uint4 &v, int k) { return k == 0 ? v.x : k == 1 ? v.y : k == 2 ? v.z : v.w; }

// XS = false: one block per row, one warp per head.  XS = true (cross
// attention with beams): one block per sentence, one warp per (beam, head) --
// the beams of a sentence read the same keys and values, which their block
// then fetches from L2 once and serves from L1.
template <int DH, bool XS>
__global__ void __launch_bounds__(XS ? 32 * 32 : 32 * 16) attn_decode(AttnDecArgs a) {
    pdl_grid_wait();
    if (a.skip && *a.skip) return;
    extern __shared__ int dsm[];
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = XS ? blockIdx.x * a.beam + w / a.H : blockIdx.x;
    const int h = XS ? w % a.H : w;
    int n, t = 0;
    if (a.cross) {
        n = a.src_len[r / a.beam];
        n = n < 1 ? 1 : (n > a.T ? a.T : n);  // lengths are validated on the host path; clamp on the device path
    } else if (a.n_keys) {
        n = a.n_keys[r];
        t = n - 1;
    } else {
        t = *a.t_ptr;
        n = t + 1;
    }
    const int cap = a.T;  // key capacity: cache length / padded source length
    int *prow = dsm;      // [cap] physical row of every key position (shared by the heads of this row)
    int *sc = XS ? dsm + w * cap : dsm + cap + h * cap;  // per warp [cap]: scores, then weights
    if (!XS) {
        for (int j = threadIdx.x; j < n; j += blockDim.x) {
            int p;
            if (a.cross) p = r / a.beam;
            else p = (a.anc && j < t) ? a.anc[(size_t)r * a.T + j] : r;
            prow[j] = p;
        }
        __syncthreads();
        if (h >= a.H) return;
    }
    const int psent = r / a.beam;  // XS: the sentence of every key
    auto prow_of = [&](int j) { return XS ? psent : prow[j]; };

    constexpr int QC = DH / 16;
    int4 qv[QC];
    const int4 *qp = reinterpret_cast<const int4 *>(a.q + (size_t)r * a.H * DH + h * DH);
#pragma unroll
    for (int c = 0; c < QC; c++) qv[c] = qp[c];

    float mx = -INFINITY;
#pragma unroll 4
    for (int j = lane; j < n; j += 32) {
        const int4 *kr = reinterpret_cast<const int4 *>(a.kc + (((size_t)prow_of(j) * a.H + h) * a.T + j) * DH);
        int acc = 0;
#pragma unroll
        for (int c = 0; c < QC; c++) acc = dot16(qv[c], kr[c], acc);
        float s = __fmul_rn(__int2float_rn(acc), a.sigma);
        sc[j] = __float_as_int(s);
        mx = fmaxf(mx, s);
    }
    mx = warp_max_f(mx);
    long long Z = 0;
    for (int j = lane; j < n; j += 32) {
        int E = softmax_weight(__fadd_rn(__int_as_float(sc[j]), -mx));
        sc[j] = E;
        Z += E;
    }
    Z = warp_sum_ll(Z);
    __syncwarp();

    // context: the warp takes CG keys at a time, one per group of 8 lanes;
    // lane gl of a group holds EPG consecutive elements of the head, read as
    // one EPG-byte load per key.  N_e = sum_j E_j v_j[e] is split into 12-bit
    // halves of E_j so that every partial stays an exact int32.
    constexpr int CG = 4, LPG = 32 / CG, EPG = DH / LPG;
    using VecT = typename std::conditional<EPG == 4, uint32_t, typename std::conditional<EPG == 8, uint2, uint4>::type>::type;
    const int grp = lane / LPG, gl = lane % LPG;
    int hi[EPG], lo[EPG];
#pragma unroll
    for (int u = 0; u < EPG; u++) hi[u] = lo[u] = 0;
    auto vload = [&](int j) -> VecT {
        return *reinterpret_cast<const VecT *>(a.vc + (((size_t)prow_of(j) * a.H + h) * a.T + j) * DH + gl * EPG);
    };
    auto vacc = [&](int j, const VecT &raw) {
        const int E = sc[j];
        const int Eh = E >> 12, El = E & 4095;
#pragma unroll
        for (int u = 0; u < EPG; u++) {
            const int v = (int)(int8_t)(vec_word(raw, u >> 2) >> (8 * (u & 3)));
            hi[u] += Eh * v;
            lo[u] += El * v;
        }
    };
    // groups of UJ rounds: every value load of the batch is issued before any
    // is used, so their latencies overlap
    constexpr int UJ = DH == 128 ? 2 : 4;
    int j0 = 0;
    for (; j0 + CG * UJ <= n; j0 += CG * UJ) {
        VecT raw[UJ];
#pragma unroll
        for (int u = 0; u < UJ; u++) raw[u] = vload(j0 + u * CG + grp);
#pragma unroll
        for (int u = 0; u < UJ; u++) vacc(j0 + u * CG + grp, raw[u]);
    }
    for (int j = j0 + grp; j < n; j += CG) vacc(j, vload(j));
    // sum over the CG groups (lanes gl, gl+8, gl+16, gl+24): every lane gets the totals
#pragma unroll
    for (int u = 0; u < EPG; u++) {
#pragma unroll
        for (int o = LPG; o < 32; o <<= 1) {
            hi[u] += __shfl_xor_sync(0xFFFFFFFFu, hi[u], o);
            lo[u] += __shfl_xor_sync(0xFFFFFFFFu, lo[u], o);
        }
    }
    // lane (grp, gl) writes elements gl * EPG + grp * EPG / CG + [0, EPG / CG)
    constexpr int OPL = EPG / CG;
    const size_t o = (size_t)r * a.H * DH + h * DH + gl * EPG + grp * OPL;
#pragma unroll
    for (int u = 0; u < EPG; u++) {
        if (u / OPL == grp) {
            long long N = (long long)hi[u] * 4096 + lo[u];
            const int8_t v = q8_quotient(N, Z, a.rho, rn32_div);
            a.ctx[o + u - grp * OPL] = v;
            if (a.ctx16) a.ctx16[o + u - grp * OPL] = __short2half_rn(v);
        }
    }
}

cudaError_t launch_attention_decode(const AttnDecArgs &a, cudaStream_t st) {
    if (a.H > 16 || a.T < 1 || a.T > DEC_MAX_KEYS) return cudaErrorInvalidValue;
    // cross attention with beams: the beams of a sentence share a block, when
    // there are sentences enough for half of the SMs (measured on 152 SMs:
    // 3.8 us per step faster at 128 sentences, 1.7 us slower at 32)
    const bool xs = a.cross && a.beam > 1 && a.beam * a.H <= 32 && a.R % a.beam == 0 &&
                    2 * (a.R / a.beam) >= device_sm_count();
    const size_t smem = (size_t)(xs ? a.beam * a.H : 1 + a.H) * a.T * sizeof(int);
    const dim3 block(32 * a.H * (xs ? a.beam : 1));
    const int grid = xs ? a.R / a.beam : a.R;
    switch (a.dh) {
        case 32:
            if (xs) launch_pdl(attn_decode<32, true>, grid, block, smem, st, a);
            else launch_pdl(attn_decode<32, false>, grid, block, smem, st, a);
            break;
        case 64:
            if (xs) launch_pdl(attn_decode<64, true>, grid, block, smem, st, a);
            else launch_pdl(attn_decode<64, false>, grid, block, smem, st, a);
            break;
        case 128:
            if (xs) launch_pdl(attn_decode<128, true>, grid, block, smem, st, a);
            else launch_pdl(attn_decode<128, false>, grid, block, smem, st, a);
            break;
        default:
            return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// encoder self-attention
// ---------------------------------------------------------------------------
constexpr int ENC_WARPS = 4;
constexpr int ENC_MAX_KEYS = 512;
constexpr int ENC_QCHUNK = 32;

template <int DH>
__global__ void __launch_bounds__(32 * ENC_WARPS) attn_encoder(AttnEncArgs a, int qchunk) {
    pdl_grid_wait();
    extern __shared__ __align__(16) uint8_t esm[];
    constexpr int KS = DH + 16;  // padded key row: conflict-free 16-byte lane reads
    const int bh = blockIdx.x;
    const int b = bh / a.H, h = bh - b * a.H;
    const int S = a.S;
    int len = a.len[b];
    len = len < 1 ? 1 : (len > S ? S : len);  // validated on the host path; clamp on the device path
    uint8_t *Ks = esm;                         // [S][KS]
    int8_t *Vs = reinterpret_cast<int8_t *>(esm + (size_t)S * KS);  // [S][DH]
    int *wsm = reinterpret_cast<int *>(esm + (size_t)S * KS + (size_t)S * DH);  // [warps][S]
    const int ld = 3 * a.d;
    const int8_t *base = a.qkv + (size_t)b * S * ld;
    // stage K and V of this head (valid keys only)
    constexpr int CH = DH / 16;
    for (int i = threadIdx.x; i < len * CH; i += blockDim.x) {
        int j = i / CH, c = i - j * CH;
        const int4 *src = reinterpret_cast<const int4 *>(base + (size_t)j * ld + a.d + h * DH);
        reinterpret_cast<int4 *>(Ks + (size_t)j * KS)[c] = src[c];
        const int4 *vsrc = reinterpret_cast<const int4 *>(base + (size_t)j * ld + 2 * a.d + h * DH);
        reinterpret_cast<int4 *>(Vs + (size_t)j * DH)[c] = vsrc[c];
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    int *sc = wsm + warp * S;
    const int q0 = blockIdx.y * qchunk;
    const int q1 = min(q0 + qchunk, S);
    constexpr int EPL = DH / 32;
    for (int qi = q0 + warp; qi < q1; qi += ENC_WARPS) {
        int4 qv[CH];
        const int4 *qp = reinterpret_cast<const int4 *>(base + (size_t)qi * ld + h * DH);
#pragma unroll
        for (int c = 0; c < CH; c++) qv[c] = qp[c];
        float mx = -INFINITY;
        for (int j = lane; j < len; j += 32) {
            const int4 *kr = reinterpret_cast<const int4 *>(Ks + (size_t)j * KS);
            int acc = 0;
#pragma unroll
            for (int c = 0; c < CH; c++) acc = dot16(qv[c], kr[c], acc);
            float s = __fmul_rn(__int2float_rn(acc), a.sigma);
            sc[j] = __float_as_int(s);
            mx = fmaxf(mx, s);
        }
        mx = warp_max_f(mx);
        long long Z = 0;
        for (int j = lane; j < len; j += 32) {
            int E = softmax_weight(__fadd_rn(__int_as_float(sc[j]), -mx));
            sc[j] = E;
            Z += E;
        }
        Z = warp_sum_ll(Z);
        __syncwarp();
        int hi[EPL], lo[EPL];
#pragma unroll
        for (int u = 0; u < EPL; u++) hi[u] = lo[u] = 0;
        for (int j = 0; j < len; j++) {
            int E = sc[j];
            int Eh = E >> 12, El = E & 4095;
            const int8_t *vr = Vs + (size_t)j * DH + lane * EPL;
#pragma unroll
            for (int u = 0; u < EPL; u++) {
                int v = vr[u];
                hi[u] += Eh * v;
                lo[u] += El * v;
            }
        }
        const size_t o = ((size_t)b * S + qi) * a.d + h * DH + lane * EPL;
#pragma unroll
        for (int u = 0; u < EPL; u++) {
            long long N = (long long)hi[u] * 4096 + lo[u];
            const int8_t v = q8_quotient(N, Z, a.rho, rn32_div);
            a.ctx[o + u] = v;
            if (a.ctx16) a.ctx16[o + u] = __short2half_rn(v);
        }
        __syncwarp();
    }
}

// ---------------------------------------------------------------------------
// encoder self-attention on the int8 tensor cores (mma.sync m16n8k32, exact
// int32 accumulation), d_h = 64 and up to 256 keys.  Same arithmetic as
// attn_encoder: the scores q . k_j are the same exact integers; the weights E_j
// in [0, 2^24] are split into four bytes E_j = sum_k e_kj 2^(8k), each byte a
// u8 operand of its own product with V (sum_j e_kj v_j[e] <= 256 * 255 * 128 <
// 2^31: exact), and N_e = sum_k 2^(8k) (sum_j e_kj v_j[e]) is rebuilt in int64.
//
// One block per (sentence, head, 64 queries), four warps of 16 queries each.
// Shared memory: Q [64][64] and K [Sp][64] in 64-byte rows, V^T [64][Sp], and
// per warp the weight bytes [4][16][Sp] (Sp = key count padded to a power of
// two >= 32), 16-byte chunks XOR-swizzled by row so that ldmatrix phases hit
// distinct bank groups.  Keys past the source length score -inf (weight 0).
// ---------------------------------------------------------------------------
constexpr int ENC_MMA_WARPS = 4;

MNMT_DEV uint32_t att_smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
MNMT_DEV void att_ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
MNMT_DEV void att_mma_s8(int (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
MNMT_DEV void att_mma_u8s8(int (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.u8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
// byte offset of (row, 16-byte chunk) in 64-byte rows: chunk ^ (row / 2) % 4
MNMT_DEV int sw64(int row, int chunk) { return row * 64 + ((chunk ^ ((row >> 1) & 3)) << 4); }
// byte offset of (row, byte col) in rows of `len` bytes (len = 16 * nch, nch a
// power of two): chunk ^ (row mod min(nch, 8))
MNMT_DEV int swl(int row, int col, int len, int msk) {
    return row * len + ((((col >> 4) ^ (row & msk))) << 4) + (col & 15);
}

__global__ void __launch_bounds__(32 * ENC_MMA_WARPS) attn_encoder_mma(AttnEncArgs a, int Sp) {
    pdl_grid_wait();
    extern __shared__ __align__(128) uint8_t emm[];
    constexpr int DH = 64;
    const int bh = blockIdx.x;
    const int b = bh / a.H, h = bh - b * a.H;
    const int S = a.S;
    int len = a.len[b];
    len = len < 1 ? 1 : (len > S ? S : len);
    const int q0 = blockIdx.y * 64;
    const int nch = Sp >> 4, msk = (nch < 8 ? nch : 8) - 1;
    uint8_t *Qs = emm;                       // [64][64]
    uint8_t *Ks = Qs + 64 * 64;              // [Sp][64]
    uint8_t *Vt = Ks + (size_t)Sp * 64;      // [64][Sp]
    uint8_t *Es = Vt + (size_t)64 * Sp;      // [warps][4][16][Sp]; first V row-major [Sp][64]
    const int ld = 3 * a.d;
    const int8_t *base = a.qkv + (size_t)b * S * ld;
    // stage Q (64 queries), K and V (valid keys; the rest zero)
    for (int i = threadIdx.x; i < 64 * 4; i += blockDim.x) {
        const int r = i >> 2, c = i & 3, q = q0 + r;
        int4 v = make_int4(0, 0, 0, 0);
        if (q < S) v = reinterpret_cast<const int4 *>(base + (size_t)q * ld + h * DH)[c];
        *reinterpret_cast<int4 *>(Qs + sw64(r, c)) = v;
    }
    for (int i = threadIdx.x; i < Sp * 4; i += blockDim.x) {
        const int j = i >> 2, c = i & 3;
        int4 kv = make_int4(0, 0, 0, 0), vv = make_int4(0, 0, 0, 0);
        if (j < len) {
            kv = reinterpret_cast<const int4 *>(base + (size_t)j * ld + a.d + h * DH)[c];
            vv = reinterpret_cast<const int4 *>(base + (size_t)j * ld + 2 * a.d + h * DH)[c];
        }
        *reinterpret_cast<int4 *>(Ks + sw64(j, c)) = kv;
        reinterpret_cast<int4 *>(Es + (size_t)j * DH)[c] = vv;
    }
    __syncthreads();
    // V^T: word (e, keys 4w .. 4w + 3) from four rows of V
    for (int i = threadIdx.x; i < DH * (Sp >> 2); i += blockDim.x) {
        const int e = i & (DH - 1), j = 4 * (i >> 6);
        const uint32_t x = (uint32_t)Es[(size_t)j * DH + e] | ((uint32_t)Es[(size_t)(j + 1) * DH + e] << 8) |
                           ((uint32_t)Es[(size_t)(j + 2) * DH + e] << 16) |
                           ((uint32_t)Es[(size_t)(j + 3) * DH + e] << 24);
        *reinterpret_cast<uint32_t *>(Vt + swl(e, j, Sp, msk)) = x;
    }
    __syncthreads();

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int jq = lane >> 3, i8 = lane & 7, g = lane >> 2, tq = lane & 3;
    uint8_t *Ew = Es + (size_t)warp * 4 * 16 * Sp;
    // Q fragments of this warp's 16 queries (two k-steps of 32)
    uint32_t af[2][4];
#pragma unroll
    for (int kk = 0; kk < 2; kk++)
        att_ldmatrix_x4(af[kk], att_smem_u32(Qs + sw64(warp * 16 + (jq & 1) * 8 + i8, kk * 2 + (jq >> 1))));
    // scores of 16 keys (two n-tiles) per call: exact int32, then fl(acc sigma),
    // -inf past the source length
    auto scores16 = [&](int k0, float (&sv)[2][4]) {
        int acc[2][4] = {{0, 0, 0, 0}, {0, 0, 0, 0}};
#pragma unroll
        for (int kk = 0; kk < 2; kk++) {
            uint32_t r[4];
            att_ldmatrix_x4(r, att_smem_u32(Ks + sw64(k0 + (jq >> 1) * 8 + i8, kk * 2 + (jq & 1))));
            att_mma_s8(acc[0], af[kk], r[0], r[1]);
            att_mma_s8(acc[1], af[kk], r[2], r[3]);
        }
#pragma unroll
        for (int t = 0; t < 2; t++)
#pragma unroll
            for (int q = 0; q < 4; q++) {
                const int key = k0 + t * 8 + tq * 2 + (q & 1);
                sv[t][q] = key < len ? __fmul_rn(__int2float_rn(acc[t][q]), a.sigma) : -INFINITY;
            }
    };
    // pass 1: each row's maximum score
    float mx0 = -INFINITY, mx1 = -INFINITY;  // rows g and g + 8
    for (int k0 = 0; k0 < Sp; k0 += 16) {
        float sv[2][4];
        scores16(k0, sv);
#pragma unroll
        for (int t = 0; t < 2; t++) {
            mx0 = fmaxf(mx0, fmaxf(sv[t][0], sv[t][1]));
            mx1 = fmaxf(mx1, fmaxf(sv[t][2], sv[t][3]));
        }
    }
#pragma unroll
    for (int o = 1; o < 4; o <<= 1) {
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xFFFFFFFFu, mx0, o));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xFFFFFFFFu, mx1, o));
    }
    // pass 2: weights E (the scores again), their bytes into shared memory, Z
    long long z0 = 0, z1 = 0;
    for (int k0 = 0; k0 < Sp; k0 += 16) {
        float sv[2][4];
        scores16(k0, sv);
#pragma unroll
        for (int t = 0; t < 2; t++) {
            int E[4];
#pragma unroll
            for (int q = 0; q < 4; q++) E[q] = softmax_weight(__fadd_rn(sv[t][q], -(q < 2 ? mx0 : mx1)));
            z0 += (long long)E[0] + E[1];
            z1 += (long long)E[2] + E[3];
            const int key = k0 + t * 8 + tq * 2;
#pragma unroll
            for (int L = 0; L < 4; L++) {
                const uint32_t lo2 = ((uint32_t)(E[0] >> (8 * L)) & 255u) | (((uint32_t)(E[1] >> (8 * L)) & 255u) << 8);
                const uint32_t hi2 = ((uint32_t)(E[2] >> (8 * L)) & 255u) | (((uint32_t)(E[3] >> (8 * L)) & 255u) << 8);
                *reinterpret_cast<uint16_t *>(Ew + (size_t)L * 16 * Sp + swl(g, key, Sp, msk)) = (uint16_t)lo2;
                *reinterpret_cast<uint16_t *>(Ew + (size_t)L * 16 * Sp + swl(g + 8, key, Sp, msk)) = (uint16_t)hi2;
            }
        }
    }
#pragma unroll
    for (int o = 1; o < 4; o <<= 1) {
        z0 += __shfl_xor_sync(0xFFFFFFFFu, z0, o);
        z1 += __shfl_xor_sync(0xFFFFFFFFu, z1, o);
    }
    __syncwarp();
    // context: per weight byte L, sum_j e_Lj v_j[e] on the tensor cores (u8 x s8)
    long long N[8][4];
#pragma unroll
    for (int nt = 0; nt < 8; nt++)
#pragma unroll
        for (int q = 0; q < 4; q++) N[nt][q] = 0;
#pragma unroll 1
    for (int L = 0; L < 4; L++) {
        int acc[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; nt++)
#pragma unroll
            for (int q = 0; q < 4; q++) acc[nt][q] = 0;
        const uint8_t *EL = Ew + (size_t)L * 16 * Sp;
        for (int ks = 0; ks < (Sp >> 5); ks++) {
            uint32_t ea[4];
            att_ldmatrix_x4(ea, att_smem_u32(EL + swl((jq & 1) * 8 + i8, (ks * 2 + (jq >> 1)) * 16, Sp, msk)));
#pragma unroll
            for (int nj = 0; nj < 4; nj++) {
                uint32_t r[4];
                att_ldmatrix_x4(r, att_smem_u32(Vt + swl(nj * 16 + (jq >> 1) * 8 + i8, (ks * 2 + (jq & 1)) * 16, Sp, msk)));
                att_mma_u8s8(acc[2 * nj], ea, r[0], r[1]);
                att_mma_u8s8(acc[2 * nj + 1], ea, r[2], r[3]);
            }
        }
#pragma unroll
        for (int nt = 0; nt < 8; nt++)
#pragma unroll
            for (int q = 0; q < 4; q++) N[nt][q] += (long long)acc[nt][q] << (8 * L);
    }
    // row g (q < 2) or g + 8 of the warp's queries, element nt * 8 + 2 tq + (q & 1)
#pragma unroll
    for (int nt = 0; nt < 8; nt++)
#pragma unroll
        for (int q = 0; q < 4; q++) {
            const int qrow = q0 + warp * 16 + g + (q >> 1) * 8;
            if (qrow < S) {
                const int e = nt * 8 + tq * 2 + (q & 1);
                const int8_t v = q8_quotient(N[nt][q], q < 2 ? z0 : z1, a.rho, rn32_div);
                const size_t o = ((size_t)b * S + qrow) * a.d + h * DH + e;
                a.ctx[o] = v;
                if (a.ctx16) a.ctx16[o] = __short2half_rn(v);
            }
        }
}

static int enc_mma_keys(int S) {
    int sp = 32;
    while (sp < S) sp <<= 1;
    return sp;
}
static size_t enc_mma_smem(int Sp) { return 64 * 64 + (size_t)Sp * 64 * 2 + (size_t)ENC_MMA_WARPS * 4 * 16 * Sp; }
template <int DH>
static cudaError_t launch_enc(const AttnEncArgs &a, cudaStream_t st) {
    size_t smem = (size_t)a.S * (DH + 16) + (size_t)a.S * DH + (size_t)ENC_WARPS * a.S * sizeof(int);
    auto k = attn_encoder<DH>;
    // queries per block: the most (up to 32) that still gives every SM two
    // blocks; small batches get one query per warp so the GPU fills up
    int qc = ENC_QCHUNK;
    while (qc > ENC_WARPS && (long)a.B * a.H * ((a.S + qc - 1) / qc) < 2 * 152) qc >>= 1;
    dim3 grid(a.B * a.H, (a.S + qc - 1) / qc);
    launch_pdl(k, grid, 32 * ENC_WARPS, smem, st, a, qc);
    return cudaGetLastError();
}

cudaError_t launch_attention_encoder(const AttnEncArgs &a, cudaStream_t st) {
    if (a.S < 1 || a.S > ENC_MAX_KEYS) return cudaErrorInvalidValue;
    // the tensor-core kernel when its grid fills the GPU (a handful of
    // sentences run faster on the dp4a kernel's finer query chunks)
    if (a.dh == 64 && a.S <= 256 && (long)a.B * a.H * ((a.S + 63) / 64) >= device_sm_count()) {
        const int Sp = enc_mma_keys(a.S);
        dim3 grid(a.B * a.H, (a.S + 63) / 64);
        launch_pdl(attn_encoder_mma, grid, 32 * ENC_MMA_WARPS, enc_mma_smem(Sp), st, a, Sp);
        return cudaGetLastError();
    }
    switch (a.dh) {
        case 32:
            return launch_enc<32>(a, st);
        case 64:
            return launch_enc<64>(a, st);
        case 128:
            return launch_enc<128>(a, st);
        default:
            return cudaErrorInvalidValue;
    }
}

}  // namespace mnmt

namespace mnmt {
// Opt the attention kernels into the shared memory their largest shapes use
// (called once per process before any launch or stream capture).
cudaError_t attention_init() {
    cudaError_t err = cudaSuccess;
    int dec = (1 + 16) * DEC_MAX_KEYS * (int)sizeof(int);
    const int xs = 32 * DEC_MAX_KEYS * (int)sizeof(int);  // up to 32 (beam, head) warps
    if (!err) err = cudaFuncSetAttribute(attn_decode<32, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dec);
    if (!err) err = cudaFuncSetAttribute(attn_decode<64, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dec);
    if (!err) err = cudaFuncSetAttribute(attn_decode<128, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, dec);
    if (!err) err = cudaFuncSetAttribute(attn_decode<32, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, xs);
    if (!err) err = cudaFuncSetAttribute(attn_decode<64, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, xs);
    if (!err) err = cudaFuncSetAttribute(attn_decode<128, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, xs);
    auto enc = [](int dh) { return ENC_MAX_KEYS * (dh + 16) + ENC_MAX_KEYS * dh + ENC_WARPS * ENC_MAX_KEYS * 4; };
    if (!err) err = cudaFuncSetAttribute(attn_encoder<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, enc(32));
    if (!err) err = cudaFuncSetAttribute(attn_encoder<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, enc(64));
    if (!err) err = cudaFuncSetAttribute(attn_encoder<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, enc(128));
    if (!err)
        err = cudaFuncSetAttribute(attn_encoder_mma, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)enc_mma_smem(256));
    return err;
}
}  // namespace mnmt
