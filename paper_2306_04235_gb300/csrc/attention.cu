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
    return err;
}
}  // namespace mnmt
