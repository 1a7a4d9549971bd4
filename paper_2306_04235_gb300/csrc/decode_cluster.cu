// decode_cluster.cu -- one decoder step of a small greedy batch (R <= 4 rows)
// on a single thread-block cluster, then the vocabulary projection fused with
// the greedy update.
//
// A batch-1 decode step is a chain of ~13 dependent matrix-vector products and
// two attentions per decoder layer (App. A), each only 16-260 KB of weights:
// the step is bound by latency, not bandwidth.  Instead of one kernel per
// operation, one cluster of NC CTAs (8 or 16 SMs) runs the whole decoder:
//   * every CTA holds the full activation vectors of the step in shared memory
//     (residual stream fp32 [R][d], LN output, q/k/v, context, FFN hidden);
//   * a linear layer is split by output columns: CTA c computes its column
//     slice from its weight slice and writes the result into the shared
//     memory of every CTA of the cluster (distributed shared memory), then a
//     hardware cluster barrier publishes it;
//   * LayerNorm and attention (all heads, the step's query rows) are computed
//     redundantly by every CTA, which removes two barriers per attention;
//   * each CTA streams its weight slices from L2/HBM into a 3-slot shared
//     memory ring with cp.async, two phases ahead of use.
// Per step: 1 + 6 * n_dec cluster barriers, no global synchronisation, no
// spin loops.  The arithmetic is exactly that of the other kernels (Fig. 5
// quantisation points, fixed-point LayerNorm and softmax), so the step is
// bit-identical to the multi-kernel path.
#include <cooperative_groups.h>

#include "common.cuh"
#include "internal.h"

namespace cg = cooperative_groups;

namespace mnmt {

constexpr int DC_THREADS = 256;
constexpr int DC_WARPS = DC_THREADS / 32;
constexpr int DC_NB = 3;  // weight ring slots

// ---------------------------------------------------------------------------
// helpers
// ---------------------------------------------------------------------------
MNMT_DEV uint32_t dc_smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
MNMT_DEV void dc_cp16(void *dst_smem, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dc_smem_u32(dst_smem)), "l"(src));
}
MNMT_DEV void dc_commit() { asm volatile("cp.async.commit_group;\n" ::); }
MNMT_DEV void dc_wait_ring() { asm volatile("cp.async.wait_group %0;\n" ::"n"(DC_NB - 2)); }

// signed bytes of a 32-bit word
MNMT_DEV int sb0(int x) { return (x << 24) >> 24; }
MNMT_DEV int sb1(int x) { return (x << 16) >> 24; }
MNMT_DEV int sb2(int x) { return (x << 8) >> 24; }
MNMT_DEV int sb3(int x) { return x >> 24; }

struct DcSlice {
    const int8_t *w;
    const float *s, *b;
    int rows, K;
};

// weight slice of phase ph for CTA c: phase 0 is the factorised embedding
// projection (empty when not factorised), then per layer qkv, o, q2, o2, w1, w2
MNMT_DEV DcSlice dc_slice(const DcParams &P, int ph, int c) {
    DcSlice s{nullptr, nullptr, nullptr, 0, 0};
    const int nsd = P.d / P.nc, ns3 = 3 * P.d / P.nc, nsf = P.F / P.nc;
    const DcLin *L = nullptr;
    int n0 = 0;
    if (ph == 0) {
        if (!P.factorised) return s;
        L = &P.proj;
        s.rows = nsd;
        s.K = P.E;
        n0 = c * nsd;
    } else {
        const int l = (ph - 1) / 6, k = (ph - 1) % 6;
        const DcLayer &Y = P.layer[l];
        switch (k) {
            case 0: L = &Y.qkv; s.rows = ns3; s.K = P.d; n0 = c * ns3; break;
            case 1: L = &Y.o; s.rows = nsd; s.K = P.d; n0 = c * nsd; break;
            case 2: L = &Y.q2; s.rows = nsd; s.K = P.d; n0 = c * nsd; break;
            case 3: L = &Y.o2; s.rows = nsd; s.K = P.d; n0 = c * nsd; break;
            case 4: L = &Y.w1; s.rows = nsf; s.K = P.d; n0 = c * nsf; break;
            default: L = &Y.w2; s.rows = nsd; s.K = P.F; n0 = c * nsd; break;
        }
    }
    s.w = L->w + (size_t)n0 * s.K;
    s.s = L->s + n0;
    s.b = L->b + n0;
    return s;
}

// ring slot layout: W rows (rows * K bytes), then s[rows], b[rows] (fp32)
MNMT_DEV void dc_prefetch(const DcParams &P, int ph, int c, uint8_t *ring, int slot_bytes, int nphase) {
    if (ph < nphase) {
        DcSlice s = dc_slice(P, ph, c);
        uint8_t *dst = ring + (size_t)(ph % DC_NB) * slot_bytes;
        const int wchunks = s.rows * s.K / 16, vchunks = s.rows * 4 / 16;
        for (int i = threadIdx.x; i < wchunks + 2 * vchunks; i += DC_THREADS) {
            if (i < wchunks) {
                dc_cp16(dst + i * 16, s.w + (size_t)i * 16);
            } else if (i < wchunks + vchunks) {
                int j = i - wchunks;
                dc_cp16(dst + wchunks * 16 + j * 16, reinterpret_cast<const uint8_t *>(s.s) + j * 16);
            } else {
                int j = i - wchunks - vchunks;
                dc_cp16(dst + wchunks * 16 + vchunks * 16 + j * 16, reinterpret_cast<const uint8_t *>(s.b) + j * 16);
            }
        }
    }
    dc_commit();
}

// y-values of a GEMV slice held in shared memory: for each local row n (of
// `rows`) and input row m (< R), acc = W[n] . A[m]; epi(m, n, acc, s_w, b)
template <typename F>
MNMT_DEV void dc_gemv(const uint8_t *slot, int rows, int K, const int8_t *A, int lda, int R, F epi) {
    const int8_t *W = reinterpret_cast<const int8_t *>(slot);
    const float *sw = reinterpret_cast<const float *>(slot + rows * K);
    const float *bb = sw + rows;
    const int kc = K / 16;
    const int lpc = kc >= 32 ? 32 : kc;  // K >= 128 so lpc >= 8
    const int gpw = 32 / lpc;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int grp = lane / lpc, sl = lane % lpc;
    for (int r0 = warp * gpw; r0 < rows; r0 += DC_WARPS * gpw) {
        const int n = r0 + grp;
        int acc[DC_RMAX];
#pragma unroll
        for (int m = 0; m < DC_RMAX; m++) acc[m] = 0;
        if (n < rows) {
            const int4 *wr = reinterpret_cast<const int4 *>(W + (size_t)n * K);
            for (int c = sl; c < kc; c += lpc) {
                int4 w = wr[c];
#pragma unroll
                for (int m = 0; m < DC_RMAX; m++)
                    if (m < R) acc[m] = dot16(reinterpret_cast<const int4 *>(A + (size_t)m * lda)[c], w, acc[m]);
            }
        }
#pragma unroll
        for (int m = 0; m < DC_RMAX; m++)
            for (int o = lpc / 2; o > 0; o >>= 1) acc[m] += __shfl_xor_sync(0xFFFFFFFFu, acc[m], o);
        if (sl == 0 && n < rows) {
#pragma unroll
            for (int m = 0; m < DC_RMAX; m++)
                if (m < R) epi(m, n, acc[m], sw[n], bb[n]);
        }
    }
}

// copy stage [R][row_bytes] into every CTA's full buffer at column offset
MNMT_DEV void dc_bcast(cg::cluster_group &cl, const uint8_t *stage, int R, int row_bytes, uint8_t *full,
                       int full_row_bytes, int col_off, int nc) {
    const int cpr = row_bytes / 16;
    const int total = nc * R * cpr;
    for (int i = threadIdx.x; i < total; i += DC_THREADS) {
        const int dst = i / (R * cpr), rem = i - dst * R * cpr;
        const int m = rem / cpr, ch = rem - m * cpr;
        int4 v = reinterpret_cast<const int4 *>(stage + (size_t)m * row_bytes)[ch];
        uint8_t *local = full + (size_t)m * full_row_bytes + col_off + ch * 16;
        *reinterpret_cast<int4 *>(cl.map_shared_rank(local, dst)) = v;
    }
}

// LayerNorm of the R rows of r (one warp per row), q8 into a (and, when
// write_back, the normalised fp32 row back into r)
MNMT_DEV void dc_layernorm(float *r, int R, int d, const float *g, const float *b, float inv, int8_t *a,
                           bool write_back, int *status) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp < R) {
        float x[16], y[16];
#pragma unroll
        for (int u = 0; u < 16; u++) {
            int i = u * 32 + lane;
            x[u] = i < d ? r[(size_t)warp * d + i] : 0.0f;
        }
        if (!warp_layernorm16(x, d, g, b, y, lane)) {
            if (lane == 0) set_status(status, MNMT_EOVERFLOW);
        }
#pragma unroll
        for (int u = 0; u < 16; u++) {
            int i = u * 32 + lane;
            if (i < d) {
                a[(size_t)warp * d + i] = q8(y[u], inv);
                if (write_back) r[(size_t)warp * d + i] = y[u];
            }
        }
    }
}

MNMT_DEV void dc_quant_rows(const float *r, int R, int d, float inv, int8_t *a) {
    for (int i = threadIdx.x; i < R * d; i += DC_THREADS) a[i] = q8(r[i], inv);
}

// attention of every (row, head) of the step, redundantly in each CTA.
// self: keys 0..t-1 from the layer's cache, key t from the step's k/v rows;
// cross: keys j < src_len of the row's sentence from the cross cache.
template <int DH>
MNMT_DEV void dc_attention(const DcParams &P, const DcLayer &Y, bool cross, const int8_t *q, int q_ld,
                           const int8_t *knew, const int8_t *vnew, int kv_ld, int t, int8_t *ctx, int *att) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int H = P.H, T = P.T, S = P.S;
    float sigma = cross ? Y.sigma2 : Y.sigma1, rho = cross ? Y.rho2 : Y.rho1;
    int *sc = att + warp * P.att_cap;
    constexpr int QC = DH / 16;
    constexpr int C = DH / 16, G = 32 / C;
    for (int item = warp; item < P.R * H; item += DC_WARPS) {
        const int m = item / H, h = item - m * H;
        int n;
        const int8_t *kb, *vb;
        int kstride;
        if (cross) {
            n = P.src_len[m];
            n = n < 1 ? 1 : (n > S ? S : n);
            kb = Y.cross_k + ((size_t)m * H + h) * S * DH;
            vb = Y.cross_v + ((size_t)m * H + h) * S * DH;
        } else {
            n = t + 1;
            kb = Y.self_k + ((size_t)m * H + h) * T * DH;
            vb = Y.self_v + ((size_t)m * H + h) * T * DH;
        }
        kstride = DH;
        int4 qv[QC];
#pragma unroll
        for (int c = 0; c < QC; c++) qv[c] = reinterpret_cast<const int4 *>(q + (size_t)m * q_ld + h * DH)[c];
        float mx = -INFINITY;
        for (int j = lane; j < n; j += 32) {
            const int4 *kr = (!cross && j == t)
                                 ? reinterpret_cast<const int4 *>(knew + (size_t)m * kv_ld + h * DH)
                                 : reinterpret_cast<const int4 *>(kb + (size_t)j * kstride);
            int acc = 0;
#pragma unroll
            for (int c = 0; c < QC; c++) acc = dot16(qv[c], kr[c], acc);
            float s = __fmul_rn(__int2float_rn(acc), sigma);
            sc[j] = __float_as_int(s);
            mx = fmaxf(mx, s);
        }
        mx = warp_max_f(mx);
        __syncwarp();
        long long Z = 0;
        for (int j = lane; j < n; j += 32) {
            int E = softmax_weight(__fadd_rn(__int_as_float(sc[j]), -mx));
            sc[j] = E;
            Z += E;
        }
        Z = warp_sum_ll(Z);
        __syncwarp();
        // context: lane = (key group g, 16-value chunk c)
        const int g = lane / C, c = lane - g * C;
        int hi[16], lo[16];
#pragma unroll
        for (int u = 0; u < 16; u++) hi[u] = lo[u] = 0;
        for (int j = g; j < n; j += G) {
            const int E = sc[j];
            const int Eh = E >> 12, El = E & 4095;
            const int4 v = (!cross && j == t) ? reinterpret_cast<const int4 *>(vnew + (size_t)m * kv_ld + h * DH)[c]
                                              : reinterpret_cast<const int4 *>(vb + (size_t)j * kstride)[c];
            const int w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
            for (int q4 = 0; q4 < 4; q4++) {
                int b0 = sb0(w4[q4]), b1 = sb1(w4[q4]), b2 = sb2(w4[q4]), b3 = sb3(w4[q4]);
                hi[q4 * 4 + 0] += Eh * b0; lo[q4 * 4 + 0] += El * b0;
                hi[q4 * 4 + 1] += Eh * b1; lo[q4 * 4 + 1] += El * b1;
                hi[q4 * 4 + 2] += Eh * b2; lo[q4 * 4 + 2] += El * b2;
                hi[q4 * 4 + 3] += Eh * b3; lo[q4 * 4 + 3] += El * b3;
            }
        }
#pragma unroll
        for (int o = C; o < 32; o <<= 1) {
#pragma unroll
            for (int u = 0; u < 16; u++) {
                hi[u] += __shfl_xor_sync(0xFFFFFFFFu, hi[u], o);
                lo[u] += __shfl_xor_sync(0xFFFFFFFFu, lo[u], o);
            }
        }
        if (g == 0) {
            const double dz = __ll2double_rn(Z);
            int8_t *out = ctx + (size_t)m * P.d + h * DH + c * 16;
#pragma unroll
            for (int u = 0; u < 16; u++) {
                long long N = (long long)hi[u] * 4096 + lo[u];
                out[u] = q8(__double2float_rn(__ddiv_rn(__ll2double_rn(N), dz)), rho);
            }
        }
        __syncwarp();
    }
}

// ---------------------------------------------------------------------------
// the step kernel
// ---------------------------------------------------------------------------
template <int DH>
__global__ void __launch_bounds__(DC_THREADS, 1) decode_cluster_kernel(const DcParams *__restrict__ Pp) {
    const DcParams &P = *Pp;
    if (*P.done) return;  // uniform for the whole cluster
    cg::cluster_group cl = cg::this_cluster();
    const int c = (int)cl.block_rank();
    const int nc = P.nc;
    const int R = P.R, d = P.d, F = P.F;
    const int t = *P.t_ptr;
    const int nsd = d / nc, ns3 = 3 * d / nc, nsf = F / nc;

    extern __shared__ __align__(16) uint8_t smem[];
    float *r_full = reinterpret_cast<float *>(smem + P.off_r);
    int8_t *a_full = reinterpret_cast<int8_t *>(smem + P.off_a);
    int8_t *qkv_full = reinterpret_cast<int8_t *>(smem + P.off_qkv);
    int8_t *ctx_full = reinterpret_cast<int8_t *>(smem + P.off_ctx);
    int8_t *q2_full = reinterpret_cast<int8_t *>(smem + P.off_q2);
    int8_t *h_full = reinterpret_cast<int8_t *>(smem + P.off_h);
    uint8_t *stage = smem + P.off_stage;
    int *att = reinterpret_cast<int *>(smem + P.off_att);
    uint8_t *ring = smem + P.off_ring;
    const int nphase = 1 + 6 * P.n_dec;

    for (int ph = 0; ph < DC_NB - 1; ph++) dc_prefetch(P, ph, c, ring, P.slot_bytes, nphase);
    int ph = 0;
    auto begin_phase = [&]() -> const uint8_t * {
        dc_wait_ring();
        __syncthreads();
        dc_prefetch(P, ph + DC_NB - 1, c, ring, P.slot_bytes, nphase);
        return ring + (size_t)(ph % DC_NB) * P.slot_bytes;
    };

    // ---- embedding slice -> r_full (all CTAs) ----
    {
        const uint8_t *slot = begin_phase();
        float *st = reinterpret_cast<float *>(stage);
        const int8_t *W = reinterpret_cast<const int8_t *>(slot);
        const float *sw = reinterpret_cast<const float *>(slot + nsd * P.E);
        const float *bb = sw + nsd;
        for (int i = threadIdx.x; i < R * nsd; i += DC_THREADS) {
            const int m = i / nsd, nl = i - m * nsd, n = c * nsd + nl;
            int id = P.tok[m];
            if (id < 0 || id >= P.V) {
                set_status(P.status, MNMT_EINVAL);
                id = 0;
            }
            const float es = P.emb_s[id];
            float x;
            if (!P.factorised) {
                float v = __fmul_rn(__fmul_rn((float)P.emb_q[(size_t)id * P.E + n], es), P.emb_scale);
                x = __fadd_rn(v, P.pe[(size_t)t * d + n]);
            } else {
                const int4 *qr = reinterpret_cast<const int4 *>(P.emb_q + (size_t)id * P.E);
                const int4 *wr = reinterpret_cast<const int4 *>(W + (size_t)nl * P.E);
                int acc = 0;
                for (int k = 0; k < P.E / 16; k++) acc = dot16(qr[k], wr[k], acc);
                float y = dequant_bias(acc, es, sw[nl], bb[nl]);
                x = __fadd_rn(__fmul_rn(y, P.emb_scale), P.pe[(size_t)t * d + n]);
            }
            st[m * nsd + nl] = x;
        }
        __syncthreads();
        dc_bcast(cl, stage, R, nsd * 4, reinterpret_cast<uint8_t *>(r_full), d * 4, c * nsd * 4, nc);
        cl.sync();
        ph++;
    }

    for (int l = 0; l < P.n_dec; l++) {
        const DcLayer &Y = P.layer[l];
        // ---- self-attention: q/k/v slice ----
        {
            if (P.pre_ln) dc_layernorm(r_full, R, d, Y.ln1_g, Y.ln1_b, 1.0f / Y.s_in1, a_full, false, P.status);
            else dc_quant_rows(r_full, R, d, 1.0f / Y.s_in1, a_full);
            const uint8_t *slot = begin_phase();
            int8_t *st = reinterpret_cast<int8_t *>(stage);
            const int n0 = c * ns3;
            dc_gemv(slot, ns3, d, a_full, d, R, [&](int m, int nl, int acc, float sw, float bias) {
                const int n = n0 + nl;
                int8_t v = q8(dequant_bias(acc, Y.s_in1, sw, bias), Y.inv_qkv[n]);
                st[m * ns3 + nl] = v;
                if (n >= d) {  // K / V of position t into the layer's cache
                    const int seg = n >= 2 * d;
                    const int cc = n - (seg ? 2 * d : d);
                    const int h = cc / DH, i = cc - h * DH;
                    int8_t *dst = seg ? Y.self_v : Y.self_k;
                    dst[(((size_t)m * P.H + h) * P.T + t) * DH + i] = v;
                }
            });
            __syncthreads();
            dc_bcast(cl, stage, R, ns3, reinterpret_cast<uint8_t *>(qkv_full), 3 * d, n0, nc);
            cl.sync();
            ph++;
        }
        // ---- attention (all heads) + W_o slice + gamma-residual ----
        {
            dc_attention<DH>(P, Y, false, qkv_full, 3 * d, qkv_full + d, qkv_full + 2 * d, 3 * d, t, ctx_full, att);
            const uint8_t *slot = begin_phase();  // includes the barrier that publishes ctx_full
            float *st = reinterpret_cast<float *>(stage);
            const int n0 = c * nsd;
            dc_gemv(slot, nsd, d, ctx_full, d, R, [&](int m, int nl, int acc, float sw, float bias) {
                float y = dequant_bias(acc, Y.s_ctx1, sw, bias);
                st[m * nsd + nl] = __fadd_rn(__fmul_rn(Y.gamma1, r_full[(size_t)m * d + n0 + nl]), y);
            });
            __syncthreads();
            dc_bcast(cl, stage, R, nsd * 4, reinterpret_cast<uint8_t *>(r_full), d * 4, n0 * 4, nc);
            cl.sync();
            ph++;
        }
        // ---- cross-attention: q slice ----
        {
            if (P.pre_ln) {
                dc_layernorm(r_full, R, d, Y.ln2_g, Y.ln2_b, 1.0f / Y.s_in2, a_full, false, P.status);
            } else {
                dc_layernorm(r_full, R, d, Y.ln1_g, Y.ln1_b, 1.0f / Y.s_in2, a_full, true, P.status);
            }
            const uint8_t *slot = begin_phase();
            int8_t *st = reinterpret_cast<int8_t *>(stage);
            const int n0 = c * nsd;
            dc_gemv(slot, nsd, d, a_full, d, R, [&](int m, int nl, int acc, float sw, float bias) {
                st[m * nsd + nl] = q8(dequant_bias(acc, Y.s_in2, sw, bias), Y.inv_q2[n0 + nl]);
            });
            __syncthreads();
            dc_bcast(cl, stage, R, nsd, reinterpret_cast<uint8_t *>(q2_full), d, n0, nc);
            cl.sync();
            ph++;
        }
        // ---- cross-attention (all heads) + W_o slice + gamma-residual ----
        {
            dc_attention<DH>(P, Y, true, q2_full, d, nullptr, nullptr, 0, t, ctx_full, att);
            const uint8_t *slot = begin_phase();
            float *st = reinterpret_cast<float *>(stage);
            const int n0 = c * nsd;
            dc_gemv(slot, nsd, d, ctx_full, d, R, [&](int m, int nl, int acc, float sw, float bias) {
                float y = dequant_bias(acc, Y.s_ctx2, sw, bias);
                st[m * nsd + nl] = __fadd_rn(__fmul_rn(Y.gamma2, r_full[(size_t)m * d + n0 + nl]), y);
            });
            __syncthreads();
            dc_bcast(cl, stage, R, nsd * 4, reinterpret_cast<uint8_t *>(r_full), d * 4, n0 * 4, nc);
            cl.sync();
            ph++;
        }
        // ---- FFN1 slice (ReLU + q8) ----
        {
            if (P.pre_ln) {
                dc_layernorm(r_full, R, d, Y.ln3_g, Y.ln3_b, 1.0f / Y.s_in3, a_full, false, P.status);
            } else {
                dc_layernorm(r_full, R, d, Y.ln2_g, Y.ln2_b, 1.0f / Y.s_in3, a_full, true, P.status);
            }
            const uint8_t *slot = begin_phase();
            int8_t *st = reinterpret_cast<int8_t *>(stage);
            const int n0 = c * nsf;
            dc_gemv(slot, nsf, d, a_full, d, R, [&](int m, int nl, int acc, float sw, float bias) {
                float y = dequant_bias(acc, Y.s_in3, sw, bias);
                st[m * nsf + nl] = q8(y > 0.0f ? y : 0.0f, Y.inv_h[n0 + nl]);
            });
            __syncthreads();
            dc_bcast(cl, stage, R, nsf, reinterpret_cast<uint8_t *>(h_full), F, n0, nc);
            cl.sync();
            ph++;
        }
        // ---- FFN2 slice + gamma-residual ----
        {
            const uint8_t *slot = begin_phase();
            float *st = reinterpret_cast<float *>(stage);
            const int n0 = c * nsd;
            dc_gemv(slot, nsd, F, h_full, F, R, [&](int m, int nl, int acc, float sw, float bias) {
                float y = dequant_bias(acc, Y.s_h, sw, bias);
                st[m * nsd + nl] = __fadd_rn(__fmul_rn(Y.gamma3, r_full[(size_t)m * d + n0 + nl]), y);
            });
            __syncthreads();
            dc_bcast(cl, stage, R, nsd * 4, reinterpret_cast<uint8_t *>(r_full), d * 4, n0 * 4, nc);
            cl.sync();
            ph++;
        }
        if (!P.pre_ln) {
            // post-LN: the FFN's LayerNorm normalises the stream in place; the
            // next sublayer input is quantised from it
            const bool last = l + 1 == P.n_dec;
            float inv = last ? 1.0f / P.s_dout : 1.0f / P.layer[l + 1].s_in1;
            dc_layernorm(r_full, R, d, Y.ln3_g, Y.ln3_b, inv, a_full, true, P.status);
            __syncthreads();
        }
    }
    // ---- final LayerNorm + quantisation -> vocabulary input ----
    if (P.pre_ln) dc_layernorm(r_full, R, d, P.fin_g, P.fin_b, 1.0f / P.s_dout, a_full, false, P.status);
    __syncthreads();
    if (c == 0) {
        for (int i = threadIdx.x; i < R * d; i += DC_THREADS) {
            P.act_out[i] = a_full[i];
            if (P.resid_out) P.resid_out[i] = r_full[i];
        }
    }
    // every CTA must still hold its shared memory while others may write to it
    cl.sync();
}

// ---------------------------------------------------------------------------
// vocabulary projection + greedy argmax + greedy update (last block)
// ---------------------------------------------------------------------------
template <int MT>
__global__ void __launch_bounds__(256) vocab_greedy_kernel(const int8_t *__restrict__ A, const int8_t *__restrict__ W,
                                                           const float *__restrict__ s_w,
                                                           const float *__restrict__ bias, float s_x, int M, int N,
                                                           int K, unsigned long long *keys, int *ticket,
                                                           GreedyArgs g) {
    if (*g.done) return;
    extern __shared__ int4 vsm[];  // [MT][K/16]
    const int kc = K >> 4;
    for (int i = threadIdx.x; i < MT * kc; i += 256) {
        int m = i / kc, c = i - m * kc;
        vsm[i] = m < M ? reinterpret_cast<const int4 *>(A + (size_t)m * K)[c] : make_int4(0, 0, 0, 0);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int lpc = kc >= 32 ? 32 : kc;
    const int gpw = 32 / lpc;
    const int grp = lane / lpc, sl = lane % lpc;
    constexpr int U = 4;
    const int cpb = 8 * gpw * U;
    unsigned long long best[MT];
#pragma unroll
    for (int m = 0; m < MT; m++) best[m] = 0ull;
    for (int base = blockIdx.x * cpb; base < N; base += gridDim.x * cpb) {
        int acc[U][MT];
#pragma unroll
        for (int u = 0; u < U; u++)
#pragma unroll
            for (int m = 0; m < MT; m++) acc[u][m] = 0;
        for (int c0 = 0; c0 < kc; c0 += lpc) {
            const int c = c0 + sl;
            int4 w[U];
#pragma unroll
            for (int u = 0; u < U; u++) {
                int n = base + (u * 8 + warp) * gpw + grp;
                w[u] = (n < N && c < kc) ? __ldg(reinterpret_cast<const int4 *>(W + (size_t)n * K) + c)
                                         : make_int4(0, 0, 0, 0);
            }
            if (c < kc) {
#pragma unroll
                for (int m = 0; m < MT; m++) {
                    int4 a = vsm[m * kc + c];
#pragma unroll
                    for (int u = 0; u < U; u++) acc[u][m] = dot16(a, w[u], acc[u][m]);
                }
            }
        }
#pragma unroll
        for (int u = 0; u < U; u++) {
#pragma unroll
            for (int m = 0; m < MT; m++)
                for (int o = lpc / 2; o > 0; o >>= 1) acc[u][m] += __shfl_xor_sync(0xFFFFFFFFu, acc[u][m], o);
            const int n = base + (u * 8 + warp) * gpw + grp;
            if (sl == 0 && n < N) {
#pragma unroll
                for (int m = 0; m < MT; m++) {
                    if (m < M) {
                        unsigned long long k = pack_key(dequant_bias(acc[u][m], s_x, s_w[n], bias[n]), (uint32_t)n);
                        best[m] = k > best[m] ? k : best[m];
                    }
                }
            }
        }
    }
    __shared__ unsigned long long red[8][MT];
    __shared__ int s_last;
#pragma unroll
    for (int m = 0; m < MT; m++) {
        unsigned long long v = warp_max_u64(best[m]);
        if (lane == 0) red[warp][m] = v;
    }
    __syncthreads();
    if (threadIdx.x < MT && (int)threadIdx.x < M) {
        unsigned long long v = 0;
        for (int w = 0; w < 8; w++) v = red[w][threadIdx.x] > v ? red[w][threadIdx.x] : v;
        atomicMax(keys + threadIdx.x, v);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        s_last = atomicAdd(ticket, 1) == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (!s_last) return;
    // last block: greedy update of every row (keys read and cleared atomically)
    __threadfence();
    const int t = *g.t_ptr;
    int fin_all = 1;
    for (int r = threadIdx.x; r < g.R; r += 256) {
        unsigned long long k = atomicExch(keys + r, 0ull);
        int y = (int)key_index(k);
        int f = g.fin[r];
        int out = f ? g.pad : y;
        g.hist[(size_t)t * g.R + r] = out;
        g.tok[r] = out;
        if (!f && y == g.eos) f = 1;
        g.fin[r] = f;
        fin_all &= f;
    }
    int all = __syncthreads_and(fin_all);
    if (threadIdx.x == 0) {
        if (all || t + 1 >= *g.tmax_ptr) *g.done = 1;
        *g.t_ptr = t + 1;
        *ticket = 0;
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
// CTAs per cluster: one 16-column slice of d per CTA, at most 16 CTAs
int dc_cluster_size(int d) {
    int nc = d / 16;
    if (nc > 16) nc = 16;
    return nc >= 2 ? nc : 0;
}

size_t dc_layout(DcParams &P) {
    // shared-memory carve-up (16-byte aligned pieces)
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t at = off;
        off += (bytes + 15) & ~(size_t)15;
        return (int)at;
    };
    const int R = P.R, d = P.d, F = P.F, nc = P.nc;
    P.off_r = take((size_t)R * d * 4);
    P.off_a = take((size_t)R * d);
    P.off_qkv = take((size_t)R * 3 * d);
    P.off_ctx = take((size_t)R * d);
    P.off_q2 = take((size_t)R * d);
    P.off_h = take((size_t)R * F);
    int stage_bytes = R * (d / nc) * 4;
    if (R * 3 * d / nc > stage_bytes) stage_bytes = R * 3 * d / nc;
    if (R * F / nc > stage_bytes) stage_bytes = R * F / nc;
    P.off_stage = take(stage_bytes);
    P.att_cap = P.T > P.S ? P.T : P.S;
    P.off_att = take((size_t)DC_WARPS * P.att_cap * 4);
    // largest weight slice of any phase (rows * K + 8 * rows)
    int slot = 0;
    auto upd = [&](int rows, int K) {
        int b = rows * K + 8 * rows;
        if (b > slot) slot = b;
    };
    if (P.factorised) upd(d / nc, P.E);
    upd(3 * d / nc, d);
    upd(d / nc, d);
    upd(F / nc, d);
    upd(d / nc, F);
    P.slot_bytes = (slot + 15) & ~15;
    P.off_ring = take((size_t)DC_NB * P.slot_bytes);
    return off;
}

cudaError_t decode_cluster_init() {
    const int max_smem = 227 * 1024;
    cudaError_t err = cudaSuccess;
    auto setk = [&](const void *k) {
        if (err == cudaSuccess) err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem);
        if (err == cudaSuccess) err = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    };
    setk((const void *)decode_cluster_kernel<32>);
    setk((const void *)decode_cluster_kernel<64>);
    setk((const void *)decode_cluster_kernel<128>);
    return err;
}

// can one cluster of nc CTAs with smem bytes each be resident?
bool decode_cluster_fits(int dh, int nc, size_t smem) {
    if (smem > 227 * 1024) return false;
    const void *k = dh == 32 ? (const void *)decode_cluster_kernel<32>
                             : (dh == 64 ? (const void *)decode_cluster_kernel<64> : (const void *)decode_cluster_kernel<128>);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(nc);
    cfg.blockDim = dim3(DC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = nc;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, k, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return clusters >= 1;
}

cudaError_t launch_decode_cluster(const DcParams *dP, int dh, int nc, size_t smem, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(nc);
    cfg.blockDim = dim3(DC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = nc;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    switch (dh) {
        case 32: return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<32>, dP);
        case 64: return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<64>, dP);
        case 128: return cudaLaunchKernelEx(&cfg, decode_cluster_kernel<128>, dP);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_vocab_greedy(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                                int M, int N, int K, unsigned long long *keys, int *ticket, const GreedyArgs &g,
                                cudaStream_t st) {
    const int kc = K / 16;
    const int lpc = kc >= 32 ? 32 : kc;
    const int cpb = 8 * (32 / lpc) * 4;
    int blocks = (N + cpb - 1) / cpb;
    if (blocks > 2 * 152) blocks = 2 * 152;
    size_t smem;
    switch (M) {
        case 1: smem = (size_t)1 * kc * 16; vocab_greedy_kernel<1><<<blocks, 256, smem, st>>>(A, W, s_w, bias, s_x, M, N, K, keys, ticket, g); break;
        case 2: smem = (size_t)2 * kc * 16; vocab_greedy_kernel<2><<<blocks, 256, smem, st>>>(A, W, s_w, bias, s_x, M, N, K, keys, ticket, g); break;
        default: smem = (size_t)4 * kc * 16; vocab_greedy_kernel<4><<<blocks, 256, smem, st>>>(A, W, s_w, bias, s_x, M, N, K, keys, ticket, g); break;
    }
    return cudaGetLastError();
}

}  // namespace mnmt
