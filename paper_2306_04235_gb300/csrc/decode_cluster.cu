// decode_cluster.cu -- one decoder step of a small greedy batch (R <= 4 rows)
// on a single thread-block cluster, then the vocabulary projection fused with
// the greedy update.
//
// A batch-1 decode step is a chain of dependent matrix-vector products and two
// attentions per decoder layer (App. A), each only 16-260 KB of weights: the
// step is bound by latency, not bandwidth.  Instead of one kernel per
// operation, one cluster of NC CTAs (up to 16 SMs) runs the whole decoder:
//   * every CTA holds the full activation vectors of the step in shared memory
//     (residual stream fp32 [R][d], LN output, q/k/v, context, FFN hidden);
//   * a linear layer is split by output columns: CTA c computes its column
//     slice from its weight slice and stores it into the shared memory of
//     every CTA of the cluster (distributed shared memory) with st.async,
//     whose bytes complete on the receiver's exchange mbarrier: each CTA waits
//     only until its own copy of the vector is whole;
//   * LayerNorm and attention (all heads of the step's rows) are computed
//     redundantly by every CTA, which removes two exchanges per attention;
//   * weight slices stream from L2/HBM into a 3-slot shared-memory ring by 1-D
//     bulk copies (an mbarrier per slot), three phases ahead of use; the keys
//     and values the step attends to are staged into shared memory at kernel
//     start when they fit.
// The step is one compact phase loop with one exchange per phase, a single
// cluster barrier (every CTA's mbarriers are set before the first exchange),
// no global synchronisation and only bounded waits.
// The arithmetic is exactly that of the other kernels (Fig. 5 quantisation
// points, fixed-point LayerNorm and softmax), so the step is bit-identical to
// the multi-kernel path.
#include <cooperative_groups.h>

#include <cstdlib>

#include "common.cuh"
#include "internal.h"
#include "mbarrier.cuh"

namespace cg = cooperative_groups;

// Phase timing for the debug build (compiled with -DMNMT_DC_STAMPS only): CTA 0,
// thread 0 records %globaltimer at the phase boundaries of decode step
// DC_STAMP_STEP, and the vocabulary kernel of the step before records its
// start, the end of its wait and its end.  Slots: 0 kernel start, 1 / 2
// around the grid wait, 3 phase loop start, 4 + 4 ph .. 7 + 4 ph the phase's
// ring wait / input prep / slice GEMV / exchange ends, 100
// / 101 / 102 final LayerNorm start / end / kernel end, 110 .. 113 vocabulary
// kernel (block 0 start, before / after its wait, end).
constexpr int DC_STAMP_STEP = 20;
#ifdef MNMT_DC_STAMPS
__device__ unsigned long long g_dc_ns[128];
extern "C" int mnmt_dc_stamps(unsigned long long *out) {
    return (int)cudaMemcpyFromSymbol(out, g_dc_ns, sizeof(g_dc_ns));
}
__device__ __forceinline__ unsigned long long dc_gtime() {
    unsigned long long x;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(x));
    return x;
}
#define DC_STAMP(cond, id) \
    do { if ((cond) && (id) < 128) g_dc_ns[id] = dc_gtime(); } while (0)
#else
#define DC_STAMP(cond, id) \
    do { } while (0)
#endif

namespace mnmt {

constexpr int DC_THREADS = 256;
constexpr int DC_WARPS = DC_THREADS / 32;
constexpr int DC_NB = 3;  // weight ring slots

MNMT_DEV uint32_t dc_smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
MNMT_DEV void dc_cp16(void *dst_smem, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dc_smem_u32(dst_smem)), "l"(src));
}
MNMT_DEV void dc_commit() { asm volatile("cp.async.commit_group;\n" ::); }

// programmatic dependent launch: wait for the preceding kernel of the stream
// (and the memory it wrote); allow the following kernel to launch
MNMT_DEV void dc_grid_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
MNMT_DEV void dc_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory"); }

// out-of-line copies of the exact roundings (one copy of the code each)
__device__ __noinline__ float dc_rn32_div(long long n, long long z) { return rn32_div(n, z); }
__device__ __noinline__ float dc_rn32_pow2_full(long long s, int e) { return rn32_pow2(s, e); }
// the common case inline (one conversion, exact while the result is a normal
// float), the rest out of line
MNMT_DEV float dc_rn32_pow2(long long s, int e) {
    if (s != 0) {
        const uint32_t fb = __float_as_uint(__ll2float_rn(s));
        const int fe = (int)((fb >> 23) & 0xFFu) + e;
        if (fe >= 1 && fe <= 254) return __uint_as_float(fb + ((uint32_t)e << 23));
    }
    return dc_rn32_pow2_full(s, e);
}

// nearest float to s 2^e / (dodd 2^kd): the power-of-two case inline, an odd
// factor (widths such as 384 = 3 * 128) out of line.  The odd case is
// rn32_scaled_div's method (an integer quotient of at least 50 significant
// bits plus a sticky bit) with its 64-bit division replaced by a multiply-high
// by zm = floor(2^64 / dodd) (host-computed): for num < 2^63 the estimate is
// the quotient or one less, which the remainder corrects.
__device__ __noinline__ float dc_rn32_scaled_div(long long S, int e, int kd, unsigned z, unsigned long long zm) {
    if (S == 0) return 0.0f;
    const unsigned long long a = S < 0 ? 0ull - (unsigned long long)S : (unsigned long long)S;
    const int nb = 64 - __clzll(a);
    const int t = nb < 62 ? 62 - nb : 0;
    const unsigned long long num = a << t;
    unsigned long long q = __umul64hi(num, zm), r = num - q * z;
    if (r >= z) {
        q++;
        r -= z;
    }
    const float f = rn32_pow2((long long)(2ull * q + (r != 0ull ? 1ull : 0ull)), e - kd - t - 1);
    return S < 0 ? -f : f;
}
MNMT_DEV float dc_rn32_scaled(long long s, int e, int kd, int dodd, unsigned long long zm) {
    if (dodd == 1) return dc_rn32_pow2(s, e - kd);
    return dc_rn32_scaled_div(s, e, kd, (unsigned)dodd, zm);
}

// signed bytes of a 32-bit word
MNMT_DEV int sb0(int x) { return (x << 24) >> 24; }
MNMT_DEV int sb1(int x) { return (x << 16) >> 24; }
MNMT_DEV int sb2(int x) { return (x << 8) >> 24; }
MNMT_DEV int sb3(int x) { return x >> 24; }

// async copy of `bytes` (a multiple of 16) from global to shared memory
MNMT_DEV void dc_copy(void *dst, const void *src, int bytes) {
    for (int i = threadIdx.x; i < bytes / 16; i += DC_THREADS)
        dc_cp16(static_cast<uint8_t *>(dst) + i * 16, static_cast<const uint8_t *>(src) + i * 16);
}

// Index arithmetic of the step avoids integer division by run-time values
// (a multi-instruction sequence on the critical path of every phase):
// quotients come from multiply-high by a host-computed ceil(2^32 / d) (exact
// for i, d < 2^16; mg == 0 stands for d == 1), from shifts by powers of two,
// or from a few compares when the quotient is a row index below DC_RMAX.
MNMT_DEV int dc_udiv(int i, uint32_t mg) { return mg ? (int)__umulhi((uint32_t)i, mg) : i; }
template <int RM = DC_RMAX>
MNMT_DEV int dc_row_of(int i, int d, int R) {  // i / d for i < R d, R <= RM
    int r = 0;
#pragma unroll
    for (int k = 1; k < RM; k++) r += (k < R && i >= k * d) ? 1 : 0;
    return r;
}

// ring slot layout: W rows (rows * K bytes), then s[rows], b[rows], inv[rows] (fp32)
// Phase ph's slice goes to slot ph % DC_NB as up to five 1-D bulk copies (the
// copy engine moves them: no per-thread copy instructions queue ahead of the
// phase's own shared-memory work) that complete on the slot's mbarrier; the
// barrier gets one arrival per phase, copies or not, so phase ph always waits
// for parity (ph / DC_NB) & 1.  Issued by thread `who`; slices, offsets and
// sizes are whole 16-byte chunks (the cluster size is chosen so).
MNMT_DEV void dc_prefetch(const DcParams &P, int ph, int c, uint8_t *ring, uint32_t bars, int who = 0) {
    if ((int)threadIdx.x != who || ph >= 1 + 6 * P.n_dec) return;
    const DcPhase &f = P.phase[ph];
    const uint32_t bar = bars + 8u * (uint32_t)(ph % DC_NB);
    if (!f.rows) {
        mbar_arrive(bar);
        return;
    }
    const uint32_t dst = dc_smem_u32(ring + (size_t)(ph % DC_NB) * P.slot_bytes);
    const uint32_t wb = (uint32_t)(f.rows * (f.bits == 4 ? f.K / 2 : f.K)), vb = (uint32_t)f.rows * 4u;
    const uint32_t total = wb + vb * (2u + (f.inv ? 1u : 0u) + (f.m ? 1u : 0u));
    // the slot's previous contents were read by ordinary loads before the
    // block barrier that precedes this call; order them before the copy's writes
    asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
    mbar_expect_tx(bar, total);
    bulk_load(dst, f.w + (size_t)c * wb, wb, bar);
    bulk_load(dst + wb, f.s + c * f.rows, vb, bar);
    bulk_load(dst + wb + vb, f.b + c * f.rows, vb, bar);
    if (f.inv) bulk_load(dst + wb + 2 * vb, f.inv + c * f.rows, vb, bar);
    if (f.m) bulk_load(dst + wb + 3 * vb, f.m + c * f.rows, vb, bar);
}

// wait for phase ph's slice; a wait that gives up records MNMT_ETIMEOUT
MNMT_DEV void dc_wait_slice(const DcParams &P, int ph, uint32_t bars) {
    if (!mbar_wait(bars + 8u * (uint32_t)(ph % DC_NB), (uint32_t)(ph / DC_NB) & 1u)) set_status(P.status, MNMT_ETIMEOUT);
}

// Exchange between the CTAs of the cluster.  A phase's slice goes to every
// CTA (itself included) as st.async stores, each completing its bytes on the
// receiver's exchange mbarrier for that phase (two, used by alternate
// phases); a CTA waits on its own barrier until the whole vector has arrived
// instead of a cluster-wide barrier.  No store can overwrite data a receiver
// still reads: a CTA sends phase ph + 1 only after receiving phase ph from
// every CTA, i.e. after every CTA finished the GEMV of phase ph (and with it
// every read of the buffers that phase ph + 1 overwrites).
MNMT_DEV uint32_t dc_mapa(uint32_t local, int rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(local), "r"(rank));
    return r;
}
MNMT_DEV void dc_st_async4(uint32_t remote, int4 v, uint32_t remote_bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];\n" ::"r"(
                     remote),
                 "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(remote_bar)
                 : "memory");
}
MNMT_DEV void dc_st_async2(uint32_t remote, unsigned x, unsigned y, uint32_t remote_bar) {
    asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.b32 [%0], {%1, %2}, [%3];\n" ::"r"(remote),
                 "r"(x), "r"(y), "r"(remote_bar)
                 : "memory");
}

// copy stage [R][row_bytes] into every CTA's full buffer at column offset,
// completing on each receiver's exchange barrier xbar (local address)
__device__ __noinline__ void dc_bcast(const DcPhase &f, const uint8_t *stage, int R, int row_bytes, uint8_t *full,
                                      int full_row_bytes, int col_off, int nc, uint32_t xbar) {
    const int cpr = f.cpr;  // row_bytes / 16
    const int total = nc * R * cpr;
    for (int i = threadIdx.x; i < total; i += DC_THREADS) {
        const int dst = dc_udiv(i, f.mg_rc), rem = i - dst * R * cpr;
        const int m = dc_udiv(rem, f.mg_c), ch = rem - m * cpr;
        const int4 v = reinterpret_cast<const int4 *>(stage + (size_t)m * row_bytes)[ch];
        const uint32_t local = dc_smem_u32(full + (size_t)m * full_row_bytes + col_off + ch * 16);
        dc_st_async4(dc_mapa(local, dst), v, dc_mapa(xbar, dst));
    }
}

// Block-wide LayerNorm of the R rows of r (same arithmetic as
// warp_layernorm): element e of the flattened [R][d] array belongs to thread
// e % 256; each warp's 32 elements lie in one row, so the exact int64 sums are
// warp reductions (redux.sync) whose partials meet in shared memory, d/32
// partials per row.  The row's largest and smallest values arrive with the
// residual itself (mm [R][nc] ordered-bit pairs, one per CTA slice, written
// by the epilogue that produced r), which gives both grids without a pass of
// their own: max|r| = max(|max r|, |min r|) and, fl(x - mu) being monotone in
// x, max|fl(r - mu)| = max(|fl(max r - mu)|, |fl(min r - mu)|).  Three passes:
// exact sum of r, exact sum of (r - mu)^2, normalise.  q8(LN(r), inv) goes to
// a; with write_back the normalised row also replaces r.  Ends with a block
// barrier.
MNMT_DEV long long dc_row_sum(const long long *part, int row, int spr) {
    long long s = 0;
#pragma unroll
    for (int k = 0; k < 16; k++)  // spr = d / 32 <= 16: every load issued at once
        if (k < spr) s += part[row * spr + k];
    return s;
}

// the row's max and min from the nc slice records (one warp, all lanes)
MNMT_DEV void dc_row_extremes(const unsigned *mm, int row, int nc, float &hi, float &lo) {
    const int lane = threadIdx.x & 31;
    const unsigned kh = lane < nc ? mm[(row * nc + lane) * 2 + 0] : 0u;
    const unsigned kl = lane < nc ? mm[(row * nc + lane) * 2 + 1] : 0xFFFFFFFFu;
    hi = from_ordered_bits(__reduce_max_sync(0xFFFFFFFFu, kh));
    lo = from_ordered_bits(__reduce_min_sync(0xFFFFFFFFu, kl));
}

// RM: the kernel's row bound; TWO: 0 / 1 when the row width is known to be at
// most / more than 256 (else -1: decided at run time)
template <int RM, int TWO>
__device__ __noinline__ void dc_layernorm(float *r, int R, int d, const float *g, const float *b, float inv,
                                          int8_t *a, int write_back, int *status, const unsigned *mm, int nc,
                                          long long *part_l, int kd, int dodd, unsigned long long zm) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    // a warp takes chunks of cw elements of one row: 32 (one per lane) up to
    // 256 elements, else 64 (two per lane, independent chains), so rows of up
    // to 512 elements still take one round per pass
    const int n = R * d, two = TWO >= 0 ? TWO : (n > DC_THREADS ? 1 : 0), cs = 5 + two, cw = 32 << two;
    const int spr = d >> cs;  // partial slots (chunks) per row
    // pass 1: exact sum of x on the grid of max |x|
#pragma unroll 1
    for (int e0 = warp * cw; e0 < n; e0 += DC_WARPS * cw) {
        float hi, lo;
        dc_row_extremes(mm, dc_row_of<RM>(e0, d, R), nc, hi, lo);
        const float am = fmaxf(fabsf(hi), fabsf(lo));
        if (!(am < 0x1p32f) && lane == 0) set_status(status, MNMT_EOVERFLOW);
        const int sh = 52 - exp_bound(am);
        long long v = fx_scale(r[e0 + lane], sh);
        if (two) v += fx_scale(r[e0 + 32 + lane], sh);
        const long long s = warp_sum_exact(v);
        if (lane == 0) part_l[e0 >> cs] = s;
    }
    __syncthreads();
    // pass 2: exact sum of c^2 = fl(x - mean)^2 on the grid of max |c|
#pragma unroll 1
    for (int e0 = warp * cw; e0 < n; e0 += DC_WARPS * cw) {
        const int row = dc_row_of<RM>(e0, d, R);
        float hi, lo;
        dc_row_extremes(mm, row, nc, hi, lo);
        const int ea = exp_bound(fmaxf(fabsf(hi), fabsf(lo)));
        const float mu = dc_rn32_scaled(dc_row_sum(part_l, row, spr), ea - 52, kd, dodd, zm);
        const int eb = exp_bound(fmaxf(fabsf(__fsub_rn(hi, mu)), fabsf(__fsub_rn(lo, mu))));
        const int sh = 52 - 2 * eb;
        const float cv = __fsub_rn(r[e0 + lane], mu);
        long long v = fx_scale(__fmul_rn(cv, cv), sh);
        if (two) {
            const float cw2 = __fsub_rn(r[e0 + 32 + lane], mu);
            v += fx_scale(__fmul_rn(cw2, cw2), sh);
        }
        const long long s = warp_sum_exact(v);
        if (lane == 0) part_l[64 + (e0 >> cs)] = s;
        if (lane == 0 && e0 == row * d) {
            reinterpret_cast<float *>(part_l + 128)[2 * row] = mu;  // per row: mu, 2^eb grid
            reinterpret_cast<int *>(part_l + 128)[2 * row + 1] = eb;
        }
    }
    __syncthreads();
    // pass 3: normalise, scale, shift, quantise
#pragma unroll 1
    for (int e0 = warp * cw; e0 < n; e0 += DC_WARPS * cw) {
        const int row = dc_row_of<RM>(e0, d, R), e = e0 + lane, i = e - row * d;
        const float mu = reinterpret_cast<const float *>(part_l + 128)[2 * row];
        const int eb = reinterpret_cast<const int *>(part_l + 128)[2 * row + 1];
        const float var = dc_rn32_scaled(dc_row_sum(part_l + 64, row, spr), 2 * eb - 52, kd, dodd, zm);
        const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, 1e-5f)));
        const float y = __fadd_rn(__fmul_rn(__fmul_rn(__fsub_rn(r[e], mu), rstd), g[i]), b[i]);
        float y2 = 0.0f;
        if (two) y2 = __fadd_rn(__fmul_rn(__fmul_rn(__fsub_rn(r[e + 32], mu), rstd), g[i + 32]), b[i + 32]);
        a[e] = q8(y, inv);
        if (write_back) r[e] = y;
        if (two) {
            a[e + 32] = q8(y2, inv);
            if (write_back) r[e + 32] = y2;
        }
    }
    __syncthreads();
}

// Attention of every (row, head) of the step, redundantly in each CTA.  The 8
// warps split the keys of an item (row, head) into ranges: scores and the
// partial maximum per range, then weights, partial Z and partial context sums
// per range; the partials are exact integers, so they combine in any order.
// self: keys 0..t-1 from the layer's cache (staged or global), key t from the
// step's own k/v rows; cross: keys j < src_len of the row's sentence.
// LW >= 0: 2^LW warps per item fixed at compile time (LW = 0: each warp holds
// a whole item -- no cross-warp maximum, and it writes its context itself)
template <int DH, int RM, int LW>
__device__ __forceinline__ void dc_attention(const DcParams &P, int l, int cross, const int8_t *q, int q_ld,
                                          const int8_t *knew, const int8_t *vnew, int kv_ld, int t, int8_t *ctx,
                                          int *att, float *red_f, long long *pz, long long *pn,
                                          const uint8_t *smem, const int *src_len_s) {
    const DcLayer &Y = P.layer[l];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int H = P.H, T = P.T, S = P.S, R = P.R;
    const float sigma = cross ? Y.sigma2 : Y.sigma1, rho = cross ? Y.rho2 : Y.rho1;
    const int items = R * H;
    const int lw = LW >= 0 ? LW : P.att_lw;                 // 2^lw warps per item
    const int ip = LW >= 0 ? (DC_WARPS >> LW) : P.att_ip;  // items per round
    const int wpi = 1 << lw;
    constexpr int QC = DH / 16;
    for (int base = 0; base < items; base += ip) {
        const int it = base + (warp >> lw), part = warp & (wpi - 1);
        const bool live = it < items;
        const int m = live ? dc_row_of<RM>(it, H, R) : 0, h = live ? it - m * H : 0;
        int n;
        const int8_t *kb, *vb;
        if (cross) {
            n = src_len_s[m];
            n = n < 1 ? 1 : (n > S ? S : n);
            if (P.kv_staged) {
                const int8_t *cb = reinterpret_cast<const int8_t *>(smem + P.off_kvc);
                kb = cb + (((size_t)(l * 2 + 0) * R + m) * H + h) * S * DH;
                vb = cb + (((size_t)(l * 2 + 1) * R + m) * H + h) * S * DH;
            } else {
                kb = Y.cross_k + ((size_t)m * H + h) * S * DH;
                vb = Y.cross_v + ((size_t)m * H + h) * S * DH;
            }
        } else {
            n = t + 1;
            if (P.kv_staged) {
                const int8_t *sbp = reinterpret_cast<const int8_t *>(smem + P.off_kvs);
                kb = sbp + (((size_t)(l * 2 + 0) * R + m) * H + h) * T * DH;
                vb = sbp + (((size_t)(l * 2 + 1) * R + m) * H + h) * T * DH;
            } else {
                kb = Y.self_k + ((size_t)m * H + h) * T * DH;
                vb = Y.self_v + ((size_t)m * H + h) * T * DH;
            }
        }
        const int per = (n + wpi - 1) >> lw;
        const int j0 = part * per, j1 = min(n, j0 + per);
        int *sc = att + (warp >> lw) * P.att_cap;
        float mx = -INFINITY;
        if (live) {
            int4 qv[QC];
#pragma unroll
            for (int c = 0; c < QC; c++) qv[c] = reinterpret_cast<const int4 *>(q + (size_t)m * q_ld + h * DH)[c];
            for (int j = j0 + lane; j < j1; j += 32) {
                const int4 *kr = (!cross && j == t)
                                     ? reinterpret_cast<const int4 *>(knew + (size_t)m * kv_ld + h * DH)
                                     : reinterpret_cast<const int4 *>(kb + (size_t)j * DH);
                int acc = 0;
#pragma unroll
                for (int c = 0; c < QC; c++) acc = dot16(qv[c], kr[c], acc);
                const float sv = __fmul_rn(__int2float_rn(acc), sigma);
                sc[j] = __float_as_int(sv);
                mx = fmaxf(mx, sv);
            }
        }
        mx = warp_max_f(mx);
        if (LW != 0) {  // the item's maximum over its warps
            if (lane == 0) red_f[warp] = mx;
            __syncthreads();
            mx = -INFINITY;
            for (int w = 0; w < wpi; w++) mx = fmaxf(mx, red_f[(warp >> lw) * wpi + w]);
        }
        int zl = 0;
        if (live)
            for (int j = j0 + lane; j < j1; j += 32) {
                const int E = softmax_weight(__fadd_rn(__int_as_float(sc[j]), -mx));
                sc[j] = E;
                zl += E;  // at most 32 keys per lane: < 2^30
            }
        const long long z = warp_sum_exact(zl);
        __syncwarp();
        // context: the warp's keys KPI at a time, LPK lanes per key and 4
        // consecutive elements of the head per lane; the key groups' exact
        // integer partial sums meet by shuffles
        constexpr int LPK = DH / 4, KPI = 32 / LPK;
        const int kg = lane / LPK, el = (lane % LPK) * 4;
        int hi[4] = {0, 0, 0, 0}, lo[4] = {0, 0, 0, 0};
        if (live) {
#pragma unroll 2
            for (int j = j0 + kg; j < j1; j += KPI) {
                const int E = sc[j];
                const int Eh = E >> 12, El = E & 4095;
                const int8_t *vr = (!cross && j == t) ? vnew + (size_t)m * kv_ld + h * DH : vb + (size_t)j * DH;
                const char4 x4 = *reinterpret_cast<const char4 *>(vr + el);
                const int v[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
                for (int u = 0; u < 4; u++) {
                    hi[u] += Eh * v[u];
                    lo[u] += El * v[u];
                }
            }
        }
#pragma unroll
        for (int o = LPK; o < 32; o <<= 1)
#pragma unroll
            for (int u = 0; u < 4; u++) {
                hi[u] += __shfl_xor_sync(0xFFFFFFFFu, hi[u], o);
                lo[u] += __shfl_xor_sync(0xFFFFFFFFu, lo[u], o);
            }
        if (LW == 0) {
            // the warp holds its item's whole sums: its lanes write the
            // context, the KPI lanes of a group sharing its 4 elements
            if (live) {
                constexpr int UPL = 4 / KPI;
#pragma unroll
                for (int u = 0; u < 4; u++)
                    if (u / UPL == kg)
                        ctx[(size_t)m * P.d + h * DH + el + u] =
                            q8_quotient((long long)hi[u] * 4096 + lo[u], z, rho, dc_rn32_div);
            }
            __syncthreads();
            continue;
        }
        if (kg == 0)
#pragma unroll
            for (int u = 0; u < 4; u++) pn[warp * DH + el + u] = (long long)hi[u] * 4096 + lo[u];
        if (lane == 0) pz[warp] = z;
        __syncthreads();
        for (int x = threadIdx.x; x < ip * DH; x += DC_THREADS) {
            const int ii = x / DH, e = x - ii * DH;
            const int it2 = base + ii;
            if (it2 < items) {
                long long N = 0, Z = 0;
                for (int w = 0; w < wpi; w++) {
                    N += pn[(ii * wpi + w) * DH + e];
                    Z += pz[ii * wpi + w];
                }
                const int m2 = dc_row_of<RM>(it2, H, R), h2 = it2 - m2 * H;
                ctx[(size_t)m2 * P.d + h2 * DH + e] = q8_quotient(N, Z, rho, dc_rn32_div);
            }
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// the step kernel: one generic phase body run 1 + 6 * n_dec times
// ---------------------------------------------------------------------------
// commit the greedy selection of decode step tp (one thread): the token per
// row into the history and the next input, the finished flags, the cleared
// keys for the next vocabulary kernel, the step counter; done if requested
__device__ __noinline__ void dc_commit_greedy(const DcParams &P, int tp, const int *out, const int *fin, int done) {
    for (int m = 0; m < P.R; m++) {
        P.hist[(size_t)tp * P.R + m] = out[m];
        P.tok_w[m] = out[m];
        P.fin[m] = fin[m];
        P.keys[m] = 0ull;
    }
    *P.t_w = tp + 1;
    if (done) *P.done_w = 1;
    *P.pending = 0;
}

enum { K_EMB = -1, K_QKV = 0, K_O = 1, K_Q2 = 2, K_O2 = 3, K_W1 = 4, K_W2 = 5 };

// bytes a CTA receives in the exchange of phase ph (host-computed): the full
// int8 vector (qkv, q2, h) or the fp32 residual plus every slice's [R]
// max / min pair
MNMT_DEV uint32_t dc_xbytes(const DcParams &P, int ph) { return P.phase[ph].xbytes; }

// W4: the model's attention / FFN linears hold 4-bit codes (a separate
// instantiation, so the int8 step carries no 4-bit code)
template <int DH, bool W4, int RM, int FL>
__global__ void __launch_bounds__(DC_THREADS, 1) decode_cluster_kernel(const DcParams *__restrict__ Pp) {
    // Launched as a programmatic dependent of the previous step's vocabulary
    // kernel: everything up to dc_grid_wait() reads only data that no kernel
    // of the decode loop writes (parameters, weights, LayerNorm vectors, the
    // encoder's cross keys / values), so it overlaps the previous kernel.
    // `done` only turns 0 -> 1 within a translation: seen set, it is final.
    if (*Pp->done) return;  // uniform for the whole cluster
#ifdef MNMT_DC_STAMPS
    const unsigned long long ns_start = dc_gtime();
#endif
    extern __shared__ __align__(16) uint8_t smem[];
    {
        // the parameter block lives in shared memory for the whole step
        const int n16 = (int)(sizeof(DcParams) / 16);
        for (int i = threadIdx.x; i < n16; i += DC_THREADS)
            reinterpret_cast<int4 *>(smem)[i] = reinterpret_cast<const int4 *>(Pp)[i];
        if (threadIdx.x == 0) {
            // the weight ring's mbarriers and the two exchange barriers, one
            // arrival per phase each; the exchange barriers of phases 0 and 1
            // are armed with the bytes they receive
            const uint32_t b0 = dc_smem_u32(smem + Pp->off_bar);
            for (int i = 0; i < DC_NB + 2; i++) mbar_init(b0 + 8u * (uint32_t)i, 1u);
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
            for (int i = 0; i < 2; i++) mbar_expect_tx(b0 + 8u * (uint32_t)(DC_NB + i), dc_xbytes(*Pp, i));
        }
        __syncthreads();
        // the barriers are set before any CTA of the cluster may store into
        // this one (each waits for every arrival before its first exchange)
        asm volatile("barrier.cluster.arrive.release;\n" ::: "memory");
    }
    const DcParams &P = *reinterpret_cast<const DcParams *>(smem);
    // FL >= 0: the model's pre-LN (bit 0) and factorised-embedding (bit 1)
    // flags and R * d > 256 (bit 2) fixed at compile time, so the other
    // variants' code is not in the kernel; FL < 0: read from the parameters
    const bool pre_ln = FL < 0 ? P.pre_ln != 0 : (FL & 1) != 0;
    const bool factorised = FL < 0 ? P.factorised != 0 : (FL & 2) != 0;
    constexpr int TW = FL < 0 ? -1 : ((FL >> 2) & 1);  // row width above 256 (bit 2); bits 3-4: log2 warps per attention item
    const uint32_t bars = dc_smem_u32(smem + P.off_bar), xbars = bars + 8u * DC_NB;
    cg::cluster_group cl = cg::this_cluster();
    const int c = (int)cl.block_rank();
    const int nc = P.nc;
    const int R = P.R, d = P.d, F = P.F, H = P.H;

    float *r_full = reinterpret_cast<float *>(smem + P.off_r);
    int8_t *a_full = reinterpret_cast<int8_t *>(smem + P.off_a);
    int8_t *qkv_full = reinterpret_cast<int8_t *>(smem + P.off_qkv);
    int8_t *ctx_full = reinterpret_cast<int8_t *>(smem + P.off_ctx);
    int8_t *q2_full = reinterpret_cast<int8_t *>(smem + P.off_q2);
    int8_t *h_full = reinterpret_cast<int8_t *>(smem + P.off_h);
    // the slice's staging buffer alternates by phase: a thread may still be
    // storing the previous phase's slice to other CTAs (the exchange only
    // waits for what this CTA receives) when a faster one writes the next
    uint8_t *const stage2 = smem + P.off_stage;
    int *att = reinterpret_cast<int *>(smem + P.off_att);
    uint8_t *ring = smem + P.off_ring;
    float *lnp = reinterpret_cast<float *>(smem + P.off_ln);                  // [n_dec][6][d] + final [2][d]
    float *red_f = reinterpret_cast<float *>(smem + P.off_red);               // [8]
    long long *red_l = reinterpret_cast<long long *>(smem + P.off_red + 64);  // [8]
    long long *pn = reinterpret_cast<long long *>(smem + P.off_red + 128);    // [8][DH]
    int *tok_s = reinterpret_cast<int *>(smem + P.off_red + 128 + 8 * DH * 8);  // [R]
    unsigned *mm = reinterpret_cast<unsigned *>(smem + P.off_part);               // [R][nc][2] slice max / min of r
    long long *part_l = reinterpret_cast<long long *>(smem + P.off_part + 512);    // [2][64] LN partials, [R] (mu, eb)
    const int nphase = 1 + 6 * P.n_dec;

    // the LayerNorm vectors of every layer (+ the final LN), the first DC_NB
    // weight slices and the cross keys / values the step attends to
    dc_copy(lnp, P.ln_all, (6 * P.n_dec + 2) * d * 4);
    for (int i = 0; i < DC_NB; i++) dc_prefetch(P, i, c, ring, bars);
    if (P.kv_staged) {
        // one layer's cross K (or V) is one contiguous [R][H][S][dh] block: the
        // 2 * n_dec blocks go in one flat loop of 16-byte chunks
        const int cpb = R * P.S * d / 16;
        for (int blk = 0; blk < 2 * P.n_dec; blk++) {
            const DcLayer &Y = P.layer[blk >> 1];
            const int8_t *src = blk & 1 ? Y.cross_v : Y.cross_k;
            uint8_t *dst = smem + P.off_kvc + (size_t)blk * cpb * 16;
            for (int ch = threadIdx.x; ch < cpb; ch += DC_THREADS) dc_cp16(dst + (size_t)ch * 16, src + (size_t)ch * 16);
        }
    }
    // ---- the previous step's results: token, position, self keys / values ----
#ifdef MNMT_DC_STAMPS
    const unsigned long long ns_w0 = dc_gtime();
#endif
    dc_grid_wait();
    // every word of the decode state this step reads, in one round of loads
    const int done_v = *P.done, t_v = *P.t_ptr, pend_v = *P.pending, tmax_v = *P.tmax_ptr;
    unsigned long long key_v = 0ull;
    int fin_v = 0, tok_v = 0, srcl_v = 0;
    if (threadIdx.x < R) {
        key_v = P.keys[threadIdx.x];
        fin_v = P.fin[threadIdx.x];
        tok_v = P.tok[threadIdx.x];
        srcl_v = P.src_len[threadIdx.x];
    }
    if (done_v) {  // uniform for the whole cluster; no copy may outlive the CTA
        asm volatile("cp.async.wait_all;\n" ::);
        for (int i = 0; i < DC_NB; i++) dc_wait_slice(P, i, bars);
        return;
    }
    int t = t_v;
    // The previous step's vocabulary kernel left its greedy selection pending
    // (row maxima in keys): apply it here -- every CTA computes the same
    // tokens and finished flags from the same data; CTA 0 commits them (token,
    // history, flags, step counter, cleared keys) at the end of this step, or
    // at once if the translation has just finished.
    static_assert(4 * DC_RMAX <= 16, "tokens, pending tokens, flags and source lengths share the 16-int token area");
    int *s_out = tok_s + DC_RMAX, *s_fin = tok_s + 2 * DC_RMAX;  // no static shared memory: the
                                                                 // dynamic carve-up may take all 227 KB
    int *src_len_s = tok_s + 3 * DC_RMAX;
    if (threadIdx.x < R) src_len_s[threadIdx.x] = srcl_v;  // read from phase 0 on (after its block barrier)
    const bool pend = pend_v != 0;
    if (pend) {
        if (threadIdx.x < R) {
            const int y = (int)key_index(key_v);
            s_out[threadIdx.x] = fin_v ? P.pad : y;
            s_fin[threadIdx.x] = (fin_v || y == P.eos) ? 1 : 0;
        }
        __syncthreads();
        int all = 1;
        for (int m = 0; m < R; m++) all &= s_fin[m];
        if (all || t + 1 >= tmax_v) {  // uniform over the cluster
            if (c == 0 && threadIdx.x == 0) dc_commit_greedy(P, t, s_out, s_fin, 1);
            asm volatile("cp.async.wait_all;\n" ::);
            for (int i = 0; i < DC_NB; i++) dc_wait_slice(P, i, bars);
            return;
        }
        t = t + 1;
    }
    const bool stamp = c == 0 && threadIdx.x == 0 && t == DC_STAMP_STEP;
    (void)stamp;
#ifdef MNMT_DC_STAMPS
    if (stamp) {
        g_dc_ns[0] = ns_start;
        g_dc_ns[1] = ns_w0;
        g_dc_ns[2] = dc_gtime();
    }
#endif
    if (threadIdx.x < R) {
        int id = pend ? s_out[threadIdx.x] : tok_v;
        if (id < 0 || id >= P.V) {
            set_status(P.status, MNMT_EINVAL);
            id = 0;
        }
        tok_s[threadIdx.x] = id;
    }
    if (P.kv_staged && t > 0) {
        // positions 0..t-1 of every (layer, K/V, row, head): segments of t * dh
        // bytes, [T][dh] apart in the cache, one warp per segment
        const int cps = t * (DH / 16), RH = R * H;
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        for (int lkv = 0; lkv < 2 * P.n_dec; lkv++) {
            const DcLayer &Y = P.layer[lkv >> 1];
            const int8_t *src0 = lkv & 1 ? Y.self_v : Y.self_k;
            for (int mh = warp; mh < RH; mh += DC_WARPS) {
                uint8_t *dst = smem + P.off_kvs + ((size_t)lkv * RH + mh) * P.T * DH;
                const int8_t *src = src0 + (size_t)mh * P.T * DH;
                for (int ch = lane; ch < cps; ch += 32) dc_cp16(dst + (size_t)ch * 16, src + (size_t)ch * 16);
            }
        }
    }
    DC_STAMP(stamp, 3);
    asm volatile("barrier.cluster.wait.acquire;\n" ::: "memory");

    for (int ph = 0; ph < nphase; ph++) {
        const int kind = ph == 0 ? K_EMB : (ph - 1) % 6;
        const int l = ph == 0 ? 0 : (ph - 1) / 6;
        const DcLayer &Y = P.layer[l];
        // from the last phase on, the vocabulary kernel may launch and fetch its weights
        if (ph == nphase - 1) dc_launch_dependents();
        // Each thread waits for the slice itself.  Every buffer this phase's
        // prep writes was last read before the block barrier that follows the
        // previous phase's GEMV; what this CTA receives is complete once the
        // exchange wait that ended that phase returns.  Phase 0 reads the
        // tokens of the prologue, phase 1 on the LayerNorm vectors and (phase 2
        // on) the staged keys / values: both cross a block barrier.
        if (ph == 1) asm volatile("cp.async.wait_all;\n" ::: "memory");
        dc_wait_slice(P, ph, bars);
        if (ph <= 1) __syncthreads();
        DC_STAMP(stamp, 4 + 4 * ph);
        const uint8_t *slot = ring + (size_t)(ph % DC_NB) * P.slot_bytes;
        const float *lnl = lnp + (size_t)6 * l * d;

        // ---- the phase's input vector ----
        const int8_t *A = a_full;
        int K = d;
        if (kind == K_EMB) {
            if (factorised)
                for (int i = threadIdx.x; i < R * P.E; i += DC_THREADS)
                for (int m = 0; m < R; m++)
                    if (i >= m * P.E && i < (m + 1) * P.E) a_full[i] = P.emb_q[(size_t)tok_s[m] * P.E + (i - m * P.E)];
            K = P.E;
        } else if (kind == K_QKV || kind == K_Q2 || kind == K_W1) {
            // pre-LN: LN of this sublayer; post-LN: LN of the previous sublayer's
            // residual (written back), or plain quantisation for the first one
            const int w = kind == K_QKV ? 0 : (kind == K_Q2 ? 2 : 4);
            const float inv_in = kind == K_QKV ? Y.inv_in1 : (kind == K_Q2 ? Y.inv_in2 : Y.inv_in3);
            if (pre_ln) {
                dc_layernorm<RM, TW>(r_full, R, d, lnl + w * d, lnl + (w + 1) * d, inv_in, a_full, 0, P.status, mm, nc, part_l, P.ln_kd, P.ln_dodd, P.ln_zm);
            } else if (kind == K_QKV) {
                for (int i = threadIdx.x; i < R * d; i += DC_THREADS) a_full[i] = q8(r_full[i], inv_in);
            } else {
                dc_layernorm<RM, TW>(r_full, R, d, lnl + (w - 2) * d, lnl + (w - 1) * d, inv_in, a_full, 1, P.status, mm, nc,
                             part_l, P.ln_kd, P.ln_dodd, P.ln_zm);
            }
        } else if (kind == K_O || kind == K_O2) {
            const int cross = kind == K_O2;
            dc_attention<DH, RM, (FL < 0 ? -1 : ((FL >> 3) & 3))>(P, l, cross, cross ? q2_full : qkv_full, cross ? d : 3 * d, qkv_full + d,
                             qkv_full + 2 * d, 3 * d, t, ctx_full, att, red_f, red_l, pn, smem, src_len_s);
            A = ctx_full;
        } else {  // K_W2
            A = h_full;
            K = F;
        }
        __syncthreads();
        DC_STAMP(stamp, 5 + 4 * ph);

        // ---- the phase's slice of outputs ----
        const int rows = ph == 0 ? P.phase[0].cpr * 4 : P.phase[ph].rows;  // phase 0: d / nc fp32 values
        const int n0 = c * rows;
        const int out_f32 = P.phase[ph].out_f32;
        const float sx = P.phase[ph].sx, gam = P.phase[ph].gam;
        uint8_t *stage = stage2 + (ph & 1) * P.stage_bytes;
        float *stf = reinterpret_cast<float *>(stage);
        int8_t *sti = reinterpret_cast<int8_t *>(stage);
        if (kind == K_EMB && !factorised) {
            for (int i = threadIdx.x; i < R * rows; i += DC_THREADS) {
                const int m = dc_row_of<RM>(i, rows, R), nl = i - m * rows, n = n0 + nl, id = tok_s[m];
                const float v = __fmul_rn(__fmul_rn((float)P.emb_q[(size_t)id * P.E + n], P.emb_s[id]), P.emb_scale);
                stf[i] = __fadd_rn(v, P.pe[(size_t)t * d + n]);
            }
        } else {
            // the slot: W rows (rows * K int8 codes, or rows * K / 2 bytes of
            // packed 4-bit codes), then s, b, inv [rows] and, for min-max
            // 4-bit rows, the offsets m [rows]
            const DcPhase &f = P.phase[ph];
            const bool w4 = W4 && kind != K_EMB && f.bits == 4;
            const int rb = w4 ? K / 2 : K;  // weight bytes per row
            const int8_t *W = reinterpret_cast<const int8_t *>(slot);
            const float *sw = reinterpret_cast<const float *>(slot + rows * rb);
            const float *bb = sw + rows;
            const float *iv = bb + rows;
            const float *mw = (w4 && f.m) ? iv + rows : nullptr;
            const int kc = rb / 16;  // 16-byte weight chunks per row (4-bit: one run of 32 codes each)
            // lpr = 2^lg lanes per row (host-chosen: a power of two dividing kc,
            // at most 32, no more than spreads the slice's rows over the block's
            // 256 threads; each lane takes kc / lpr chunks)
            const int lg = f.lg, lpr = 1 << lg;
            const int cpl = kc >> lg;
            const int rpw = 32 >> lg;              // rows per warp pass
            const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
            const int sub = lane & (lpr - 1);
            const int4 ones = make_int4(0x01010101, 0x01010101, 0x01010101, 0x01010101);
            for (int r0 = warp * rpw; r0 < rows; r0 += DC_WARPS * rpw) {
                const int nl = r0 + (lane >> lg);
                int acc[RM], a1[RM];  // a1: 4-bit rows, the activation codes' sums
#pragma unroll
                for (int m = 0; m < RM; m++) acc[m] = a1[m] = 0;
                if (nl < rows) {
                    const int4 *wr = reinterpret_cast<const int4 *>(W + (size_t)nl * rb);
                    for (int q = 0; q < cpl; q++) {
                        const int k = q * lpr + sub;  // consecutive lanes read consecutive chunks
                        const int4 w = wr[k];
                        if (w4) {
                            const int4 lo = make_int4(w.x & 0x0F0F0F0F, w.y & 0x0F0F0F0F, w.z & 0x0F0F0F0F,
                                                      w.w & 0x0F0F0F0F);
                            const int4 hi = make_int4((w.x >> 4) & 0x0F0F0F0F, (w.y >> 4) & 0x0F0F0F0F,
                                                      (w.z >> 4) & 0x0F0F0F0F, (w.w >> 4) & 0x0F0F0F0F);
#pragma unroll
                            for (int m = 0; m < RM; m++)
                                if (m < R) {
                                    const int4 *am = reinterpret_cast<const int4 *>(A + (size_t)m * K);
                                    const int4 x0 = am[2 * k], x1 = am[2 * k + 1];
                                    acc[m] = dot16(x1, hi, dot16(x0, lo, acc[m]));
                                    a1[m] = dot16(x1, ones, dot16(x0, ones, a1[m]));
                                }
                        } else {
#pragma unroll
                            for (int m = 0; m < RM; m++)
                                if (m < R)
                                    acc[m] = dot16(reinterpret_cast<const int4 *>(A + (size_t)m * K)[k], w, acc[m]);
                        }
                    }
                }
#pragma unroll
                for (int m = 0; m < RM; m++)
                    if (m < R)
                        for (int o = lpr / 2; o > 0; o >>= 1) {
                            acc[m] += __shfl_xor_sync(0xFFFFFFFFu, acc[m], o);
                            if (w4) a1[m] += __shfl_xor_sync(0xFFFFFFFFu, a1[m], o);
                        }
                if (sub == 0 && nl < rows) {
                    const int n = n0 + nl;
#pragma unroll
                    for (int m = 0; m < RM; m++) {
                        if (m >= R) break;
                        if (kind == K_EMB) {
                            const float y = dequant_bias(acc[m], P.emb_s[tok_s[m]], sw[nl], bb[nl]);
                            stf[m * rows + nl] = __fadd_rn(__fmul_rn(y, P.emb_scale), P.pe[(size_t)t * d + n]);
                            continue;
                        }
                        float y;
                        if (!w4) {
                            y = dequant_bias(acc[m], sx, sw[nl], bb[nl]);
                        } else if (!mw) {  // symmetric 4-bit rows: stored code v + 8
                            y = dequant_bias(acc[m] - 8 * a1[m], sx, sw[nl], bb[nl]);
                        } else {  // min-max rows: W = s u + r
                            const float tt = __fmul_rn(__int2float_rn(acc[m]), __fmul_rn(sx, sw[nl]));
                            const float oo = __fmul_rn(__int2float_rn(a1[m]), __fmul_rn(sx, mw[nl]));
                            y = __fadd_rn(__fadd_rn(tt, oo), bb[nl]);
                        }
                        if (out_f32) {
                            stf[m * rows + nl] = __fadd_rn(__fmul_rn(gam, r_full[(size_t)m * d + n]), y);
                        } else {
                            const int8_t v = q8(kind == K_W1 && !(y > 0.0f) ? 0.0f : y, iv[nl]);
                            sti[m * rows + nl] = v;
                            if (kind == K_QKV && n >= d) {  // K / V of position t into the layer's cache
                                const int seg = n >= 2 * d;
                                const int cc = n - (seg ? 2 * d : d);
                                const int hh = cc / DH, ii = cc - hh * DH;
                                (seg ? Y.self_v : Y.self_k)[(((size_t)m * H + hh) * P.T + t) * DH + ii] = v;
                            }
                        }
                    }
                }
            }
        }
        __syncthreads();
        DC_STAMP(stamp, 6 + 4 * ph);
        // the slot is free again: the slice of phase ph + DC_NB goes into it,
        // issued by the last warp, which the small broadcasts leave idle (a
        // thread issuing bulk copies is held for a few hundred ns)
        dc_prefetch(P, ph + DC_NB, c, ring, bars, DC_THREADS - 32);
        // ---- publish the slice to every CTA ----
        const uint32_t xbar = xbars + 8u * (uint32_t)(ph & 1);
        if (out_f32) {
            // the slice's largest and smallest residual value per row (rows <= 32),
            // for the next LayerNorm's grids
            if (threadIdx.x < 32 * R) {
                const int m = threadIdx.x >> 5, ln = threadIdx.x & 31;
                unsigned kmax = 0u, kmin = 0xFFFFFFFFu;
                for (int i = ln; i < rows; i += 32) {
                    const unsigned k = ordered_bits(stf[m * rows + i]);
                    kmax = k > kmax ? k : kmax;
                    kmin = k < kmin ? k : kmin;
                }
                const unsigned kh = __reduce_max_sync(0xFFFFFFFFu, kmax);
                const unsigned kl = __reduce_min_sync(0xFFFFFFFFu, kmin);
                if (ln < nc)
                    dc_st_async2(dc_mapa(dc_smem_u32(mm + (m * nc + c) * 2), ln), kh, kl, dc_mapa(xbar, ln));
            }
            dc_bcast(P.phase[ph], stage, R, rows * 4, reinterpret_cast<uint8_t *>(r_full), d * 4, n0 * 4, nc, xbar);
        } else {
            int8_t *full = kind == K_QKV ? qkv_full : (kind == K_Q2 ? q2_full : h_full);
            const int width = kind == K_QKV ? 3 * d : (kind == K_Q2 ? d : F);
            dc_bcast(P.phase[ph], stage, R, rows, reinterpret_cast<uint8_t *>(full), width, n0, nc, xbar);
        }
        // the whole vector of this phase, from every CTA
        if (!mbar_wait(xbar, (uint32_t)(ph >> 1) & 1u)) set_status(P.status, MNMT_ETIMEOUT);
        if (threadIdx.x == 0 && ph + 2 < nphase) mbar_expect_tx(xbar, dc_xbytes(P, ph + 2));
        DC_STAMP(stamp, 7 + 4 * ph);
        if (kind == K_W2 && !pre_ln) {
            // post-LN: the FFN's LayerNorm normalises the stream in place
            const bool last = l + 1 == P.n_dec;
            const float inv = last ? P.inv_dout : P.layer[l + 1].inv_in1;
            dc_layernorm<RM, TW>(r_full, R, d, lnl + 4 * d, lnl + 5 * d, inv, a_full, 1, P.status, mm, nc, part_l, P.ln_kd, P.ln_dodd, P.ln_zm);
        }
    }
    DC_STAMP(stamp, 100);
    // ---- final LayerNorm + quantisation -> vocabulary input ----
    if (pre_ln)
        dc_layernorm<RM, TW>(r_full, R, d, lnp + (size_t)6 * P.n_dec * d, lnp + (size_t)(6 * P.n_dec + 1) * d,
                     P.inv_dout, a_full, 0, P.status, mm, nc, part_l, P.ln_kd, P.ln_dodd, P.ln_zm);
    __syncthreads();
    if (c == 0) {
        for (int i = threadIdx.x; i < R * d; i += DC_THREADS) {
            P.act_out[i] = a_full[i];
            if (P.resid_out) P.resid_out[i] = r_full[i];
        }
    }
    DC_STAMP(stamp, 101);
    if (pend && c == 0 && threadIdx.x == 0) dc_commit_greedy(P, t - 1, s_out, s_fin, 0);
    // no closing cluster barrier: the last exchange has delivered everything
    // any CTA stores into this one
    DC_STAMP(stamp, 102);
}

// ---------------------------------------------------------------------------
// vocabulary projection + greedy argmax + greedy update (last block).  Each
// block owns a contiguous range of output rows, held in shared memory.
// ---------------------------------------------------------------------------
template <int MT>
__global__ void __launch_bounds__(256) vocab_greedy_kernel(const int8_t *__restrict__ A, const int8_t *__restrict__ W,
                                                           const float *__restrict__ s_w,
                                                           const float *__restrict__ bias, float s_x, int M, int N,
                                                           int K, int rows_per_block, unsigned long long *keys,
                                                           int *ticket, GreedyArgs g) {
    // Launched as a programmatic dependent of the step kernel: the block's
    // weight rows, scales and biases (static) are fetched into shared memory
    // while the step kernel finishes; only the input row waits for it.
#ifdef MNMT_DC_STAMPS
    const unsigned long long v_start = dc_gtime();
#endif
    dc_launch_dependents();
    extern __shared__ __align__(16) int4 vsm[];  // [rows][K/16] weights, [MT][K/16] input, [rows] scale, [rows] bias
    const int kc = K >> 4;
    const int n0 = blockIdx.x * rows_per_block;
    const int nr = min(rows_per_block, N - n0);
    int4 *ws = vsm;
    int4 *as = vsm + (size_t)rows_per_block * kc;
    float *scs = reinterpret_cast<float *>(as + MT * kc);
    float *bss = scs + rows_per_block;
    for (int i = threadIdx.x; i < nr * kc; i += 256) dc_cp16(ws + i, reinterpret_cast<const int4 *>(W + (size_t)n0 * K) + i);
    dc_commit();
    for (int i = threadIdx.x; i < nr; i += 256) {
        scs[i] = __fmul_rn(s_x, s_w[n0 + i]);
        bss[i] = bias[n0 + i];
    }
#ifdef MNMT_DC_STAMPS
    const unsigned long long v_w0 = dc_gtime();
#endif
    const int am = dc_row_of((int)threadIdx.x, kc, MT <= DC_RMAX ? MT : DC_RMAX);  // row of this thread's input chunk
    const bool aload = (int)threadIdx.x < MT * kc && am < M;
    const int4 *asrc = reinterpret_cast<const int4 *>(A + (size_t)am * K) + ((int)threadIdx.x - am * kc);
    dc_grid_wait();
    // the done flag and the first chunk of input rows in one round of loads
    const int done_v = *g.done;
    int4 a0 = make_int4(0, 0, 0, 0);
    if (aload) a0 = *asrc;
#ifdef MNMT_DC_STAMPS
    if (blockIdx.x == 0 && threadIdx.x == 0 && *g.t_ptr == DC_STAMP_STEP - 1) {
        g_dc_ns[110] = v_start;
        g_dc_ns[111] = v_w0;
        g_dc_ns[112] = dc_gtime();
    }
#endif
    if (done_v) {  // no copy may outlive the block
        asm volatile("cp.async.wait_all;\n" ::);
        return;
    }
    if ((int)threadIdx.x < MT * kc) as[threadIdx.x] = a0;
    for (int i = threadIdx.x + 256; i < MT * kc; i += 256) {
        const int m = i / kc, c = i - m * kc;
        as[i] = m < M ? reinterpret_cast<const int4 *>(A + (size_t)m * K)[c] : make_int4(0, 0, 0, 0);
    }
    asm volatile("cp.async.wait_all;\n" ::);
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // a lane pair per weight row (16 rows per warp and pass): lane l takes the
    // chunks k = (l & 1) + 2 j of its row, j rotated by the row so that the
    // warp's 16-byte loads spread over the shared-memory banks; one shuffle
    // joins the pair
    const int half = lane & 1, hk = kc >> 1;
    unsigned long long best[MT];
#pragma unroll
    for (int m = 0; m < MT; m++) best[m] = 0ull;
    for (int r0 = warp * 16; r0 < nr; r0 += 8 * 16) {
        const int row = r0 + (lane >> 1);
        int acc[MT];
#pragma unroll
        for (int m = 0; m < MT; m++) acc[m] = 0;
        if (row < nr) {
            int jj = (hk & (hk - 1)) == 0 ? (row & (hk - 1)) : row % hk;
            const int4 *wr = ws + (size_t)row * kc;
            for (int j = 0; j < hk; j++) {
                const int cc = half + 2 * jj;
                const int4 w = wr[cc];
#pragma unroll
                for (int m = 0; m < MT; m++) acc[m] = dot16(as[m * kc + cc], w, acc[m]);
                jj = jj + 1 == hk ? 0 : jj + 1;
            }
        }
#pragma unroll
        for (int m = 0; m < MT; m++) acc[m] += __shfl_xor_sync(0xFFFFFFFFu, acc[m], 1);
        if (half == 0 && row < nr) {
#pragma unroll
            for (int m = 0; m < MT; m++) {
                if (m < M) {
                    const float y = __fadd_rn(__fmul_rn(__int2float_rn(acc[m]), scs[row]), bss[row]);
                    const unsigned long long k = pack_key(y, (uint32_t)(n0 + row));
                    best[m] = k > best[m] ? k : best[m];
                }
            }
        }
    }
    __shared__ unsigned long long red[8][MT];
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
    // The greedy bookkeeping of this step (token, history, finished flags,
    // step counter) is left to the next step kernel, which reads the keys
    // after waiting for this grid anyway, or to the greedy update closing a
    // run of steps: no fence, ticket or last-block pass on the step's path.
    if (blockIdx.x == 0 && threadIdx.x == 0) *g.pending = 1;
    DC_STAMP(blockIdx.x == 0 && threadIdx.x == 0 && *g.t_ptr == DC_STAMP_STEP - 1, 113);
    (void)ticket;
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
// CTAs per cluster: a slice of at least 16 columns of d per CTA, at most
// MNMT_DC_MAX_CTAS (default 16, the largest cluster; measured fastest) CTAs
int dc_cluster_size(int d, int F, int E) {
    int cap = 16;
    if (const char *e = getenv("MNMT_DC_MAX_CTAS")) cap = atoi(e);
    if (cap < 2) cap = 2;
    if (cap > 16) cap = 16;
    // every phase's slice (d, 3d, F or the factorised width's d columns per
    // CTA, as int8 or fp32) must be a whole number of 16-byte chunks
    for (int nc = cap; nc >= 2; nc--)
        if (d % (16 * nc) == 0 && (3 * d) % (16 * nc) == 0 && F % (16 * nc) == 0 && E % 16 == 0) return nc;
    return 0;
}

// Fills the phase table and the shared-memory carve-up; returns the bytes of
// shared memory one CTA needs (staging the keys / values when they fit in
// max_smem).
size_t dc_layout(DcParams &P, size_t max_smem) {
    const int R = P.R, d = P.d, F = P.F, nc = P.nc;
    // phase table: slices of CTA c are rows [c * rows, (c + 1) * rows)
    DcPhase z = {nullptr, nullptr, nullptr, nullptr, nullptr, 0, 0, 8};
    P.phase[0] = z;
    if (P.factorised) P.phase[0] = DcPhase{P.proj.w, P.proj.s, P.proj.b, nullptr, nullptr, d / nc, P.E, 8};
    auto ph = [](const DcLin &x, const float *inv, int rows, int K) {
        return DcPhase{x.w, x.s, x.b, inv, x.m, rows, K, x.bits};
    };
    for (int l = 0; l < P.n_dec; l++) {
        const DcLayer &Y = P.layer[l];
        DcPhase *f = &P.phase[1 + 6 * l];
        f[0] = ph(Y.qkv, Y.inv_qkv, 3 * d / nc, d);
        f[1] = ph(Y.o, nullptr, d / nc, d);
        f[2] = ph(Y.q2, Y.inv_q2, d / nc, d);
        f[3] = ph(Y.o2, nullptr, d / nc, d);
        f[4] = ph(Y.w1, Y.inv_h, F / nc, d);
        f[5] = ph(Y.w2, nullptr, d / nc, F);
    }
    // exchange geometry: slices of fp32 residual values (embedding, O, O2, W2)
    // or int8 codes (qkv, q2, h); the slice GEMV's lane groups and epilogue
    // constants
    auto magic = [](int v) { return v > 1 ? (uint32_t)((0x100000000ull + (uint64_t)v - 1) / (uint64_t)v) : 0u; };
    for (int ph = 0; ph < 1 + 6 * P.n_dec; ph++) {
        const int kind = ph == 0 ? -1 : (ph - 1) % 6;
        const bool f32 = kind == -1 || kind == 1 || kind == 3 || kind == 5;
        const int rows = ph == 0 ? d / nc : P.phase[ph].rows;
        const int cpr = f32 ? rows / 4 : rows / 16;
        P.phase[ph].cpr = cpr;
        P.phase[ph].mg_rc = magic(R * cpr);
        P.phase[ph].mg_c = magic(cpr);
        DcPhase &f = P.phase[ph];
        const int kc = (f.bits == 4 ? f.K / 2 : f.K) / 16;
        int lpr = kc & -kc;
        if (lpr > 32) lpr = 32;
        while (lpr > 1 && f.rows * lpr > DC_THREADS) lpr >>= 1;
        int lg = 0;
        while ((1 << lg) < lpr) lg++;
        f.lg = kc > 0 ? lg : 0;
        f.out_f32 = f32 ? 1 : 0;
        f.xbytes = (uint32_t)(f32 ? R * d * 4 + R * nc * 8 : R * (kind == 0 ? 3 * d : (kind == 2 ? d : F)));
        const DcLayer &Y = P.layer[ph == 0 ? 0 : (ph - 1) / 6];
        switch (kind) {
            case 0: f.sx = Y.s_in1; f.gam = 0.0f; break;
            case 1: f.sx = Y.s_ctx1; f.gam = Y.gamma1; break;
            case 2: f.sx = Y.s_in2; f.gam = 0.0f; break;
            case 3: f.sx = Y.s_ctx2; f.gam = Y.gamma2; break;
            case 4: f.sx = Y.s_in3; f.gam = 0.0f; break;
            case 5: f.sx = Y.s_h; f.gam = Y.gamma3; break;
            default: f.sx = 0.0f; f.gam = 0.0f; break;
        }
    }
    {
        const int items = R * P.H;
        const int ip = items >= DC_WARPS ? DC_WARPS : (items > 4 ? 8 : (items > 2 ? 4 : (items > 1 ? 2 : 1)));
        int lw = 0;
        while ((DC_WARPS >> lw) > ip) lw++;  // DC_WARPS / ip = 2^lw warps per item
        P.att_ip = ip;
        P.att_lw = lw;
        int kd = 0;
        while (((d >> kd) & 1) == 0) kd++;
        P.ln_kd = kd;
        P.ln_dodd = d >> kd;
        P.ln_zm = P.ln_dodd > 1 ? ~0ull / (unsigned long long)P.ln_dodd : 0ull;  // floor(2^64 / dodd), dodd odd
    }
    // shared-memory carve-up (16-byte aligned pieces)
    size_t off = 0;
    auto take = [&](size_t bytes) {
        size_t at = off;
        off += (bytes + 15) & ~(size_t)15;
        return (int)at;
    };
    take(sizeof(DcParams));  // the parameter block itself
    P.off_ln = take((size_t)(6 * P.n_dec + 2) * d * 4);
    P.off_r = take((size_t)R * d * 4);
    P.off_a = take((size_t)R * d);
    P.off_qkv = take((size_t)R * 3 * d);
    P.off_ctx = take((size_t)R * d);
    P.off_q2 = take((size_t)R * d);
    P.off_h = take((size_t)R * F);
    int stage_bytes = R * (d / nc) * 4;
    if (R * 3 * d / nc > stage_bytes) stage_bytes = R * 3 * d / nc;
    if (R * F / nc > stage_bytes) stage_bytes = R * F / nc;
    P.stage_bytes = (stage_bytes + 15) & ~15;
    P.off_stage = take(2 * (size_t)P.stage_bytes);  // two, alternating by phase
    P.att_cap = P.T > P.S ? P.T : P.S;
    P.off_att = take((size_t)DC_WARPS * P.att_cap * 4);
    P.off_red = take(128 + (size_t)DC_WARPS * P.dh * 8 + 16 * 4);  // reductions, context partials, tokens
    P.off_part = take(512 + 1024 + 64);  // slice extremes [R][nc][2], LN partials [2][64], per-row (mu, eb)
    if (R * d > 64 * 32) return (size_t)-1;                         // 64 warp chunks of partials
    P.off_bar = take(8 * (DC_NB + 2));  // weight ring, then the two exchange barriers
    int slot = 0;
    for (int ph = 0; ph < 1 + 6 * P.n_dec; ph++) {
        const DcPhase &f = P.phase[ph];
        int b = f.rows * (f.bits == 4 ? f.K / 2 : f.K) + (f.m ? 16 : 12) * f.rows;
        if (b > slot) slot = b;
    }
    P.slot_bytes = (slot + 15) & ~15;
    P.off_ring = take((size_t)DC_NB * P.slot_bytes);
    // keys / values of every decoder layer: cross [L][2][R][H][S][dh], self [L][2][R][H][T][dh]
    const size_t kvc = (size_t)P.n_dec * 2 * R * P.S * d, kvs = (size_t)P.n_dec * 2 * R * P.T * d;
    P.kv_staged = 0;
    if (off + kvc + kvs + 32 <= max_smem) {
        P.kv_staged = 1;
        P.off_kvc = take(kvc);
        P.off_kvs = take(kvs);
    }
    return off;
}

// the step kernel of a head width, weight format and row count: int8 single-row
// steps (greedy batch 1) run an instantiation whose slice GEMV keeps one row
// of accumulators (a smaller kernel; the step is sensitive to its code size)
// (flags: the model's pre-LN / factorised-embedding / width > 256 bits and
// the attention's log2 warps per item, or -1; the single-row d_h = 64 steps
// of the measured models have them compiled in)
static const void *dc_kernel(int dh, bool w4, bool one_row, int flags = -1) {
    if (w4 && one_row && dh == 64 && flags == 11) return (const void *)decode_cluster_kernel<64, true, 1, 11>;
    if (w4)
        return dh == 32 ? (const void *)decode_cluster_kernel<32, true, DC_RMAX, -1>
                        : (dh == 64 ? (const void *)decode_cluster_kernel<64, true, DC_RMAX, -1>
                                    : (const void *)decode_cluster_kernel<128, true, DC_RMAX, -1>);
    if (one_row) {
        // small (pre-LN, factorised, 2 warps per head), 10MB (pre-LN, 2 warps
        // per head), 20MB (pre-LN, d > 256, one warp per head)
        if (dh == 64 && flags == 11) return (const void *)decode_cluster_kernel<64, false, 1, 11>;
        if (dh == 64 && flags == 9) return (const void *)decode_cluster_kernel<64, false, 1, 9>;
        if (dh == 64 && flags == 5) return (const void *)decode_cluster_kernel<64, false, 1, 5>;
        return dh == 32 ? (const void *)decode_cluster_kernel<32, false, 1, -1>
                        : (dh == 64 ? (const void *)decode_cluster_kernel<64, false, 1, -1>
                                    : (const void *)decode_cluster_kernel<128, false, 1, -1>);
    }
    return dh == 32 ? (const void *)decode_cluster_kernel<32, false, DC_RMAX, -1>
                    : (dh == 64 ? (const void *)decode_cluster_kernel<64, false, DC_RMAX, -1>
                                : (const void *)decode_cluster_kernel<128, false, DC_RMAX, -1>);
}

cudaError_t decode_cluster_init() {
    const int max_smem = 227 * 1024;
    cudaError_t err = cudaSuccess;
    auto setk = [&](const void *k) {
        if (err == cudaSuccess) err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, max_smem);
        if (err == cudaSuccess) err = cudaFuncSetAttribute(k, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    };
    for (int dh : {32, 64, 128})
        for (int v = 0; v < 3; v++) setk(dc_kernel(dh, v == 1, v == 2));
    for (int fl : {5, 9, 11}) setk(dc_kernel(64, false, true, fl));
    setk(dc_kernel(64, true, true, 11));
    // the vocabulary kernel keeps its SMs in the largest shared-memory
    // configuration, so the next step's cluster (about 200 KB per CTA) can
    // become resident beside it as soon as it is allowed to launch
    for (const void *k : {(const void *)vocab_greedy_kernel<1>, (const void *)vocab_greedy_kernel<2>,
                          (const void *)vocab_greedy_kernel<4>})
        if (err == cudaSuccess)
            err = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout, cudaSharedmemCarveoutMaxShared);
    for (const void *k : {(const void *)vocab_greedy_kernel<1>, (const void *)vocab_greedy_kernel<2>,
                          (const void *)vocab_greedy_kernel<4>})
        if (err == cudaSuccess) err = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, 100 * 1024);
    return err;
}

// can one cluster of nc CTAs with smem bytes each be resident?
bool decode_cluster_fits(int dh, int nc, size_t smem, bool w4, bool one_row, int flags) {
    if (smem > 227 * 1024) return false;
    const void *k = dc_kernel(dh, w4, one_row, flags);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(nc);
    cfg.blockDim = dim3(DC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = nc;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    int clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&clusters, k, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return clusters >= 1;
}

cudaError_t launch_decode_cluster(const DcParams *dP, int dh, int nc, size_t smem, bool w4, bool one_row,
                                  int flags, cudaStream_t st) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(nc);
    cfg.blockDim = dim3(DC_THREADS);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    // a programmatic dependent of the previous step's vocabulary kernel: the
    // cluster launches as soon as its SMs are free and runs its prologue
    // (parameters, LayerNorm vectors, cross keys / values) before it waits
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = nc;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    if (dh != 32 && dh != 64 && dh != 128) return cudaErrorInvalidValue;
    void *args[] = {(void *)&dP};
    return cudaLaunchKernelExC(&cfg, dc_kernel(dh, w4, one_row, flags), args);
}

cudaError_t launch_vocab_greedy(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                                int M, int N, int K, unsigned long long *keys, int *ticket, const GreedyArgs &g,
                                int reserved_sms, cudaStream_t st) {
    if (M < 1 || M > 4 || K % 32) return cudaErrorInvalidValue;  // whole chunk pairs per row
    // two blocks per SM, each holding its contiguous rows in shared memory, on
    // the SMs the step's cluster does not occupy: every block is resident (and
    // prefetching its rows) while the step runs, and the next step's cluster
    // finds its SMs free and runs its prologue while this kernel finishes
    int free_sms = device_sm_count() - reserved_sms;
    if (free_sms < 16) free_sms = 16;
    int blocks = 2 * free_sms;
    int rows = (N + blocks - 1) / blocks;
    if ((size_t)rows * K > 96 * 1024) rows = (96 * 1024) / K;
    blocks = (N + rows - 1) / rows;
    const int mt = M == 1 ? 1 : (M == 2 ? 2 : 4);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(blocks);
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = (size_t)rows * K + (size_t)mt * K + 8 * (size_t)rows;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    switch (mt) {
        case 1: return cudaLaunchKernelEx(&cfg, vocab_greedy_kernel<1>, A, W, s_w, bias, s_x, M, N, K, rows, keys, ticket, g);
        case 2: return cudaLaunchKernelEx(&cfg, vocab_greedy_kernel<2>, A, W, s_w, bias, s_x, M, N, K, rows, keys, ticket, g);
        default: return cudaLaunchKernelEx(&cfg, vocab_greedy_kernel<4>, A, W, s_w, bias, s_x, M, N, K, rows, keys, ticket, g);
    }
}

}  // namespace mnmt
