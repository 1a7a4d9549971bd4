// rows.cu -- row-wise kernels of the INT8 encoder-decoder: embedding gather
// (+ factorised projection), LayerNorm + requantisation, and the search steps
// (greedy argmax bookkeeping, beam log-softmax / top-k / reorder, init and
// final backtracking).
//
// LayerNorm (App. A / App. D) keeps the mean and the biased variance as exact
// fixed-point sums: each row's largest magnitude (an order-free maximum) sets a
// power-of-two grid on which every term r_i 2^(52-ea) or c_i^2 2^(52-2eb) is an
// integer below 2^52, accumulated in int64.  Any reduction tree therefore gives
// the same mean and rstd bits.
#include "common.cuh"
#include "internal.h"

namespace mnmt {

// ---------------------------------------------------------------------------
// LayerNorm kernel: one block of LN_T threads per row, thread t holding the
// VPT contiguous elements t*VPT ..  The row is short (d <= 2048) and a decode
// step has only a few hundred rows, so the work of a row is spread over four
// or eight warps to shorten each thread's dependent chain; the order-free maxima and
// exact fixed-point sums combine across warps through shared memory.  The
// row, gamma and beta are loaded together before the skip flag is tested.
// ---------------------------------------------------------------------------
template <int VPT, int LN_T>
__global__ void __launch_bounds__(LN_T) layernorm_kernel(LnArgs a) {
    pdl_grid_wait();
    __shared__ unsigned s_amax[LN_T / 32], s_bmax[LN_T / 32];
    __shared__ long long s_s1[LN_T / 32], s_s2[LN_T / 32];
    const int row = blockIdx.x, d = a.d;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    const int i0 = threadIdx.x * VPT;
    const float *r = a.r + (size_t)row * d;
    float x[VPT], gv[VPT], bv[VPT];
#pragma unroll
    for (int v = 0; v < VPT; v++) {
        const bool in = i0 + v < d;
        x[v] = in ? r[i0 + v] : 0.0f;
        gv[v] = in ? a.g[i0 + v] : 0.0f;
        bv[v] = in ? a.b[i0 + v] : 0.0f;
    }
    if (a.skip && *a.skip) return;
    // row maximum magnitude -> the grid of the exact sum of the elements
    unsigned am = 0;
#pragma unroll
    for (int v = 0; v < VPT; v++) am = max(am, __float_as_uint(x[v]) & 0x7FFFFFFFu);  // padding is 0
    am = __reduce_max_sync(0xFFFFFFFFu, am);
    if (lane == 0) s_amax[w] = am;
    __syncthreads();
    am = s_amax[0];
#pragma unroll
    for (int k = 1; k < LN_T / 32; k++) am = max(am, s_amax[k]);
    const float amax = __uint_as_float(am);
    if (!(amax < 0x1p32f)) {
        if (threadIdx.x == 0) set_status(a.status, MNMT_EOVERFLOW);
        return;
    }
    const int ea = exp_bound(amax);
    long long s1 = 0;
#pragma unroll
    for (int v = 0; v < VPT; v++) s1 += fx_scale(x[v], 52 - ea);  // padding adds 0
    s1 = warp_sum_exact(s1);
    if (lane == 0) s_s1[w] = s1;
    __syncthreads();
    s1 = 0;
#pragma unroll
    for (int k = 0; k < LN_T / 32; k++) s1 += s_s1[k];
    const float mu = rn32_scaled_div(s1, ea - 52, d);
    // centred values -> their maximum magnitude -> the grid of the variance sum
    float c[VPT];
    unsigned bm = 0;
#pragma unroll
    for (int v = 0; v < VPT; v++) {
        c[v] = __fsub_rn(x[v], mu);
        if (i0 + v < d) bm = max(bm, __float_as_uint(c[v]) & 0x7FFFFFFFu);
    }
    bm = __reduce_max_sync(0xFFFFFFFFu, bm);
    if (lane == 0) s_bmax[w] = bm;
    __syncthreads();
    bm = s_bmax[0];
#pragma unroll
    for (int k = 1; k < LN_T / 32; k++) bm = max(bm, s_bmax[k]);
    const int eb = exp_bound(__uint_as_float(bm));
    long long s2 = 0;
#pragma unroll
    for (int v = 0; v < VPT; v++)
        if (i0 + v < d) s2 += fx_scale(__fmul_rn(c[v], c[v]), 52 - 2 * eb);
    s2 = warp_sum_exact(s2);
    if (lane == 0) s_s2[w] = s2;
    __syncthreads();
    s2 = 0;
#pragma unroll
    for (int k = 0; k < LN_T / 32; k++) s2 += s_s2[k];
    const float var = rn32_scaled_div(s2, 2 * eb - 52, d);
    const float rstd = __fdiv_rn(1.0f, __fsqrt_rn(__fadd_rn(var, 1e-5f)));
    pdl_allow_next();  // only the normalise-and-store pass is left
#pragma unroll
    for (int v = 0; v < VPT; v++) {
        const int i = i0 + v;
        if (i < d) {
            const float y = __fadd_rn(__fmul_rn(__fmul_rn(c[v], rstd), gv[v]), bv[v]);
            if (a.out_f) a.out_f[(size_t)row * d + i] = y;
            if (a.out_q) {
                const int8_t q = q8(y, a.inv);
                a.out_q[(size_t)row * d + i] = q;
                if (a.out16) a.out16[(size_t)row * d + i] = __short2half_rn(q);
            }
        }
    }
}

template <int LN_T>
cudaError_t launch_layernorm_t(const LnArgs &a, cudaStream_t st) {
    const int vpt = (a.d + LN_T - 1) / LN_T;
    if (vpt <= 1) launch_pdl(layernorm_kernel<1, LN_T>, a.M, LN_T, 0, st, a);
    else if (vpt <= 2) launch_pdl(layernorm_kernel<2, LN_T>, a.M, LN_T, 0, st, a);
    else if (vpt <= 4) launch_pdl(layernorm_kernel<4, LN_T>, a.M, LN_T, 0, st, a);
    else if (vpt <= 8) launch_pdl(layernorm_kernel<8, LN_T>, a.M, LN_T, 0, st, a);
    else if (vpt <= 16) launch_pdl(layernorm_kernel<16, LN_T>, a.M, LN_T, 0, st, a);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

// a decode step's few hundred rows: 256 threads per row (shorter chains);
// an encoder's thousands: 128 (measured on the 512-row and 16384-row cases)
cudaError_t launch_layernorm(const LnArgs &a, cudaStream_t st) {
    if (a.M <= 0) return cudaSuccess;
    return a.M <= 1024 ? launch_layernorm_t<256>(a, st) : launch_layernorm_t<128>(a, st);
}

// ---------------------------------------------------------------------------
// embedding: one warp per row.  x = fl(fl(dequant(Eq[id]) * emb_scale) + PE[pos])
// (factorised: the E-dim int8 row feeds the E -> d linear, its row scale folded
// into the dequantisation), then r = x and the first sublayer's input
// q8(LN(x)) (pre-LN) or q8(x) (post-LN).
// ---------------------------------------------------------------------------
template <int VPL>
__global__ void __launch_bounds__(256) embed_kernel(EmbedArgs a) {
    pdl_grid_wait();
    if (a.skip && *a.skip) return;
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= a.M) return;
    int id = a.ids ? a.ids[row] : a.tok[row];
    const int pos = a.ids ? row % a.S : *a.t_ptr;
    if (id < 0 || id >= a.V) {
        if (lane == 0) set_status(a.status, MNMT_EINVAL);
        id = 0;
    }
    const float es = a.emb_s[id];
    const float *pe = a.pe + (size_t)pos * a.d;
    float x[VPL];
    if (!a.proj_w) {
        const int8_t *q = a.emb_q + (size_t)id * a.E;
#pragma unroll
        for (int u = 0; u < VPL; u++) {
            int i = u * 32 + lane;
            if (i < a.d) {
                float t = __fmul_rn(__fmul_rn((float)q[i], es), a.emb_scale);
                x[u] = __fadd_rn(t, pe[i]);
            } else {
                x[u] = 0.0f;
            }
        }
    } else {
        const int4 *q = reinterpret_cast<const int4 *>(a.emb_q + (size_t)id * a.E);
        const int ec = a.E / 16;
#pragma unroll
        for (int u = 0; u < VPL; u++) {
            int n = u * 32 + lane;
            x[u] = 0.0f;
            if (n < a.d) {
                const int4 *w = reinterpret_cast<const int4 *>(a.proj_w + (size_t)n * a.E);
                int acc = 0;
                for (int c = 0; c < ec; c++) acc = dot16(q[c], w[c], acc);
                float y = dequant_bias(acc, es, a.proj_s[n], a.proj_b[n]);
                x[u] = __fadd_rn(__fmul_rn(y, a.emb_scale), pe[n]);
            }
        }
    }
    float y[VPL];
    bool ok = true;
    if (a.ln_g) ok = warp_layernorm<VPL>(x, a.d, a.ln_g, a.ln_b, y, lane);
    if (!ok) {
        if (lane == 0) set_status(a.status, MNMT_EOVERFLOW);
        return;
    }
#pragma unroll
    for (int u = 0; u < VPL; u++) {
        int i = u * 32 + lane;
        if (i < a.d) {
            a.r[(size_t)row * a.d + i] = x[u];
            const int8_t v = q8(a.ln_g ? y[u] : x[u], a.inv);
            a.out_q[(size_t)row * a.d + i] = v;
            if (a.out16) a.out16[(size_t)row * a.d + i] = __short2half_rn(v);
        }
    }
}

cudaError_t launch_embed(const EmbedArgs &a, cudaStream_t st) {
    if (a.M <= 0) return cudaSuccess;
    dim3 grid((a.M + 7) / 8), block(256);
    int vpl = (a.d + 31) / 32;
    if (vpl <= 4) launch_pdl(embed_kernel<4>, grid, block, 0, st, a);
    else if (vpl <= 8) launch_pdl(embed_kernel<8>, grid, block, 0, st, a);
    else if (vpl <= 16) launch_pdl(embed_kernel<16>, grid, block, 0, st, a);
    else if (vpl <= 32) launch_pdl(embed_kernel<32>, grid, block, 0, st, a);
    else if (vpl <= 64) launch_pdl(embed_kernel<64>, grid, block, 0, st, a);
    else return cudaErrorInvalidValue;
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// search state
// ---------------------------------------------------------------------------
__global__ void search_init_kernel(InitArgs a) {
    pdl_grid_wait();
    int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < a.R) {
        a.tok[i] = a.bos;
        a.fin[i] = 0;
        a.cum[i] = (i % a.k == 0) ? 0.0f : -INFINITY;  // only beam 0 of a sentence starts live
        a.keys[i] = 0ull;
    }
    for (int j = i; j < a.R * a.T; j += gridDim.x * blockDim.x) {
        a.anc[j] = j / a.T;
        a.hist[j] = a.pad;
        a.parents[j] = 0;
    }
    if (i == 0) {
        *a.t_ptr = 0;
        *a.done = 0;
        a.ticket[0] = 0;
        a.ticket[1] = 0;
    }
}

cudaError_t launch_search_init(const InitArgs &a, cudaStream_t st) {
    int n = a.R * a.T;
    int blocks = (n + 255) / 256;
    if (blocks < 1) blocks = 1;
    if (blocks > 1024) blocks = 1024;
    launch_pdl(search_init_kernel, blocks, 256, 0, st, a);
    return cudaGetLastError();
}

// greedy: argmax key -> token; after EOS a sentence emits PAD
__global__ void __launch_bounds__(1024) greedy_update_kernel(GreedyArgs a) {
    pdl_grid_wait();
    if (*a.done) return;
    if (a.pending && !*a.pending) return;  // the cluster step applied it already
    const int t = *a.t_ptr;
    int fin_all = 1;
    for (int r = threadIdx.x; r < a.R; r += blockDim.x) {
        unsigned long long k = a.keys[r];
        a.keys[r] = 0ull;
        int y = (int)key_index(k);
        int f = a.fin[r];
        int out = f ? a.pad : y;
        a.hist[(size_t)t * a.R + r] = out;
        a.tok[r] = out;
        if (!f && y == a.eos) f = 1;
        a.fin[r] = f;
        fin_all &= f;
    }
    int all = __syncthreads_and(fin_all);
    if (threadIdx.x == 0) {
        if (all || t + 1 >= *a.tmax_ptr) *a.done = 1;
        *a.t_ptr = t + 1;
        if (a.pending) *a.pending = 0;
    }
}

cudaError_t launch_greedy_update(const GreedyArgs &a, cudaStream_t st) {
    int threads = a.R < 1024 ? ((a.R + 31) / 32) * 32 : 1024;
    launch_pdl(greedy_update_kernel, 1, threads, 0, st, a);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// beam search (width k <= 16)
// ---------------------------------------------------------------------------
constexpr int BEAM_MAX = 16;
constexpr int BR_THREADS = 256;

// insert key into the descending list lst[0..k) (keys are unique): the key is
// carried down the list, swapping with every smaller entry
template <int KM>
MNMT_DEV void topk_insert(unsigned long long (&lst)[KM], int k, unsigned long long key) {
#pragma unroll
    for (int i = 0; i < KM; i++) {
        if (i < k && key > lst[i]) {
            unsigned long long tmp = lst[i];
            lst[i] = key;
            key = tmp;
        }
    }
}

// rne(exp_own(x) 2^24) for x <= 0, the weight of one softmax term.  Below 2^23
// the rounding to an integer is done by adding 2^23 (whose ulp is 1) and
// reading the low bits; the few weights in [2^23, 2^24] (x within ln 2 of
// the maximum) are integers already.
MNMT_DEV int32_t softmax_weight_fast(float x) {
    const float w = __fmul_rn(exp_own(x), 16777216.0f);
    if (w < 0x1p23f) return (int32_t)(__float_as_uint(__fadd_rn(w, 0x1p23f)) - 0x4B000000u);
    return __float2int_rn(w);
}

// Block-wide selection of the n largest keys held in the threads' descending
// lists lst[0..KL): n rounds of a maximum over the list heads.  The keys land
// in sel[0..n) (0 where fewer exist); every thread must call it.
template <int KL, int NT>
__device__ void block_select(const unsigned long long (&lst)[KL], int n, unsigned long long *sel,
                             unsigned long long *s_key) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int head = 0;
    for (int i = 0; i < n; i++) {
        unsigned long long mine = 0ull;
#pragma unroll
        for (int h = 0; h < KL; h++)
            if (h == head) mine = lst[h];
        const unsigned long long w = warp_max_u64(mine);
        if (lane == 0) s_key[warp] = w;
        __syncthreads();
        unsigned long long best = s_key[0];
        for (int j = 1; j < NT / 32; j++) best = s_key[j] > best ? s_key[j] : best;
        if (mine == best && best != 0ull) head++;  // keys are unique
        if (threadIdx.x == 0) sel[i] = best;
        __syncthreads();
    }
}

// Insert key into a warp-distributed descending list (lane j < KC holds the
// j-th best key, 0 where empty; keys are unique); returns the logit of the
// list's last entry once the list is full (-inf before).
template <int KC>
MNMT_DEV float warp_list_insert(unsigned long long &wl, unsigned long long key, int lane, float thr) {
    const unsigned long long last = __shfl_sync(0xFFFFFFFFu, wl, KC - 1);
    if (key <= last) return thr;
    const int pos = __popc(__ballot_sync(0xFFFFFFFFu, lane < KC && wl > key));  // entries ranked above key
    const unsigned long long up = __shfl_up_sync(0xFFFFFFFFu, wl, 1);
    if (lane < KC) wl = lane < pos ? wl : (lane == pos ? key : up);
    const unsigned long long nl = __shfl_sync(0xFFFFFFFFu, wl, KC - 1);
    return nl != 0ull ? key_value(nl) : thr;
}

// One block per hypothesis row: the log-softmax of Sec. 3 / App. D's beam
// search (m = max, Z = sum of rne(e^(l - m) 2^24), lambda = ln Z - 24 ln 2,
// score = cum + ((l - m) - lambda)) and the k best (score, flat index) keys.
// The score is a non-decreasing function of the logit, so the k best lie
// among the logits ranked best by (logit desc, id asc): the pass that sums Z
// also keeps each warp's KC = KM + 4 best logits (a warp-wide threshold makes
// updates rare), and the k best scores are taken from the row's KC best
// logits.  That is exact unless the last of those candidates could still tie
// the k-th score (rounding can merge scores); such a row is scanned again in
// full.
// CAND = false skips the candidates and always scans the scores (fewer,
// simpler passes: better where a few rows leave the SMs short of warps).
template <int KM, int NT, bool CAND>
__global__ void __launch_bounds__(NT) beam_rows_kernel(BeamArgs a) {
    pdl_grid_wait();
    if (*a.done) return;
    constexpr int KC = KM + 4;
    static_assert(KC <= 32, "a warp holds the candidate list");
    constexpr int NW = NT / 32;
    const int r = blockIdx.x;
    const int k = a.k;
    const int V = a.V;
    const int lb = r % k;  // beam index within the sentence
    unsigned long long *out = a.cand + (size_t)r * k;
    __shared__ float s_m;
    __shared__ float s_lam;
    __shared__ int s_full;
    __shared__ long long s_z[NW];
    __shared__ float s_mx[NW];
    __shared__ unsigned long long s_key[NW];
    __shared__ unsigned long long s_wl[NW][KC];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (a.fin[r]) {
        // a finished hypothesis offers itself once, unchanged, with token PAD
        for (int i = threadIdx.x; i < k; i += NT)
            out[i] = i == 0 ? pack_key(a.cum[r], (uint32_t)(lb * V + a.pad)) : 0ull;
        return;
    }
    const float *l = a.logits + (size_t)r * V;
    const bool v4 = (V & 3) == 0 && (reinterpret_cast<uintptr_t>(l) & 15) == 0;
    const float4 *l4 = reinterpret_cast<const float4 *>(l);
    float mx = -INFINITY;
    if (v4) {
        for (int n = threadIdx.x; n < V / 4; n += NT) {
            const float4 v = l4[n];
            mx = fmaxf(mx, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)));
        }
    } else {
        for (int n = threadIdx.x; n < V; n += NT) mx = fmaxf(mx, l[n]);
    }
    mx = warp_max_f(mx);
    if (lane == 0) s_mx[warp] = mx;
    __syncthreads();
    if (threadIdx.x == 0) {
        float m = s_mx[0];
        for (int w = 1; w < NW; w++) m = fmaxf(m, s_mx[w]);
        s_m = m;
    }
    __syncthreads();
    const float m = s_m;
    // Z, and this warp's KC best (logit, id) keys
    long long z = 0;
    unsigned long long wl = 0ull;
    float thr = -INFINITY;  // warp-uniform
    // four logits per lane and step: their weights, then one warp vote on
    // whether any of them can enter the warp's list
    auto visit4 = [&](const float4 v, int n0) {
        const int32_t w4 = softmax_weight_fast(__fsub_rn(v.x, m)) + softmax_weight_fast(__fsub_rn(v.y, m)) +
                           softmax_weight_fast(__fsub_rn(v.z, m)) + softmax_weight_fast(__fsub_rn(v.w, m));
        z += w4;  // each weight <= 2^24
        unsigned msk = __ballot_sync(0xFFFFFFFFu, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)) >= thr);
        while (msk) {
            const int src = __ffs(msk) - 1;
            msk &= msk - 1;
            const int ns = __shfl_sync(0xFFFFFFFFu, n0, src);
            const float xs[4] = {__shfl_sync(0xFFFFFFFFu, v.x, src), __shfl_sync(0xFFFFFFFFu, v.y, src),
                                 __shfl_sync(0xFFFFFFFFu, v.z, src), __shfl_sync(0xFFFFFFFFu, v.w, src)};
#pragma unroll
            for (int e = 0; e < 4; e++)
                if (xs[e] >= thr) thr = warp_list_insert<KC>(wl, pack_key(xs[e], (uint32_t)(ns + e)), lane, thr);
        }
    };
    // every lane of a warp runs the same number of steps (the votes); logits
    // past the row end read as -inf (weight 0, ranked below every logit)
    const float NI = -INFINITY;
    if (!CAND) {
        if (v4) {
            for (int n = threadIdx.x; n < V / 4; n += NT) {
                const float4 v = l4[n];
                z += softmax_weight_fast(__fsub_rn(v.x, m)) + softmax_weight_fast(__fsub_rn(v.y, m)) +
                     softmax_weight_fast(__fsub_rn(v.z, m)) + softmax_weight_fast(__fsub_rn(v.w, m));
            }
        } else {
            for (int n = threadIdx.x; n < V; n += NT) z += softmax_weight_fast(__fsub_rn(l[n], m));
        }
    } else if (v4) {
        // four loads in flight per lane before the (branchy) visits
        const int n4 = V / 4;
        for (int base = warp * 32; base < n4; base += 4 * NT) {
            float4 v[4];
#pragma unroll
            for (int u = 0; u < 4; u++) {
                const int n = base + u * NT + lane;
                v[u] = n < n4 ? l4[n] : make_float4(NI, NI, NI, NI);
            }
#pragma unroll
            for (int u = 0; u < 4; u++) visit4(v[u], 4 * (base + u * NT + lane));
        }
    } else {
        for (int base = warp * 128; base < V; base += 4 * NT) {
            const int n = base + 4 * lane;
            visit4(make_float4(n < V ? l[n] : NI, n + 1 < V ? l[n + 1] : NI, n + 2 < V ? l[n + 2] : NI,
                               n + 3 < V ? l[n + 3] : NI),
                   n);
        }
    }
    z = warp_sum_ll(z);
    if (lane == 0) s_z[warp] = z;
    if (CAND && lane < KC) s_wl[warp][lane] = wl;
    __syncthreads();
    if (!CAND && threadIdx.x == 0) {
        long long Z = 0;
        for (int w = 0; w < NW; w++) Z += s_z[w];
        s_lam = __double2float_rn(__dadd_rn(log_own(__ll2double_rn(Z)), -0x1.0a2b23f3bab73p+4));
        s_full = 1;
    }
    if (CAND && warp == 0) {
        long long Z = 0;
        for (int w = 0; w < NW; w++) Z += s_z[w];
        // lambda = ln Z - 24 ln 2 (log of the normaliser of the 2^-24 weights)
        const float lam = __double2float_rn(__dadd_rn(log_own(__ll2double_rn(Z)), -0x1.0a2b23f3bab73p+4));
        // the row's KC best candidates: KC rounds of a maximum over the heads
        // of the warps' lists (lane w < NW walks list w)
        int head = 0;
        unsigned long long cand = 0ull;  // lane j ends with the j-th best
        for (int j = 0; j < KC; j++) {
            const unsigned long long mine = lane < NW && head < KC ? s_wl[lane][head] : 0ull;
            const unsigned long long best = warp_max_u64(mine);
            if (mine == best && best != 0ull) head++;
            if (lane == j) cand = best;
        }
        const int nc = V < KC ? V : KC;
        const float cum = a.cum[r];
        // final keys; lane KC-1 holds the lowest-ranked candidate
        float sc = 0.0f;
        unsigned long long fk = 0ull;
        if (lane < nc) {
            sc = __fadd_rn(cum, __fsub_rn(__fsub_rn(key_value(cand), m), lam));
            fk = pack_key(sc, (uint32_t)(lb * V) + key_index(cand));
        }
        const float sc_last = __shfl_sync(0xFFFFFFFFu, sc, nc - 1);
        // the k best final keys, best first
        unsigned long long kth = 0ull;
        for (int i = 0; i < k; i++) {
            const unsigned long long best = warp_max_u64(fk);
            if (fk == best) fk = 0ull;
            if (lane == i) kth = best;
        }
        // every other element scores <= sc_last; it cannot displace the k-th
        // key unless it can tie its score
        const unsigned long long kk = __shfl_sync(0xFFFFFFFFu, kth, k - 1);
        const bool exact = CAND && (nc == V || sc_last < key_value(kk));
        if (exact && lane < k) out[lane] = kth;
        if (lane == 0) {
            s_full = !exact;
            s_lam = lam;
        }
    }
    __syncthreads();
    if (!s_full) return;
    // full scan of the scores (rare: a tie at the candidate boundary)
    const float lam = s_lam;
    const float cum = a.cum[r];
    unsigned long long top[KM];
#pragma unroll
    for (int i = 0; i < KM; i++) top[i] = 0ull;
    for (int n = threadIdx.x; n < V; n += NT) {
        const float lp = __fsub_rn(__fsub_rn(l[n], m), lam);
        const float sc = __fadd_rn(cum, lp);
        topk_insert<KM>(top, k, pack_key(sc, (uint32_t)(lb * V + n)));
    }
    block_select<KM, NT>(top, k, out, s_key);
}

// per sentence: best k of the k*k row candidates; reorder state
__global__ void __launch_bounds__(256) beam_select_kernel(BeamArgs a) {
    pdl_grid_wait();
    if (*a.done) return;
    const int b = blockIdx.x;
    const int k = a.k, V = a.V, T = a.T;
    const int t = *a.t_ptr;
    __shared__ unsigned long long cand[BEAM_MAX * BEAM_MAX];
    __shared__ unsigned long long sel[BEAM_MAX];
    __shared__ int pfin[BEAM_MAX];
    __shared__ int s_all;
    extern __shared__ int anc_old[];  // [k][T]
    const int r0 = b * k;
    for (int i = threadIdx.x; i < k * k; i += blockDim.x) cand[i] = a.cand[(size_t)r0 * k + i];
    for (int i = threadIdx.x; i < k; i += blockDim.x) pfin[i] = a.fin[r0 + i];
    for (int i = threadIdx.x; i < k * t; i += blockDim.x) {
        int rr = i / t, j = i - rr * t;
        anc_old[rr * T + j] = a.anc[(size_t)(r0 + rr) * T + j];
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // k rounds of selection over k*k keys (unique keys, descending)
        for (int i = 0; i < k; i++) {
            unsigned long long best = 0ull;
            int bi = 0;
            for (int j = 0; j < k * k; j++)
                if (cand[j] > best) {
                    best = cand[j];
                    bi = j;
                }
            sel[i] = best;
            cand[bi] = 0ull;
        }
        int all = 1;
        for (int i = 0; i < k; i++) {
            uint32_t idx = key_index(sel[i]);
            int p = (int)(idx / (uint32_t)V), n = (int)(idx - (uint32_t)p * V);
            int f = pfin[p] || n == a.eos;
            all &= f;
        }
        s_all = all;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
        unsigned long long key = sel[i];
        uint32_t idx = key_index(key);
        int p = (int)(idx / (uint32_t)V), n = (int)(idx - (uint32_t)p * V);
        int r = r0 + i;
        a.cum[r] = key_value(key);
        a.fin[r] = pfin[p] || n == a.eos;
        a.tok[r] = n;
        a.hist[(size_t)t * (a.B * k) + r] = n;
        a.parents[(size_t)t * (a.B * k) + r] = p;
    }
    // ancestry: new row i takes parent p's positions 0..t-1 and p's own slot at t
    for (int x = threadIdx.x; x < k * (t + 1); x += blockDim.x) {
        int i = x / (t + 1), j = x - i * (t + 1);
        uint32_t idx = key_index(sel[i]);
        int p = (int)(idx / (uint32_t)V);
        a.anc[(size_t)(r0 + i) * T + j] = (j < t) ? anc_old[p * T + j] : r0 + p;
    }
    // the last block to finish decides whether every sentence is done
    __shared__ int s_last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (!s_all) atomicAdd(a.ticket + 1, 1);  // sentences still running
        int prev = atomicAdd(a.ticket, 1);
        s_last = prev == (int)gridDim.x - 1;
    }
    __syncthreads();
    if (s_last && threadIdx.x == 0) {
        __threadfence();
        int running = atomicAdd(a.ticket + 1, 0);
        if (running == 0 || t + 1 >= *a.tmax_ptr) *a.done = 1;
        a.ticket[0] = 0;
        a.ticket[1] = 0;
        *a.t_ptr = t + 1;
    }
}

cudaError_t launch_beam_step(const BeamArgs &a, cudaStream_t st) {
    if (a.k < 1 || a.k > BEAM_MAX) return cudaErrorInvalidValue;
    int R = a.B * a.k;
    // up to one row per SM: the plain scan (its simple loops keep more loads
    // in flight per warp); more rows: the candidate pass
    if (R <= device_sm_count()) {
        if (a.k <= 4) launch_pdl(beam_rows_kernel<4, BR_THREADS, false>, R, BR_THREADS, 0, st, a);
        else if (a.k <= 8) launch_pdl(beam_rows_kernel<8, BR_THREADS, false>, R, BR_THREADS, 0, st, a);
        else launch_pdl(beam_rows_kernel<16, BR_THREADS, false>, R, BR_THREADS, 0, st, a);
    } else {
        if (a.k <= 4) launch_pdl(beam_rows_kernel<4, BR_THREADS, true>, R, BR_THREADS, 0, st, a);
        else if (a.k <= 8) launch_pdl(beam_rows_kernel<8, BR_THREADS, true>, R, BR_THREADS, 0, st, a);
        else launch_pdl(beam_rows_kernel<16, BR_THREADS, true>, R, BR_THREADS, 0, st, a);
    }
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    size_t smem = (size_t)a.k * a.T * sizeof(int);
    launch_pdl(beam_select_kernel, a.B, 256, smem, st, a);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// final outputs: best hypothesis of each sentence (beam 0 after the last step),
// backtracked through the parent pointers
// ---------------------------------------------------------------------------
__global__ void finalize_kernel(FinalArgs a) {
    pdl_grid_wait();
    const int b = blockIdx.x;
    if (threadIdx.x != 0) return;
    const int steps = *a.t_ptr;
    const int R = a.B * a.k;
    int r = b * a.k;
    // walk back from the last step, writing tokens in reverse
    for (int t = steps - 1; t >= 0; t--) {
        a.out_ids[(size_t)b * a.max_len + t] = a.hist[(size_t)t * R + r];
        if (a.k > 1) r = b * a.k + a.parents[(size_t)t * R + r];
    }
    int n = steps;
    for (int t = 0; t < steps; t++)
        if (a.out_ids[(size_t)b * a.max_len + t] == a.eos) {
            n = t + 1;
            break;
        }
    for (int t = n; t < a.max_len; t++) a.out_ids[(size_t)b * a.max_len + t] = a.pad;
    a.out_lens[b] = n;
    a.out_scores[b] = a.k > 1 ? a.cum[b * a.k] : 0.0f;
}

// Opt the beam reorder kernel into the shared memory of its largest shape
// (k = 16 hypotheses x 1024 positions); once per process, before any capture.
cudaError_t rows_init() {
    return cudaFuncSetAttribute(beam_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                BEAM_MAX * 1024 * (int)sizeof(int));
}

cudaError_t launch_finalize(const FinalArgs &a, cudaStream_t st) {
    launch_pdl(finalize_kernel, a.B, 32, 0, st, a);
    return cudaGetLastError();
}

}  // namespace mnmt
