// linear_w4.cu -- quantised linear with row-wise 4-bit weights (Sec. 3.3: the
// low-bit weights are quantised row-wise; table "quantizing weights to lower
// bits", 4-8-8: 4-bit weights, 8-bit embedding and activations).
//
// A weight row holds K 4-bit codes packed two per byte in runs of 32 codes per
// 16 bytes: code j of a run in the low nibble of byte j (j < 16), code 16 + j
// in its high nibble.  Two row forms:
//   symmetric: stored code c = v + 8 for v in [-7, 7], W = s_n v;
//   min-max (App. B Eq. scale / Eq. quant): stored code u in [0, 15],
//     W = s_n u + r_n with r_n the row minimum.
// With A_u = sum_k a_k c_nk and A_1 = sum_k a_k (exact int32):
//   symmetric: acc = A_u - 8 A_1 = sum a_k v_nk, then the int8 epilogue
//              y = fl(fl(acc fl(s_x s_n)) + b_n);
//   min-max:   y = fl(fl(fl(A_u fl(s_x s_n)) + fl(A_1 fl(s_x r_n))) + b_n).
//
// linear_w4_small streams every weight row once as packed nibbles (half the
// bytes of the int8 GEMV); up to 16 activation rows sit in shared memory with
// their code sums A_1; a 16-byte weight load unpacks into two 16-code int8
// vectors (mask / shift, the codes are non-negative) for dp4a.
#include "common.cuh"
#include "epilogue.cuh"
#include "internal.h"

namespace mnmt {

constexpr int W4_THREADS = 256;

// y of output n from the exact sums A_u (acc) and A_1 (a1)
MNMT_DEV float w4_y(const Epi &e, int n, int acc, int a1, const float *__restrict__ m_w) {
    if (!m_w) return dequant_bias(acc - 8 * a1, e.s_x, e.s_w[n], e.bias[n]);
    const float t = __fmul_rn(__int2float_rn(acc), __fmul_rn(e.s_x, e.s_w[n]));
    const float o = __fmul_rn(__int2float_rn(a1), __fmul_rn(e.s_x, m_w[n]));
    return __fadd_rn(__fadd_rn(t, o), e.bias[n]);
}

// MT: activation rows held; LPC: lanes per weight row (K/32 runs spread over
// LPC lanes); U: weight rows in flight per lane group.
template <int MT, int LPC, int U>
__global__ void __launch_bounds__(W4_THREADS) linear_w4_small(const int8_t *__restrict__ A, int lda,
                                                             const uint8_t *__restrict__ Wp,
                                                             const float *__restrict__ m_w, int M, int N, int K,
                                                             Epi e) {
    pdl_grid_wait();
    if (e.skip && *e.skip) return;
    extern __shared__ int4 smA[];  // [MT][K/16]
    __shared__ int s_a1[MT];
    const int kc = K >> 4, kr = K >> 5;  // 16-code chunks of a row of A, 32-code runs of a weight row
    const int m0 = blockIdx.y * MT;
    A += (size_t)m0 * lda;
    M -= m0;
    for (int i = threadIdx.x; i < MT * kc; i += W4_THREADS) {
        const int m = i / kc, c = i - m * kc;
        smA[i] = (m < M) ? reinterpret_cast<const int4 *>(A + (size_t)m * lda)[c] : make_int4(0, 0, 0, 0);
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int m = warp; m < MT; m += W4_THREADS / 32) {
        int s = 0;
        const int4 ones = make_int4(0x01010101, 0x01010101, 0x01010101, 0x01010101);
        for (int c = lane; c < kc; c += 32) s = dot16(smA[m * kc + c], ones, s);
        s = warp_sum_i(s);
        if (lane == 0) s_a1[m] = s;
    }
    __syncthreads();
    const int t = e.t_ptr ? *e.t_ptr : 0;
    constexpr int GPW = 32 / LPC;
    constexpr int CPB = (W4_THREADS / 32) * GPW * U;
    const int grp = lane / LPC, sl = lane % LPC;
    const bool argmax = e.mode == EPI_ARGMAX;
    const size_t row_bytes = (size_t)K >> 1;
    unsigned long long best[MT];
#pragma unroll
    for (int m = 0; m < MT; m++) best[m] = 0ull;

    for (int base = blockIdx.x * CPB; base < N; base += gridDim.x * CPB) {
        int acc[U][MT];
#pragma unroll
        for (int u = 0; u < U; u++)
#pragma unroll
            for (int m = 0; m < MT; m++) acc[u][m] = 0;
        for (int c0 = 0; c0 < kr; c0 += LPC) {
            const int c = c0 + sl;
            int4 w[U];
#pragma unroll
            for (int u = 0; u < U; u++) {
                const int n = base + (u * (W4_THREADS / 32) + warp) * GPW + grp;
                w[u] = (n < N && c < kr) ? __ldg(reinterpret_cast<const int4 *>(Wp + (size_t)n * row_bytes) + c)
                                         : make_int4(0, 0, 0, 0);
            }
            if (c < kr) {
                int4 lo[U], hi[U];
#pragma unroll
                for (int u = 0; u < U; u++) {
                    lo[u] = make_int4(w[u].x & 0x0F0F0F0F, w[u].y & 0x0F0F0F0F, w[u].z & 0x0F0F0F0F,
                                      w[u].w & 0x0F0F0F0F);
                    hi[u] = make_int4((w[u].x >> 4) & 0x0F0F0F0F, (w[u].y >> 4) & 0x0F0F0F0F,
                                      (w[u].z >> 4) & 0x0F0F0F0F, (w[u].w >> 4) & 0x0F0F0F0F);
                }
#pragma unroll
                for (int m = 0; m < MT; m++) {
                    const int4 a0 = smA[m * kc + 2 * c], a1 = smA[m * kc + 2 * c + 1];
#pragma unroll
                    for (int u = 0; u < U; u++) acc[u][m] = dot16(a1, hi[u], dot16(a0, lo[u], acc[u][m]));
                }
            }
        }
#pragma unroll
        for (int u = 0; u < U; u++) {
#pragma unroll
            for (int m = 0; m < MT; m++) {
#pragma unroll
                for (int o = LPC / 2; o > 0; o >>= 1) acc[u][m] += __shfl_xor_sync(0xFFFFFFFFu, acc[u][m], o);
            }
            const int n = base + (u * (W4_THREADS / 32) + warp) * GPW + grp;
            if (sl == 0 && n < N) {
                if (argmax) {
#pragma unroll
                    for (int m = 0; m < MT; m++) {
                        if (m < M) {
                            const unsigned long long k = pack_key(w4_y(e, n, acc[u][m], s_a1[m], m_w), (uint32_t)n);
                            best[m] = k > best[m] ? k : best[m];
                        }
                    }
                } else if (e.mode == EPI_RESID) {
                    // every residual load first: the stores may alias them
                    float r[MT];
#pragma unroll
                    for (int m = 0; m < MT; m++) r[m] = m < M ? e.f32[(size_t)(m0 + m) * e.ldf + n] : 0.0f;
#pragma unroll
                    for (int m = 0; m < MT; m++)
                        if (m < M)
                            e.f32[(size_t)(m0 + m) * e.ldf + n] =
                                __fadd_rn(__fmul_rn(e.gamma, r[m]), w4_y(e, n, acc[u][m], s_a1[m], m_w));
                } else {
#pragma unroll
                    for (int m = 0; m < MT; m++)
                        if (m < M) epi_store_y(e, m0 + m, n, w4_y(e, n, acc[u][m], s_a1[m], m_w), t);
                }
            }
        }
    }
    if (argmax) {
        __shared__ unsigned long long red[W4_THREADS / 32][MT];
#pragma unroll
        for (int m = 0; m < MT; m++) {
            const unsigned long long v = warp_max_u64(best[m]);
            if (lane == 0) red[warp][m] = v;
        }
        __syncthreads();
        if (threadIdx.x < MT && (int)threadIdx.x < M) {
            unsigned long long v = 0;
            for (int w = 0; w < W4_THREADS / 32; w++) v = red[w][threadIdx.x] > v ? red[w][threadIdx.x] : v;
            atomicMax(e.keys + m0 + threadIdx.x, v);
        }
    }
}

template <int MT, int LPC>
static cudaError_t launch_w4_t(const int8_t *A, int lda, const uint8_t *Wp, const float *m_w, int M, int N, int K,
                               const Epi &e, cudaStream_t st) {
    constexpr int U = 2;
    constexpr int CPB = (W4_THREADS / 32) * (32 / LPC) * U;
    int blocks = (N + CPB - 1) / CPB;
    const int cap = 4 * device_sm_count();
    if (blocks > cap) blocks = cap;
    const dim3 grid(blocks, (M + MT - 1) / MT);
    launch_pdl(linear_w4_small<MT, LPC, U>, grid, W4_THREADS, (size_t)MT * K, st, A, lda, Wp, m_w, M, N, K, e);
    return cudaGetLastError();
}

template <int MT>
static cudaError_t launch_w4_m(const int8_t *A, int lda, const uint8_t *Wp, const float *m_w, int M, int N, int K,
                               const Epi &e, cudaStream_t st) {
    const int kr = K / 32;
    if (kr >= 32) return launch_w4_t<MT, 32>(A, lda, Wp, m_w, M, N, K, e, st);
    if (kr >= 16) return launch_w4_t<MT, 16>(A, lda, Wp, m_w, M, N, K, e, st);
    if (kr >= 8) return launch_w4_t<MT, 8>(A, lda, Wp, m_w, M, N, K, e, st);
    return launch_w4_t<MT, 4>(A, lda, Wp, m_w, M, N, K, e, st);
}

cudaError_t launch_linear_w4(const int8_t *A, int lda, const uint8_t *Wp, const float *m_w, int M, int N, int K,
                             const Epi &e, cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (K < 32 || K % 32 || K > 3072 || lda % 16) return cudaErrorInvalidValue;
    if (M == 1) return launch_w4_m<1>(A, lda, Wp, m_w, M, N, K, e, st);
    if (M <= 2) return launch_w4_m<2>(A, lda, Wp, m_w, M, N, K, e, st);
    if (M <= 4) return launch_w4_m<4>(A, lda, Wp, m_w, M, N, K, e, st);
    if (M <= 8) return launch_w4_m<8>(A, lda, Wp, m_w, M, N, K, e, st);
    return launch_w4_m<16>(A, lda, Wp, m_w, M, N, K, e, st);  // chunks of 16 rows over the grid's y
}

// symmetric rows unpacked to int8 codes v = c - 8 (the int8 kernels' operand)
__global__ void unpack_w4_sym(const uint8_t *__restrict__ Wp, size_t runs, int8_t *__restrict__ out) {
    const size_t g = (size_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (g >= runs) return;
    const int4 w = reinterpret_cast<const int4 *>(Wp)[g];
    const uint32_t x[4] = {(uint32_t)w.x, (uint32_t)w.y, (uint32_t)w.z, (uint32_t)w.w};
    uint32_t lo[4], hi[4];
#pragma unroll
    for (int i = 0; i < 4; i++) {
        lo[i] = __vsub4(x[i] & 0x0F0F0F0Fu, 0x08080808u);
        hi[i] = __vsub4((x[i] >> 4) & 0x0F0F0F0Fu, 0x08080808u);
    }
    int4 *o = reinterpret_cast<int4 *>(out + g * 32);
    o[0] = make_int4((int)lo[0], (int)lo[1], (int)lo[2], (int)lo[3]);
    o[1] = make_int4((int)hi[0], (int)hi[1], (int)hi[2], (int)hi[3]);
}

cudaError_t launch_unpack_w4_sym(const uint8_t *Wp, size_t codes, int8_t *out, cudaStream_t st) {
    if (codes % 32) return cudaErrorInvalidValue;
    const size_t runs = codes / 32;
    if (runs == 0) return cudaSuccess;
    unpack_w4_sym<<<(unsigned)((runs + 255) / 256), 256, 0, st>>>(Wp, runs, out);
    return cudaGetLastError();
}

}  // namespace mnmt
