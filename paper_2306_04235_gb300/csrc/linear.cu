// linear.cu -- quantised linear layers of the INT8 encoder-decoder (Sec. 3.3,
// Fig. 5; Eq. 3): int8 x int8 -> exact int32 accumulation, then a fused
// epilogue (dequantise with the per-channel weight scale, full-precision bias,
// then requantise / ReLU+requantise / gamma-residual / fp32 / K-V cache write /
// greedy argmax).
//
// Two kernels:
//   linear_smallm  M <= 16 rows, or up to 64 rows of a narrow layer, in chunks
//                  of <= 16 rows per grid row (batch-1 encoder, batch-1 and
//                  small-batch decode): every weight
//                  row is streamed once with 16-byte coalesced loads, the M
//                  activation rows sit in shared memory, products use dp4a and
//                  a lane group's partial sums meet by warp shuffles.  Bound by
//                  weight bytes (HBM or L2).
//   linear_mma     other M > 16: CTA tiles of the int8 GEMM on the warp-level s8
//                  tensor-core instruction (mma.sync m16n8k32, exact int32
//                  accumulate), cp.async multi-stage pipeline with XOR-swizzled
//                  shared memory and ldmatrix fragment loads.  sm_103a has no
//                  int8 form of tcgen05.mma, so this is the exact int8 tensor path.
#include "common.cuh"
#include "epilogue.cuh"
#include "internal.h"

namespace mnmt {

// ---------------------------------------------------------------------------
// small-M path
// ---------------------------------------------------------------------------
constexpr int SM_THREADS = 256;
constexpr int SMALL_CHUNKED_MAX_M = 64;

// MT: rows held (>= M); LPC: lanes per weight row (K/16 chunks spread over
// LPC lanes); U: weight rows in flight per lane group.
template <int MT, int LPC, int U>
__global__ void __launch_bounds__(SM_THREADS) linear_smallm(const int8_t *__restrict__ A, int lda,
                                                           const int8_t *__restrict__ W, int M, int N,
                                                           int K, Epi e) {
    pdl_grid_wait();
    if (e.skip && *e.skip) return;
    extern __shared__ int4 smA[];  // [MT][K/16]
    const int kc = K >> 4;
    // blockIdx.y selects the chunk of MT rows this block computes
    const int m0 = blockIdx.y * MT;
    A += (size_t)m0 * lda;
    M -= m0;
    for (int i = threadIdx.x; i < MT * kc; i += SM_THREADS) {
        int m = i / kc, c = i - m * kc;
        smA[i] = (m < M) ? reinterpret_cast<const int4 *>(A + (size_t)m * lda)[c] : make_int4(0, 0, 0, 0);
    }
    __syncthreads();
    const int t = e.t_ptr ? *e.t_ptr : 0;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int GPW = 32 / LPC;              // lane groups per warp
    constexpr int CPB = (SM_THREADS / 32) * GPW * U;  // columns per block pass
    const int grp = lane / LPC, sl = lane % LPC;
    const bool argmax = e.mode == EPI_ARGMAX;
    unsigned long long best[MT];
#pragma unroll
    for (int m = 0; m < MT; m++) best[m] = 0ull;

    for (int base = blockIdx.x * CPB; base < N; base += gridDim.x * CPB) {
        int acc[U][MT];
#pragma unroll
        for (int u = 0; u < U; u++)
#pragma unroll
            for (int m = 0; m < MT; m++) acc[u][m] = 0;
        // column of (warp, group, u): base + (u * 8 + warp) * GPW + grp
        for (int c0 = 0; c0 < kc; c0 += LPC) {
            int c = c0 + sl;
            int4 w[U];
#pragma unroll
            for (int u = 0; u < U; u++) {
                int n = base + (u * (SM_THREADS / 32) + warp) * GPW + grp;
                w[u] = (n < N && c < kc) ? __ldg(reinterpret_cast<const int4 *>(W + (size_t)n * K) + c)
                                         : make_int4(0, 0, 0, 0);
            }
            if (c < kc) {
#pragma unroll
                for (int m = 0; m < MT; m++) {
                    int4 a = smA[m * kc + c];
#pragma unroll
                    for (int u = 0; u < U; u++) acc[u][m] = dot16(a, w[u], acc[u][m]);
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
            int n = base + (u * (SM_THREADS / 32) + warp) * GPW + grp;
            if (sl == 0 && n < N) {
                if (argmax) {
#pragma unroll
                    for (int m = 0; m < MT; m++) {
                        if (m < M) {
                            float y = dequant_bias(acc[u][m], e.s_x, e.s_w[n], e.bias[n]);
                            unsigned long long k = pack_key(y, (uint32_t)n);
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
                                __fadd_rn(__fmul_rn(e.gamma, r[m]),
                                          dequant_bias(acc[u][m], e.s_x, e.s_w[n], e.bias[n]));
                } else {
#pragma unroll
                    for (int m = 0; m < MT; m++)
                        if (m < M) epi_store(e, m0 + m, n, acc[u][m], t);
                }
            }
        }
    }
    if (argmax) {
        __shared__ unsigned long long red[SM_THREADS / 32][MT];
#pragma unroll
        for (int m = 0; m < MT; m++) {
            unsigned long long v = warp_max_u64(best[m]);
            if (lane == 0) red[warp][m] = v;
        }
        __syncthreads();
        if (threadIdx.x < MT && (int)threadIdx.x < M) {
            unsigned long long v = 0;
            for (int w = 0; w < SM_THREADS / 32; w++) v = red[w][threadIdx.x] > v ? red[w][threadIdx.x] : v;
            atomicMax(e.keys + m0 + threadIdx.x, v);
        }
    }
}

// ---------------------------------------------------------------------------
// tensor-core path (mma.sync s8)
// ---------------------------------------------------------------------------
MNMT_DEV uint32_t smem_u32(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

MNMT_DEV void cp_async16(uint32_t dst, const void *src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(dst), "l"(src), "r"(src_bytes));
}
MNMT_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::); }
template <int N>
MNMT_DEV void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;\n" ::"n"(N));
}
MNMT_DEV void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
MNMT_DEV void mma_s8(int (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};\n"
        : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 64-byte shared rows, 16-byte chunks XOR-swizzled by (row / 2) % 4 so that the
// 8 rows of an ldmatrix phase hit 8 distinct bank groups.
MNMT_DEV int swz(int row, int chunk) { return row * 64 + ((chunk ^ ((row >> 1) & 3)) << 4); }

template <int BM, int BN, int WARPS_M, int WARPS_N, int STAGES>
__global__ void __launch_bounds__(WARPS_M *WARPS_N * 32)
    linear_mma(const int8_t *__restrict__ A, int lda, const int8_t *__restrict__ W, int M, int N, int K,
               Epi e) {
    constexpr int BK = 64;
    constexpr int NT = WARPS_M * WARPS_N * 32;
    constexpr int WTM = BM / WARPS_M, WTN = BN / WARPS_N;
    constexpr int MI = WTM / 16, NI = WTN / 8;
    static_assert(NI % 2 == 0, "B fragments are loaded two n8 tiles at a time");
    pdl_grid_wait();
    if (e.skip && *e.skip) return;
    extern __shared__ __align__(128) uint8_t smem[];
    uint8_t *sA = smem;
    uint8_t *sB = smem + STAGES * BM * BK;
    const int bm = blockIdx.y * BM, bn = blockIdx.x * BN;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wm = warp / WARPS_N, wn = warp % WARPS_N;
    const int ktiles = K / BK;

    int acc[MI][NI][4];
#pragma unroll
    for (int i = 0; i < MI; i++)
#pragma unroll
        for (int j = 0; j < NI; j++)
#pragma unroll
            for (int q = 0; q < 4; q++) acc[i][j][q] = 0;

    auto load_stage = [&](int stage, int kt) {
        const int k0 = kt * BK;
        uint8_t *a_s = sA + stage * BM * BK;
        uint8_t *b_s = sB + stage * BN * BK;
#pragma unroll
        for (int i = threadIdx.x; i < BM * 4; i += NT) {
            int row = i >> 2, ch = i & 3;
            int g = bm + row;
            const int8_t *src = A + (size_t)(g < M ? g : M - 1) * lda + k0 + ch * 16;
            cp_async16(smem_u32(a_s + swz(row, ch)), src, g < M ? 16 : 0);
        }
#pragma unroll
        for (int i = threadIdx.x; i < BN * 4; i += NT) {
            int row = i >> 2, ch = i & 3;
            int g = bn + row;
            const int8_t *src = W + (size_t)(g < N ? g : N - 1) * K + k0 + ch * 16;
            cp_async16(smem_u32(b_s + swz(row, ch)), src, g < N ? 16 : 0);
        }
    };

#pragma unroll
    for (int s = 0; s < STAGES - 1; s++) {
        if (s < ktiles) load_stage(s, s);
        cp_async_commit();
    }
    for (int kt = 0; kt < ktiles; kt++) {
        cp_async_wait<STAGES - 2>();
        __syncthreads();
        {
            int nk = kt + STAGES - 1;
            if (nk < ktiles) load_stage(nk % STAGES, nk);
            cp_async_commit();
        }
        const uint8_t *a_s = sA + (kt % STAGES) * BM * BK;
        const uint8_t *b_s = sB + (kt % STAGES) * BN * BK;
#pragma unroll
        for (int kk = 0; kk < 2; kk++) {
            uint32_t af[MI][4];
            uint32_t bf[NI][2];
            const int j = lane >> 3, i8 = lane & 7;
#pragma unroll
            for (int mi = 0; mi < MI; mi++) {
                int row = wm * WTM + mi * 16 + (j & 1) * 8 + i8;
                ldmatrix_x4(af[mi], smem_u32(a_s + swz(row, kk * 2 + (j >> 1))));
            }
#pragma unroll
            for (int nj = 0; nj < NI / 2; nj++) {
                int row = wn * WTN + nj * 16 + (j >> 1) * 8 + i8;
                uint32_t r[4];
                ldmatrix_x4(r, smem_u32(b_s + swz(row, kk * 2 + (j & 1))));
                bf[2 * nj][0] = r[0];
                bf[2 * nj][1] = r[1];
                bf[2 * nj + 1][0] = r[2];
                bf[2 * nj + 1][1] = r[3];
            }
#pragma unroll
            for (int mi = 0; mi < MI; mi++)
#pragma unroll
                for (int ni = 0; ni < NI; ni++) mma_s8(acc[mi][ni], af[mi], bf[ni][0], bf[ni][1]);
        }
    }
    cp_async_wait<0>();

    const int t = e.t_ptr ? *e.t_ptr : 0;
    if (e.mode == EPI_ARGMAX) {
        // per row: max key over this thread's columns, then over the 4 lanes of a quad
#pragma unroll
        for (int mi = 0; mi < MI; mi++) {
#pragma unroll
            for (int hr = 0; hr < 2; hr++) {
                int row = bm + wm * WTM + mi * 16 + (lane >> 2) + hr * 8;
                unsigned long long best = 0ull;
#pragma unroll
                for (int ni = 0; ni < NI; ni++) {
#pragma unroll
                    for (int q = 0; q < 2; q++) {
                        int col = bn + wn * WTN + ni * 8 + (lane & 3) * 2 + q;
                        if (row < M && col < N) {
                            float y = dequant_bias(acc[mi][ni][hr * 2 + q], e.s_x, e.s_w[col], e.bias[col]);
                            unsigned long long k = pack_key(y, (uint32_t)col);
                            best = k > best ? k : best;
                        }
                    }
                }
#pragma unroll
                for (int o = 1; o < 4; o <<= 1) {
                    unsigned long long w2 = __shfl_xor_sync(0xFFFFFFFFu, best, o);
                    best = w2 > best ? w2 : best;
                }
                if ((lane & 3) == 0 && row < M) atomicMax(e.keys + row, best);
            }
        }
        return;
    }
    if (e.mode == EPI_RESID) {
        // every residual load first: the stores may alias them
        float r[MI][NI][4];
#pragma unroll
        for (int mi = 0; mi < MI; mi++)
#pragma unroll
            for (int ni = 0; ni < NI; ni++)
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    int row = bm + wm * WTM + mi * 16 + (lane >> 2) + (q >> 1) * 8;
                    int col = bn + wn * WTN + ni * 8 + (lane & 3) * 2 + (q & 1);
                    r[mi][ni][q] = (row < M && col < N) ? e.f32[(size_t)row * e.ldf + col] : 0.0f;
                }
#pragma unroll
        for (int mi = 0; mi < MI; mi++)
#pragma unroll
            for (int ni = 0; ni < NI; ni++)
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    int row = bm + wm * WTM + mi * 16 + (lane >> 2) + (q >> 1) * 8;
                    int col = bn + wn * WTN + ni * 8 + (lane & 3) * 2 + (q & 1);
                    if (row < M && col < N)
                        e.f32[(size_t)row * e.ldf + col] =
                            __fadd_rn(__fmul_rn(e.gamma, r[mi][ni][q]),
                                      dequant_bias(acc[mi][ni][q], e.s_x, e.s_w[col], e.bias[col]));
                }
        return;
    }
#pragma unroll
    for (int mi = 0; mi < MI; mi++)
#pragma unroll
        for (int ni = 0; ni < NI; ni++)
#pragma unroll
            for (int q = 0; q < 4; q++) {
                int row = bm + wm * WTM + mi * 16 + (lane >> 2) + (q >> 1) * 8;
                int col = bn + wn * WTN + ni * 8 + (lane & 3) * 2 + (q & 1);
                if (row < M && col < N) epi_store(e, row, col, acc[mi][ni][q], t);
            }
}

// ---------------------------------------------------------------------------
// dispatch
// ---------------------------------------------------------------------------
template <int BM, int BN, int WM, int WN, int STAGES>
static cudaError_t mma_attr() {
    return cudaFuncSetAttribute(linear_mma<BM, BN, WM, WN, STAGES>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                STAGES * (BM + BN) * 64);
}

// Opt the tensor-core kernels into their shared memory (once per process,
// before any launch or stream capture).
cudaError_t linear_init() {
    cudaError_t err = mma_attr<128, 128, 2, 4, 4>();
    if (err == cudaSuccess) err = mma_attr<64, 64, 2, 2, 4>();
    return err;
}

template <int MT>
static cudaError_t launch_small(const int8_t *A, int lda, const int8_t *W, int M, int N, int K, const Epi &e,
                                cudaStream_t st) {
    const int kc = K / 16;
    const int chunks = (M + MT - 1) / MT;  // row chunks of MT, one per grid row
    size_t smem = (size_t)MT * kc * 16;
    int lpc = kc >= 32 ? 32 : (kc >= 16 ? 16 : 8);
    constexpr int U = 2;
    int cpb = (SM_THREADS / 32) * (32 / lpc) * U;
    int blocks = (N + cpb - 1) / cpb;
    if (blocks > 4 * 152) blocks = 4 * 152;
    if (smem > 48 * 1024) return cudaErrorInvalidValue;  // K <= 3072 at M <= 16
    const dim3 grid(blocks, chunks);
    if (lpc == 32) {
        launch_pdl(linear_smallm<MT, 32, U>, grid, SM_THREADS, smem, st, A, lda, W, M, N, K, e);
    } else if (lpc == 16) {
        launch_pdl(linear_smallm<MT, 16, U>, grid, SM_THREADS, smem, st, A, lda, W, M, N, K, e);
    } else {
        launch_pdl(linear_smallm<MT, 8, U>, grid, SM_THREADS, smem, st, A, lda, W, M, N, K, e);
    }
    return cudaGetLastError();
}

template <int BM, int BN, int WM, int WN, int STAGES>
static cudaError_t launch_mma(const int8_t *A, int lda, const int8_t *W, int M, int N, int K, const Epi &e,
                              cudaStream_t st) {
    auto k = linear_mma<BM, BN, WM, WN, STAGES>;
    size_t smem = (size_t)STAGES * (BM + BN) * 64;
    dim3 grid((N + BN - 1) / BN, (M + BM - 1) / BM);
    launch_pdl(k, grid, WM * WN * 32, smem, st, A, lda, W, M, N, K, e);
    return cudaGetLastError();
}

cudaError_t launch_linear(const int8_t *A, int lda, const int8_t *W, int M, int N, int K, const Epi &e,
                          cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (M <= 16) {
        if (M == 1) return launch_small<1>(A, lda, W, M, N, K, e, st);
        if (M <= 2) return launch_small<2>(A, lda, W, M, N, K, e, st);
        if (M <= 4) return launch_small<4>(A, lda, W, M, N, K, e, st);
        if (M <= 8) return launch_small<8>(A, lda, W, M, N, K, e, st);
        return launch_small<16>(A, lda, W, M, N, K, e, st);
    }
    // up to 64 rows over few output tiles (narrow N): chunks of 16 rows over
    // the grid's y dimension spread the work over more blocks than the IMMA
    // tiling would (the weights are re-read per chunk, from L2)
    const long tiles64 = (long)((M + 63) / 64) * ((N + 63) / 64);
    if (M <= SMALL_CHUNKED_MAX_M && K <= 2048 && tiles64 < 8) return launch_small<16>(A, lda, W, M, N, K, e, st);
    long tiles_big = (long)((M + 127) / 128) * ((N + 127) / 128);
    if (tiles_big >= 152) return launch_mma<128, 128, 2, 4, 4>(A, lda, W, M, N, K, e, st);
    return launch_mma<64, 64, 2, 2, 4>(A, lda, W, M, N, K, e, st);
}

}  // namespace mnmt
