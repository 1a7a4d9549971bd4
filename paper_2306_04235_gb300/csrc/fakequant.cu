// fakequant.cu -- fake quantisation for quantisation-aware training (App. B
// "PTQ and QAT": the quantiser of Eq. quant inserted into the float model;
// besides the weights, its scale s is learnable).
//
//   symmetric, n bits: q = clamp(rne(fl(x fl(1/s))), -(2^(n-1)-1), 2^(n-1)-1), y = fl(q s)
//   min-max,   n bits: q = clamp(rne(fl(fl(x - r) fl(1/s))), 0, 2^n - 1),       y = fl(fl(q s) + r)
// Backward: straight-through for x, and the scale / offset gradients of the
// same expression with the rounding held fixed: with t the unrounded code and
// in = (qmin <= t <= qmax): dy/dx = in, dy/ds = in ? q - t : q, dy/dr = !in.
// The two scalar gradients are sums over the whole tensor, accumulated in
// fp64 (per-block partials combined with atomicAdd).
//
// The QAT forward of a linear quantises a float input per tensor (8-bit) and a
// float weight per row (learnable row scales), then runs the quantised linear
// of the codes -- the product X_q W_q^T is exact, so the result is that of the
// inference kernels on the same codes.
#include "common.cuh"
#include "internal.h"

namespace mnmt {

struct FqRange {
    float qmin, qmax;
};

MNMT_DEV FqRange fq_range(int bits, int minmax) {
    if (minmax) return FqRange{0.0f, (float)((1 << bits) - 1)};
    const float m = (float)((1 << (bits - 1)) - 1);
    return FqRange{-m, m};
}

MNMT_DEV float fq_code(float x, float inv, float r, int minmax, FqRange rg, float *t_out) {
    const float t = minmax ? __fmul_rn(__fsub_rn(x, r), inv) : __fmul_rn(x, inv);
    if (t_out) *t_out = t;
    return fminf(fmaxf(rintf(t), rg.qmin), rg.qmax);
}

template <typename CodeT>
__global__ void fq_forward_kernel(const float *__restrict__ x, size_t n, float s, float r, int bits, int minmax,
                                  float *__restrict__ y, CodeT *__restrict__ codes) {
    const float inv = __fdiv_rn(1.0f, s);
    const FqRange rg = fq_range(bits, minmax);
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        const float q = fq_code(x[i], inv, r, minmax, rg, nullptr);
        if (codes) codes[i] = (CodeT)(int)q;
        if (y) {
            const float v = __fmul_rn(q, s);
            y[i] = minmax ? __fadd_rn(v, r) : v;
        }
    }
}

__global__ void fq_backward_kernel(const float *__restrict__ x, const float *__restrict__ g, size_t n, float s,
                                   float r, int bits, int minmax, float *__restrict__ gx, double *gs, double *gr) {
    const float inv = __fdiv_rn(1.0f, s);
    const FqRange rg = fq_range(bits, minmax);
    double as = 0.0, ar = 0.0;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (size_t)gridDim.x * blockDim.x) {
        float t;
        const float q = fq_code(x[i], inv, r, minmax, rg, &t);
        const bool in = t >= rg.qmin && t <= rg.qmax;
        const float gi = g[i];
        gx[i] = in ? gi : 0.0f;
        as += (double)gi * (in ? (double)q - (double)t : (double)q);
        if (!in) ar += (double)gi;
    }
    // block reduction in fp64, then one atomic per block
    __shared__ double red_s[32], red_r[32];
    for (int o = 16; o > 0; o >>= 1) {
        as += __shfl_xor_sync(0xFFFFFFFFu, as, o);
        ar += __shfl_xor_sync(0xFFFFFFFFu, ar, o);
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        red_s[warp] = as;
        red_r[warp] = ar;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        double ts = 0.0, tr = 0.0;
        for (int w = 0; w < (int)(blockDim.x >> 5); w++) {
            ts += red_s[w];
            tr += red_r[w];
        }
        atomicAdd(gs, ts);
        if (gr) atomicAdd(gr, minmax ? tr : 0.0);
    }
}

// per-row symmetric codes of a float weight matrix W [N][K] at row scales s_w
__global__ void fq_rows_kernel(const float *__restrict__ W, int N, int K, const float *__restrict__ s_w, int bits,
                               int8_t *__restrict__ codes) {
    const FqRange rg = fq_range(bits, 0);
    const size_t total = (size_t)N * K;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (size_t)gridDim.x * blockDim.x) {
        const int n = (int)(i / (size_t)K);
        const float inv = __fdiv_rn(1.0f, s_w[n]);
        codes[i] = (int8_t)(int)fq_code(W[i], inv, 0.0f, 0, rg, nullptr);
    }
}

static int fq_grid(size_t n) {
    size_t b = (n + 255) / 256;
    const size_t cap = (size_t)8 * device_sm_count();
    return (int)(b < 1 ? 1 : (b > cap ? cap : b));
}

cudaError_t launch_fake_quant(const float *x, size_t n, float s, float r, int bits, int minmax, float *y,
                              int32_t *codes, cudaStream_t st) {
    if (n == 0) return cudaSuccess;
    fq_forward_kernel<int32_t><<<fq_grid(n), 256, 0, st>>>(x, n, s, r, bits, minmax, y, codes);
    return cudaGetLastError();
}

cudaError_t launch_fake_quant_backward(const float *x, const float *g, size_t n, float s, float r, int bits,
                                       int minmax, float *gx, double *gs, double *gr, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(gs, 0, sizeof(double), st);
    if (e == cudaSuccess && gr) e = cudaMemsetAsync(gr, 0, sizeof(double), st);
    if (e != cudaSuccess || n == 0) return e;
    fq_backward_kernel<<<fq_grid(n), 256, 0, st>>>(x, g, n, s, r, bits, minmax, gx, gs, gr);
    return cudaGetLastError();
}

cudaError_t launch_fake_quant_linear(const float *X, const float *W, float s_x, const float *s_w, const float *bias,
                                     int M, int N, int K, int wbits, int8_t *qx, int8_t *qw, float *y,
                                     cudaStream_t st) {
    const size_t nx = (size_t)M * K, nw = (size_t)N * K;
    fq_forward_kernel<int8_t><<<fq_grid(nx), 256, 0, st>>>(X, nx, s_x, 0.0f, 8, 0, nullptr, qx);
    fq_rows_kernel<<<fq_grid(nw), 256, 0, st>>>(W, N, K, s_w, wbits, qw);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    Epi e;
    memset(&e, 0, sizeof(e));
    e.mode = EPI_F32;
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    e.f32 = y;
    e.ldf = N;
    return launch_linear(qx, K, qw, M, N, K, e, st);
}

}  // namespace mnmt
