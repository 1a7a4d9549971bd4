// epilogue.cuh -- the fused epilogue of a quantised linear (Sec. 3.3, Fig. 5),
// shared by the GEMV, IMMA and tcgen05 kernels: dequantise with the
// per-channel weight scale, add the full-precision bias, then requantise /
// ReLU + requantise / gamma-residual / fp32 / K-V cache write.
#pragma once

#include "common.cuh"
#include "internal.h"

namespace mnmt {

// epilogue of one output element from its dequantised, biased value y;
// t: decode step
MNMT_DEV void epi_store_y(const Epi &e, int m, int n, float y, int t) {
    switch (e.mode) {
        case EPI_Q8:
        case EPI_RELU_Q8: {
            const int8_t v = q8(e.mode == EPI_RELU_Q8 && !(y > 0.0f) ? 0.0f : y, e.inv_out[n]);
            e.out[(size_t)m * e.ldo + n] = v;
            if (e.out16) e.out16[(size_t)m * e.ldo + n] = __short2half_rn(v);
            break;
        }
        case EPI_RESID: {
            float *p = e.f32 + (size_t)m * e.ldf + n;
            *p = __fadd_rn(__fmul_rn(e.gamma, *p), y);
            break;
        }
        case EPI_F32:
            e.f32[(size_t)m * e.ldf + n] = y;
            break;
        case EPI_QKV_DEC: {
            int8_t v = q8(y, e.inv_out[n]);
            if (n < e.d) {
                e.out[(size_t)m * e.ldo + n] = v;
            } else {
                int seg = n >= 2 * e.d;
                int c = n - (seg ? 2 * e.d : e.d);
                int h = c / e.dh, i = c - h * e.dh;
                int8_t *dst = seg ? e.vc : e.kc;
                dst[(((size_t)m * e.H + h) * e.T + t) * e.dh + i] = v;
            }
            break;
        }
        case EPI_KV_CROSS: {
            int8_t v = q8(y, e.inv_out[n]);
            int b = m / e.S, s = m - b * e.S;
            int seg = n >= e.d;
            int c = n - (seg ? e.d : 0);
            int h = c / e.dh, i = c - h * e.dh;
            int8_t *dst = seg ? e.vc : e.kc;
            dst[(((size_t)b * e.H + h) * e.S + s) * e.dh + i] = v;
            break;
        }
        default:
            break;
    }
}

// epilogue of one output element; accf = fl(acc), the accumulator rounded to
// fp32 (exact for |acc| <= 2^24)
MNMT_DEV void epi_store_f(const Epi &e, int m, int n, float accf, int t) {
    epi_store_y(e, m, n, __fadd_rn(__fmul_rn(accf, __fmul_rn(e.s_x, e.s_w[n])), e.bias[n]), t);
}

// the same from the exact int32 accumulator
MNMT_DEV void epi_store(const Epi &e, int m, int n, int32_t acc, int t) { epi_store_f(e, m, n, __int2float_rn(acc), t); }

}  // namespace mnmt
