// gemm_tc.cu -- the quantised linear of Sec. 3.3 / Eq. 3 on the fifth-generation
// tensor cores (tcgen05), for layers where batch x beam (or batch x source
// length) makes the layer a dense contraction.
//
// Exactness.  The int8 codes are carried as fp16 (every integer of magnitude
// <= 2048 is an fp16 value), so each product a*w (|a*w| <= 2^14) is exact in
// the fp32 accumulator.  A sum of at most 1024 such products has magnitude
// <= 1024 * 128 * 128 = 2^24, so every partial sum is an integer that fp32
// represents exactly and the accumulation is exact whatever order the tensor
// core adds in.  K is therefore cut into chunks of 1024 (16 k-blocks of 64),
// each accumulated into its own TMEM columns; with two chunks the epilogue adds
// them with one fp32 addition, which returns fl(acc) -- the correctly rounded
// exact sum, the same value as (float)acc of the int32 accumulator.
//
// Pipeline (persistent CTAs, 128 x BN output tiles, 320 threads):
//   warp 0 lane 0   TMA producer: 128-byte-swizzled 128x64 (A) and BNx64 (W)
//                   fp16 tiles into a STAGES-deep shared-memory ring;
//   warp 1          allocates two TMEM accumulator buffers; lane 0 issues
//                   tcgen05.mma (M=128, N=BN, K=16 each), releases ring slots
//                   with tcgen05.commit and signals each finished tile;
//   warps 2..9      stage the per-column constants of a tile, then drain its
//                   TMEM buffer with tcgen05.ld (warp w reads lanes
//                   32*(w%4)..+31 = tile rows, half of the columns) and apply
//                   the fused epilogue of the linear while the MMAs of the
//                   next tile fill the other buffer.
// Grids of few 128 x 64 tiles run linear_tc_sk instead: the same pipeline for
// one tile per CTA, K split over a 2- or 4-CTA cluster, the partials reduced
// exactly in int32 through distributed shared memory (see its header).
// Every mbarrier wait is bounded (one second of %globaltimer); a wait that
// runs out records MNMT_ETIMEOUT in *status, the CTA stops issuing work, waits
// (bounded) for its own copies and MMAs in flight, frees its TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_fp16.h>

#include "common.cuh"
#include "epilogue.cuh"
#include "internal.h"
#include "mbarrier.cuh"
#include "mnmt.h"

namespace mnmt {
namespace {

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;             // fp16 per k-block: one 128-byte swizzle row
constexpr int TC_KB_PER_CHUNK = 16;   // 16 x 64 = 1024 products per exact fp32 chunk
constexpr int TC_EPI_WARPS = 8;                  // two warps per TMEM lane quarter
constexpr int TC_THREADS = 64 + TC_EPI_WARPS * 32;  // producer warp, MMA warp, epilogue warps

__device__ __forceinline__ uint32_t s_addr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *tm, int x, int y, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
        "[%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

// shared-memory matrix descriptor of a K-major operand tile laid out by TMA with
// 128-byte swizzling: rows of 128 bytes, 8-row (1024-byte) atoms stacked along
// M/N (stride byte offset 1024); leading byte offset unused for this layout
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1 << 16) | ((uint64_t)(1024 >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// instruction descriptor of kind::f16: D fp32, A and B fp16, both K-major
__host__ __device__ constexpr uint32_t idesc_f16(int m, int n) {
    return (1u << 4) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void mma_f16(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
        "%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

template <int NCOLS>
__device__ __forceinline__ void tmem_alloc(uint32_t slot) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot), "r"(NCOLS)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

template <int NCOLS>
__device__ __forceinline__ void tmem_free(uint32_t taddr) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(NCOLS) : "memory");
}

__host__ __device__ constexpr int pow2_cols(int c) { return c <= 32 ? 32 : c <= 64 ? 64 : c <= 128 ? 128 : c <= 256 ? 256 : 512; }

template <int BN, int STAGES>
struct TcLayout {
    static constexpr uint32_t A_BYTES = TC_BM * TC_BK * 2;
    static constexpr uint32_t B_BYTES = BN * TC_BK * 2;
    static constexpr uint32_t OFF_B = STAGES * A_BYTES;
    static constexpr uint32_t OFF_COLS = OFF_B + STAGES * B_BYTES;      // [2][3][BN] fp32
    static constexpr uint32_t OFF_BARS = OFF_COLS + 2 * 3 * BN * 4;
    static constexpr int NBARS = 2 * STAGES + 5;  // full[S], empty[S], acc_full[2], acc_empty[2], done
    static constexpr uint32_t OFF_MISC = OFF_BARS + NBARS * 8;
    static constexpr uint32_t BYTES = OFF_MISC + 16;
    static constexpr size_t SMEM = 1024 + BYTES;  // slack to align the ring to 1024 bytes
};

// named barrier over the epilogue warps only
__device__ __forceinline__ void epi_bar_sync() { asm volatile("bar.sync 1, %0;" ::"n"(TC_EPI_WARPS * 32) : "memory"); }

// 16 accumulators of one row -> int8 codes packed little-endian into 4 words:
// q8(y, inv) = clamp(rne(fl(y * inv)), -127, 127), with the clamp taken first
// (the same value: rne is monotone and +-127 are integers) and rne done by
// adding 1.5 * 2^23, whose low byte is then the two's-complement code
template <bool RELU>
__device__ __forceinline__ void q8_pack16(const float (&a)[16], const float *sc, const float *bs, const float *inv,
                                          uint32_t (&w)[4]) {
#pragma unroll
    for (int g = 0; g < 4; g++) {
        uint32_t b[4];
#pragma unroll
        for (int i = 0; i < 4; i++) {
            const int c = 4 * g + i;
            float y = __fadd_rn(__fmul_rn(a[c], sc[c]), bs[c]);
            if (RELU) y = y > 0.0f ? y : 0.0f;
            float z = __fmul_rn(y, inv[c]);
            z = fminf(fmaxf(z, -127.0f), 127.0f);
            b[i] = __float_as_uint(__fadd_rn(z, 12582912.0f));
        }
        w[g] = __byte_perm(__byte_perm(b[0], b[1], 0x0040), __byte_perm(b[2], b[3], 0x0040), 0x5410);
    }
}

// the 16-column epilogue below applies (every destination row segment of 16
// outputs is contiguous and 16-byte aligned)
__device__ __forceinline__ bool epi_vec_ok(const Epi &e) {
    const auto al = [](const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
    switch (e.mode) {
        case EPI_Q8:
        case EPI_RELU_Q8:
            return e.ldo % 16 == 0 && al(e.out) && al(e.out16);
        case EPI_RESID:
        case EPI_F32:
            return e.ldf % 4 == 0 && al(e.f32);
        case EPI_QKV_DEC:
            return e.ldo % 16 == 0 && al(e.out) && al(e.kc) && al(e.vc) && e.dh % 16 == 0 && e.d % 16 == 0;
        case EPI_KV_CROSS:
            return al(e.kc) && al(e.vc) && e.dh % 16 == 0 && e.d % 16 == 0;
        default:
            return false;
    }
}

// The epilogue of outputs (row, col0 .. col0+15) of one row, col0 a multiple
// of 16, all columns < N: the same arithmetic as epi_store_f, with one 16-byte
// access per 16 int8 codes or 4 fp32 values.
// rpre, if given, holds the 16 residual values of a RESID store, loaded earlier.
__device__ __forceinline__ void epi_store16(const Epi &e, int row, int col0, const float (&a)[16], const float *sc,
                                            const float *bs, const float *inv, int t, const float4 *rpre = nullptr) {
    if (e.mode == EPI_RESID || e.mode == EPI_F32) {
        float4 *p = reinterpret_cast<float4 *>(e.f32 + (size_t)row * e.ldf + col0);
        float4 r[4];
        if (e.mode == EPI_RESID) {
#pragma unroll
            for (int g = 0; g < 4; g++) r[g] = rpre ? rpre[g] : p[g];
        }
#pragma unroll
        for (int g = 0; g < 4; g++) {
            float y[4];
#pragma unroll
            for (int i = 0; i < 4; i++) y[i] = __fadd_rn(__fmul_rn(a[4 * g + i], sc[4 * g + i]), bs[4 * g + i]);
            if (e.mode == EPI_RESID) {
                y[0] = __fadd_rn(__fmul_rn(e.gamma, r[g].x), y[0]);
                y[1] = __fadd_rn(__fmul_rn(e.gamma, r[g].y), y[1]);
                y[2] = __fadd_rn(__fmul_rn(e.gamma, r[g].z), y[2]);
                y[3] = __fadd_rn(__fmul_rn(e.gamma, r[g].w), y[3]);
            }
            p[g] = make_float4(y[0], y[1], y[2], y[3]);
        }
        return;
    }
    uint32_t w[4];
    if (e.mode == EPI_RELU_Q8)
        q8_pack16<true>(a, sc, bs, inv, w);
    else
        q8_pack16<false>(a, sc, bs, inv, w);
    int8_t *dst;
    if (e.mode == EPI_QKV_DEC) {
        if (col0 < e.d) {
            dst = e.out + (size_t)row * e.ldo + col0;
        } else {
            const int seg = col0 >= 2 * e.d;
            const int c = col0 - (seg ? 2 * e.d : e.d);
            const int h = c / e.dh, i = c - h * e.dh;
            dst = (seg ? e.vc : e.kc) + (((size_t)row * e.H + h) * e.T + t) * e.dh + i;
        }
    } else if (e.mode == EPI_KV_CROSS) {
        const int b = row / e.S, sp = row - b * e.S;
        const int seg = col0 >= e.d;
        const int c = col0 - (seg ? e.d : 0);
        const int h = c / e.dh, i = c - h * e.dh;
        dst = (seg ? e.vc : e.kc) + (((size_t)b * e.H + h) * e.S + sp) * e.dh + i;
    } else {
        dst = e.out + (size_t)row * e.ldo + col0;
        if (e.out16) {
            // the fp16 copy of the 16 codes (exact), as two 16-byte stores
            uint32_t h[8];
#pragma unroll
            for (int k = 0; k < 8; k++) {
                const uint32_t word = w[k >> 1] >> (16 * (k & 1));
                const __half lo = __short2half_rn((short)(int8_t)(word & 0xFFu));
                const __half hi = __short2half_rn((short)(int8_t)((word >> 8) & 0xFFu));
                h[k] = (uint32_t)__half_as_ushort(lo) | ((uint32_t)__half_as_ushort(hi) << 16);
            }
            uint4 *d16 = reinterpret_cast<uint4 *>(e.out16 + (size_t)row * e.ldo + col0);
            d16[0] = make_uint4(h[0], h[1], h[2], h[3]);
            d16[1] = make_uint4(h[4], h[5], h[6], h[7]);
        }
    }
    *reinterpret_cast<uint4 *>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}

// Persistent kernel: CTA c takes output tiles c, c + gridDim.x, ... (M-tile
// index fastest, so the CTAs of one wave share weight tiles in L2).  The TMA
// ring runs continuously across tiles; the accumulator is double-buffered in
// TMEM so the epilogue of one tile overlaps the MMAs of the next.
template <int BN, int NCH, int STAGES, int NBUF>
__global__ void __launch_bounds__(TC_THREADS, 1) linear_tc(const __grid_constant__ CUtensorMap tmA,
                                                           const __grid_constant__ CUtensorMap tmB, int M, int N,
                                                           int K, Epi e, int *status) {
    pdl_grid_wait();
    using L = TcLayout<BN, STAGES>;
    constexpr int ACC_COLS = NCH * BN;  // one accumulator buffer (NBUF of them)
    constexpr int NCOLS = pow2_cols(NBUF * ACC_COLS);
    static_assert(NBUF * ACC_COLS <= 512, "TMEM holds 512 columns");
    constexpr uint32_t IDESC = idesc_f16(TC_BM, BN);
    if (e.skip && *e.skip) return;

    extern __shared__ uint8_t tc_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_raw) + 1023) & ~(uintptr_t)1023);
    float *cols = reinterpret_cast<float *>(sm + L::OFF_COLS);
    const uint32_t bars = s_addr(sm + L::OFF_BARS);
    auto full_bar = [&](int s) { return bars + 8u * s; };
    auto empty_bar = [&](int s) { return bars + 8u * (STAGES + s); };
    auto accf_bar = [&](int b) { return bars + 8u * (2 * STAGES + b); };
    auto acce_bar = [&](int b) { return bars + 8u * (2 * STAGES + 2 + b); };
    const uint32_t done_bar = bars + 8u * (2 * STAGES + 4);
    uint32_t *misc = reinterpret_cast<uint32_t *>(sm + L::OFF_MISC);  // [0] tmem base, [1] abort, [2] consumed
    volatile uint32_t *abort_flag = misc + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mt = (M + TC_BM - 1) / TC_BM;
    const int tiles = mt * ((N + BN - 1) / BN);
    const int nkb = (K + TC_BK - 1) / TC_BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; s++) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < 2; b++) {
            mbar_init(accf_bar(b), 1);
            mbar_init(acce_bar(b), TC_EPI_WARPS);
        }
        mbar_init(done_bar, 1);
        misc[1] = 0;
        misc[2] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc<NCOLS>(s_addr(misc));
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = misc[0];

    // The producer and the MMA issuer are single threads whose per-k-block
    // cost (mbarrier tests, TMA and MMA issue) bounds small grids, so their
    // loops test the shared abort flag once per tile, not per k-block.
    uint32_t issued = 0;
    if (warp == 0 && lane == 0) {
        // ---- TMA producer: k-blocks of all this CTA's tiles through the ring ----
        uint32_t it = 0;
        bool failed = false;
        const uint32_t a_ring = s_addr(sm), b_ring = s_addr(sm + L::OFF_B);
        for (int tile = blockIdx.x; tile < tiles && !failed && !*abort_flag; tile += gridDim.x) {
            const int m0 = (tile % mt) * TC_BM, n0 = (tile / mt) * BN;
            for (int kb = 0; kb < nkb; kb++, it++) {
                const int s = (int)(it % STAGES);
                if (it >= STAGES && !mbar_wait(empty_bar(s), (it / STAGES - 1) & 1)) {
                    *abort_flag = 1;
                    set_status(status, MNMT_ETIMEOUT);
                    failed = true;
                    break;
                }
                mbar_expect_tx(full_bar(s), L::A_BYTES + L::B_BYTES);
                tma_load_2d(a_ring + s * L::A_BYTES, &tmA, kb * TC_BK, m0, full_bar(s));
                tma_load_2d(b_ring + s * L::B_BYTES, &tmB, kb * TC_BK, n0, full_bar(s));
                issued = it + 1;
            }
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer ----
        uint32_t it = 0, lt = 0;
        bool failed = false;
        const uint64_t a_desc = sw128_desc(s_addr(sm)), b_desc = sw128_desc(s_addr(sm + L::OFF_B));
        for (int tile = blockIdx.x; tile < tiles && !failed && !*abort_flag; tile += gridDim.x, lt++) {
            const int buf = (int)(lt % NBUF);
            if (lt >= NBUF && !mbar_wait(acce_bar(buf), ((lt / NBUF) - 1) & 1)) {
                *abort_flag = 1;
                set_status(status, MNMT_ETIMEOUT);
                break;
            }
            tc_fence_after();
            const uint32_t dbase = tbase + (uint32_t)(buf * ACC_COLS);
            for (int kb = 0; kb < nkb; kb++, it++) {
                const int s = (int)(it % STAGES);
                if (!mbar_wait(full_bar(s), (it / STAGES) & 1)) {
                    *abort_flag = 1;
                    set_status(status, MNMT_ETIMEOUT);
                    failed = true;
                    break;
                }
                tc_fence_after();
                const uint32_t d = dbase + (uint32_t)((kb / TC_KB_PER_CHUNK) * BN);
                // descriptor start addresses advance in 16-byte units
                const uint64_t ad = a_desc + (uint64_t)((s * L::A_BYTES) >> 4);
                const uint64_t bd = b_desc + (uint64_t)((s * L::B_BYTES) >> 4);
#pragma unroll
                for (int k = 0; k < TC_BK / 16; k++)
                    mma_f16(d, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), IDESC,
                            (uint32_t)((kb % TC_KB_PER_CHUNK) | k));
                mma_commit(empty_bar(s));
            }
            if (failed) break;
            mma_commit(accf_bar(buf));
        }
        // every MMA of this CTA is issued: the stream's next kernel may launch
        // (it waits for this grid's completion before it reads anything)
        pdl_allow_next();
        misc[2] = it;          // k-blocks whose copies this thread saw land
        mma_commit(done_bar);  // arrives once every MMA issued above has completed
    } else if (warp >= 2) {
        // ---- epilogue: TMEM -> registers -> fused epilogue -> global ----
        const int ew = warp - 2;                       // 0 .. TC_EPI_WARPS-1
        const int q = warp & 3;                        // TMEM lane quarter of this warp
        const int half = ew >> 2;                      // which half of the tile's columns
        constexpr int JN = BN / 32;                    // 16-column chunks per thread and tile
        constexpr int PRE_CH = BN == 64 ? JN : 0;      // residual chunks loaded ahead
        constexpr int EPI_UNROLL = PRE_CH > 0 ? PRE_CH : 1;
        const int t = e.t_ptr ? *e.t_ptr : 0;
        const bool vec = epi_vec_ok(e);
        uint32_t lt = 0;
        for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, lt++) {
            const int buf = (int)(lt % NBUF);
            const int m0 = (tile % mt) * TC_BM, n0 = (tile / mt) * BN;
            // per-column constants of this tile, double-buffered by tile parity
            float *c_sc = cols + (lt & 1) * 3 * BN, *c_b = c_sc + BN, *c_inv = c_b + BN;
            for (int i = ew * 32 + lane; i < BN; i += TC_EPI_WARPS * 32) {
                const int n = n0 + i;
                const bool ok = n < N;
                c_sc[i] = ok ? __fmul_rn(e.s_x, e.s_w[n]) : 0.0f;
                c_b[i] = ok ? e.bias[n] : 0.0f;
                c_inv[i] = ok && e.inv_out ? e.inv_out[n] : 0.0f;
            }
            epi_bar_sync();
            const int row = m0 + 32 * q + lane;
            // 128 x 64 tiles: a residual epilogue loads its 32 residual values
            // while the tile's MMAs run (the store then waits on no load)
            float4 rpre[4 * PRE_CH > 0 ? 4 * PRE_CH : 1];
            const bool pre = PRE_CH > 0 && e.mode == EPI_RESID && vec && row < M;
            if (pre) {
#pragma unroll
                for (int jj = 0; jj < PRE_CH; jj++) {
                    const int col0 = n0 + 16 * (half * JN + jj);
                    if (col0 + 16 <= N) {
                        const float4 *p = reinterpret_cast<const float4 *>(e.f32 + (size_t)row * e.ldf + col0);
#pragma unroll
                        for (int g = 0; g < 4; g++) rpre[4 * jj + g] = p[g];
                    }
                }
            }
            // every epilogue warp runs every tile of the loop (the named barrier
            // above needs all of them); after an abort the tiles are skipped
            bool ok = *abort_flag == 0 && mbar_wait(accf_bar(buf), (lt / NBUF) & 1);
            if (!ok && *abort_flag == 0) {
                *abort_flag = 1;
                set_status(status, MNMT_ETIMEOUT);
            }
            tc_fence_after();
            ok = __all_sync(0xFFFFFFFFu, ok && *abort_flag == 0);
            const uint32_t taddr = tbase + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * ACC_COLS);
            unsigned long long best = 0ull;
#pragma unroll EPI_UNROLL
            for (int jj = 0; ok && jj < JN; jj++) {
                const int j = half * JN + jj;
                uint32_t r0[16], r1[16];
                tmem_ld16(taddr + 16 * j, r0);
                if (NCH == 2) tmem_ld16(taddr + BN + 16 * j, r1);
                tmem_wait_ld();
                float a[16];
#pragma unroll
                for (int i = 0; i < 16; i++)
                    a[i] = NCH == 2 ? __fadd_rn(__uint_as_float(r0[i]), __uint_as_float(r1[i]))
                                    : __uint_as_float(r0[i]);
                const int col0 = n0 + 16 * j;
                if (col0 >= N) continue;
                const float *sc = c_sc + 16 * j, *bs = c_b + 16 * j, *inv = c_inv + 16 * j;
                if (e.mode == EPI_ARGMAX) {
#pragma unroll
                    for (int i = 0; i < 16; i++) {
                        if (col0 + i < N) {
                            const float y = __fadd_rn(__fmul_rn(a[i], sc[i]), bs[i]);
                            const unsigned long long kk = pack_key(y, (uint32_t)(col0 + i));
                            best = kk > best ? kk : best;
                        }
                    }
                } else if (vec && col0 + 16 <= N) {
                    if (row < M) epi_store16(e, row, col0, a, sc, bs, inv, t, PRE_CH > 0 && pre ? rpre + 4 * jj : nullptr);
                } else if (row < M) {
#pragma unroll
                    for (int i = 0; i < 16; i++)
                        if (col0 + i < N) epi_store_f(e, row, col0 + i, a[i], t);
                }
            }
            // this warp is done with the accumulator buffer
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(acce_bar(buf));
            if (e.mode == EPI_ARGMAX && row < M && best) atomicMax(e.keys + row, best);
        }
    }

    // ---- teardown ----
    __syncthreads();
    if (warp == 0 && lane == 0 && *abort_flag) {
        // copies the MMA issuer never consumed are still landing in this CTA's ring
        for (uint32_t it = misc[2]; it < issued; it++) mbar_wait(full_bar((int)(it % STAGES)), (it / STAGES) & 1);
    }
    if (warp == 1) {
        if (lane == 0) mbar_wait(done_bar, 0);
        __syncwarp();
        tc_fence_after();
        tmem_free<NCOLS>(tbase);
    }
}

// ---------------------------------------------------------------------------
// int8 codes -> fp16 (exact); 16 codes per thread and step
// ---------------------------------------------------------------------------
__global__ void codes_to_f16_kernel(const int8_t *__restrict__ src, int ld_src, __half *__restrict__ dst, int ld_dst,
                                    int rows, int cols) {
    pdl_grid_wait();
    const int per_row = cols >> 4;
    const long total = (long)rows * per_row;
    for (long i = blockIdx.x * (long)blockDim.x + threadIdx.x; i < total; i += (long)gridDim.x * blockDim.x) {
        const int r = (int)(i / per_row), c = (int)(i - (long)r * per_row) << 4;
        const int4 v = *reinterpret_cast<const int4 *>(src + (size_t)r * ld_src + c);
        const int8_t *b = reinterpret_cast<const int8_t *>(&v);
        __align__(16) __half h[16];
#pragma unroll
        for (int k = 0; k < 16; k++) h[k] = __short2half_rn((short)b[k]);
        int4 *o = reinterpret_cast<int4 *>(dst + (size_t)r * ld_dst + c);
        o[0] = *reinterpret_cast<const int4 *>(h);
        o[1] = *reinterpret_cast<const int4 *>(h + 8);
    }
}

__global__ void codes_to_f16_tail(const int8_t *src, __half *dst, size_t from, size_t n) {
    pdl_grid_wait();
    size_t i = from + blockIdx.x * (size_t)blockDim.x + threadIdx.x;
    if (i < n) dst[i] = __short2half_rn((short)src[i]);
}

// ---------------------------------------------------------------------------
// Split-K over a thread-block cluster, for grids with few 128 x 64 tiles
// (the few-hundred-row linears of a batched decode step).  The S CTAs of a
// cluster share one output tile and take consecutive ranges of its k-blocks;
// each range holds at most 16 k-blocks (1024 products), so a CTA's fp32
// accumulator is an exact integer.  The partials are converted to int32 and
// reduce-scattered through distributed shared memory: CTA c owns columns
// [c BN/S, (c+1) BN/S) of the tile, receives every CTA's partial of them in
// its slot array, adds them in int32 (exact: |acc| <= 2048 * 2^14) and runs
// the linear's epilogue on (float)acc -- the correctly rounded accumulator,
// as in the unsplit kernel.  Every thread of every CTA reaches the one
// cluster barrier (also after a timed-out wait), and no CTA touches another's
// shared memory after it.
// ---------------------------------------------------------------------------
constexpr int SK_BN = 64;
constexpr int SK_STAGES = 6;

template <int S>
struct SkLayout {
    static constexpr uint32_t A_BYTES = TC_BM * TC_BK * 2;
    static constexpr uint32_t B_BYTES = SK_BN * TC_BK * 2;
    static constexpr uint32_t OFF_B = SK_STAGES * A_BYTES;
    static constexpr uint32_t OFF_RECV = OFF_B + SK_STAGES * B_BYTES;  // [S][128][BN/S] int32
    static constexpr uint32_t RECV_BYTES = S * TC_BM * (SK_BN / S) * 4;
    static constexpr uint32_t OFF_COLS = OFF_RECV + RECV_BYTES;          // [3][BN/S] fp32
    static constexpr uint32_t OFF_BARS = OFF_COLS + 3 * (SK_BN / S) * 4;
    static constexpr int NBARS = 2 * SK_STAGES + 2;                     // full[S], empty[S], acc_full, done
    static constexpr uint32_t OFF_MISC = OFF_BARS + NBARS * 8;
    static constexpr uint32_t BYTES = OFF_MISC + 16;
    static constexpr size_t SMEM = 1024 + BYTES;
};

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// shared::cluster address of the same offset in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t map_rank(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}

__device__ __forceinline__ void st_cluster_v4(uint32_t addr, int a, int b, int c, int d) {
    asm volatile("st.shared::cluster.v4.s32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(a), "r"(b), "r"(c), "r"(d)
                 : "memory");
}

__device__ __forceinline__ void cluster_barrier() {
    asm volatile("barrier.cluster.arrive.release;\n\tbarrier.cluster.wait.acquire;" ::: "memory");
}

// the two halves of a cluster barrier phase: every thread arrives once the
// CTA is set up and waits before its first access to another CTA's memory
// (all CTAs of the cluster have then started)
__device__ __forceinline__ void cluster_arrive_relaxed() { asm volatile("barrier.cluster.arrive.relaxed;" ::: "memory"); }
__device__ __forceinline__ void cluster_wait() { asm volatile("barrier.cluster.wait.acquire;" ::: "memory"); }

template <int S>
__global__ void __launch_bounds__(TC_THREADS, 1) linear_tc_sk(const __grid_constant__ CUtensorMap tmA,
                                                              const __grid_constant__ CUtensorMap tmB, int M, int N,
                                                              int K, Epi e, int *status) {
    pdl_grid_wait();
    using L = SkLayout<S>;
    constexpr int SW = SK_BN / S;  // columns this CTA finishes
    constexpr uint32_t IDESC = idesc_f16(TC_BM, SK_BN);
    if (e.skip && *e.skip) return;  // one flag for every CTA of the grid

    extern __shared__ uint8_t tc_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(tc_raw) + 1023) & ~(uintptr_t)1023);
    float *c_sc = reinterpret_cast<float *>(sm + L::OFF_COLS), *c_b = c_sc + SW, *c_inv = c_b + SW;
    const uint32_t bars = s_addr(sm + L::OFF_BARS);
    auto full_bar = [&](int s) { return bars + 8u * s; };
    auto empty_bar = [&](int s) { return bars + 8u * (SK_STAGES + s); };
    const uint32_t accf_bar = bars + 8u * (2 * SK_STAGES), done_bar = accf_bar + 8u;
    uint32_t *misc = reinterpret_cast<uint32_t *>(sm + L::OFF_MISC);  // [0] tmem base, [1] abort, [2] consumed
    volatile uint32_t *abort_flag = misc + 1;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_rank();
    const int tile = blockIdx.x / S;
    const int mt = (M + TC_BM - 1) / TC_BM;
    const int m0 = (tile % mt) * TC_BM, n0 = (tile / mt) * SK_BN;
    const int nkb = (K + TC_BK - 1) / TC_BK;
    const int per = (nkb + S - 1) / S;
    const int kb0 = min(nkb, (int)rank * per), kb1 = min(nkb, kb0 + per);
    const bool has_k = kb1 > kb0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < SK_STAGES; s++) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        mbar_init(accf_bar, 1);
        mbar_init(done_bar, 1);
        misc[1] = 0;
        misc[2] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    }
    if (warp == 1) {
        tmem_alloc<SK_BN>(s_addr(misc));
        tc_fence_before();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = misc[0];
    cluster_arrive_relaxed();

    uint32_t issued = 0;
    if (warp == 0 && lane == 0) {
        // ---- TMA producer: this CTA's k-blocks of the tile ----
        const uint32_t a_ring = s_addr(sm), b_ring = s_addr(sm + L::OFF_B);
        uint32_t it = 0;
        for (int kb = kb0; kb < kb1; kb++, it++) {
            const int s = (int)(it % SK_STAGES);
            if (it >= SK_STAGES && !mbar_wait(empty_bar(s), (it / SK_STAGES - 1) & 1)) {
                *abort_flag = 1;
                set_status(status, MNMT_ETIMEOUT);
                break;
            }
            mbar_expect_tx(full_bar(s), L::A_BYTES + L::B_BYTES);
            tma_load_2d(a_ring + s * L::A_BYTES, &tmA, kb * TC_BK, m0, full_bar(s));
            tma_load_2d(b_ring + s * L::B_BYTES, &tmB, kb * TC_BK, n0, full_bar(s));
            issued = it + 1;
        }
    } else if (warp == 1 && lane == 0) {
        // ---- MMA issuer: one accumulation over the range (<= 1024 products) ----
        const uint64_t a_desc = sw128_desc(s_addr(sm)), b_desc = sw128_desc(s_addr(sm + L::OFF_B));
        uint32_t it = 0;
        for (int kb = kb0; kb < kb1; kb++, it++) {
            const int s = (int)(it % SK_STAGES);
            if (!mbar_wait(full_bar(s), (it / SK_STAGES) & 1)) {
                *abort_flag = 1;
                set_status(status, MNMT_ETIMEOUT);
                break;
            }
            tc_fence_after();
            const uint64_t ad = a_desc + (uint64_t)((s * L::A_BYTES) >> 4);
            const uint64_t bd = b_desc + (uint64_t)((s * L::B_BYTES) >> 4);
#pragma unroll
            for (int k = 0; k < TC_BK / 16; k++)
                mma_f16(tbase, ad + (uint64_t)(2 * k), bd + (uint64_t)(2 * k), IDESC, (uint32_t)(it | k));
            mma_commit(empty_bar(s));
        }
        pdl_allow_next();  // every MMA of this CTA is issued
        misc[2] = it;
        mma_commit(accf_bar);  // also after a timed-out wait: the epilogue reaches the cluster barrier
        mma_commit(done_bar);
    }

    // ---- epilogue warps: send the partials, then finish the owned columns ----
    const int ew = warp - 2, q = warp & 3, half = ew >> 2;
    const int row = m0 + 32 * q + lane;
    const int oc = 16 * half;                          // owned chunk of this thread (within SW)
    const int col0 = n0 + (int)rank * SW + oc;
    const bool vec = epi_vec_ok(e);
    const int t = e.t_ptr ? *e.t_ptr : 0;
    float4 rpre[4];
    bool pre = false;
    if (warp >= 2) {
        for (int i = ew * 32 + lane; i < SW; i += TC_EPI_WARPS * 32) {
            const int n = n0 + (int)rank * SW + i;
            const bool in = n < N;
            c_sc[i] = in ? __fmul_rn(e.s_x, e.s_w[n]) : 0.0f;
            c_b[i] = in ? e.bias[n] : 0.0f;
            c_inv[i] = in && e.inv_out ? e.inv_out[n] : 0.0f;
        }
        pre = e.mode == EPI_RESID && vec && oc < SW && row < M && col0 + 16 <= N;
        if (pre) {
            const float4 *p = reinterpret_cast<const float4 *>(e.f32 + (size_t)row * e.ldf + col0);
#pragma unroll
            for (int g = 0; g < 4; g++) rpre[g] = p[g];
        }
        bool ok = *abort_flag == 0 && mbar_wait(accf_bar, 0);
        if (!ok && *abort_flag == 0) {
            *abort_flag = 1;
            set_status(status, MNMT_ETIMEOUT);
        }
        tc_fence_after();
        ok = __all_sync(0xFFFFFFFFu, ok && *abort_flag == 0);
        cluster_wait();  // every CTA of the cluster has started
        if (ok) {
            const uint32_t taddr = tbase + ((uint32_t)(32 * q) << 16);
            const uint32_t recv = s_addr(sm + L::OFF_RECV);
#pragma unroll
            for (int jj = 0; jj < 2; jj++) {
                const int j = 2 * half + jj;  // 16-column chunk of the tile
                int v[16];
                if (has_k) {
                    uint32_t r0[16];
                    tmem_ld16(taddr + 16 * j, r0);
                    tmem_wait_ld();
#pragma unroll
                    for (int i = 0; i < 16; i++) v[i] = __float2int_rn(__uint_as_float(r0[i]));  // exact integers
                } else {
#pragma unroll
                    for (int i = 0; i < 16; i++) v[i] = 0;
                }
                const int owner = (16 * j) / SW, cin = 16 * j - owner * SW;
                const uint32_t dst = map_rank(recv + (uint32_t)(((rank * TC_BM + 32 * q + lane) * SW + cin) * 4),
                                              (uint32_t)owner);
#pragma unroll
                for (int g = 0; g < 4; g++) st_cluster_v4(dst + 16 * g, v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]);
            }
        }
        tc_fence_before();
    }
    if (warp < 2) cluster_wait();
    // every thread of every CTA: the partials have landed in their owners
    cluster_barrier();
    if (warp >= 2 && oc < SW && *abort_flag == 0 && row < M && col0 < N) {
        const int *rv = reinterpret_cast<const int *>(sm + L::OFF_RECV);
        int acc[16];
#pragma unroll
        for (int i = 0; i < 16; i++) acc[i] = 0;
#pragma unroll
        for (int src = 0; src < S; src++) {
            const int4 *p = reinterpret_cast<const int4 *>(rv + ((size_t)src * TC_BM + 32 * q + lane) * SW + oc);
#pragma unroll
            for (int g = 0; g < 4; g++) {
                const int4 w = p[g];
                acc[4 * g] += w.x;
                acc[4 * g + 1] += w.y;
                acc[4 * g + 2] += w.z;
                acc[4 * g + 3] += w.w;
            }
        }
        float a[16];
#pragma unroll
        for (int i = 0; i < 16; i++) a[i] = __int2float_rn(acc[i]);  // fl(acc), as the unsplit kernel
        const float *sc = c_sc + oc, *bs = c_b + oc, *inv = c_inv + oc;
        if (e.mode == EPI_ARGMAX) {
            unsigned long long best = 0ull;
#pragma unroll
            for (int i = 0; i < 16; i++) {
                if (col0 + i < N) {
                    const float y = __fadd_rn(__fmul_rn(a[i], sc[i]), bs[i]);
                    const unsigned long long kk = pack_key(y, (uint32_t)(col0 + i));
                    best = kk > best ? kk : best;
                }
            }
            if (best) atomicMax(e.keys + row, best);
        } else if (vec && col0 + 16 <= N) {
            epi_store16(e, row, col0, a, sc, bs, inv, t, pre ? rpre : nullptr);
        } else {
#pragma unroll
            for (int i = 0; i < 16; i++)
                if (col0 + i < N) epi_store_f(e, row, col0 + i, a[i], t);
        }
    }

    // ---- teardown ----
    __syncthreads();
    if (warp == 0 && lane == 0 && *abort_flag) {
        for (uint32_t it = misc[2]; it < issued; it++) mbar_wait(full_bar((int)(it % SK_STAGES)), (it / SK_STAGES) & 1);
    }
    if (warp == 1) {
        if (lane == 0) mbar_wait(done_bar, 0);
        __syncwarp();
        tc_fence_after();
        tmem_free<SK_BN>(tbase);
    }
}

// One thread waits (bounded) on a barrier phase that never completes: the
// give-up path of every pipeline wait above, exercised without a fault.
__global__ void wait_timeout_selftest_kernel(int *status) {
    __shared__ __align__(8) unsigned long long bar;
    const uint32_t b = s_addr(&bar);
    if (threadIdx.x == 0) {
        mbar_init(b, 1);  // one arrival expected; none comes
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait(b, 0)) set_status(status, MNMT_ETIMEOUT);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
int g_num_sms = 148;
int g_sk_clusters[5] = {0, 0, 0, 0, 0};  // clusters of S split-K CTAs that fit at once (S = 2, 4)

bool make_map(CUtensorMap *tm, const __half *p, int cols, int rows, int ld, int box_rows) {
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {(cuuint32_t)TC_BK, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<__half *>(p), dims, strides, box, estr,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int BN, int NCH, int STAGES, int NBUF>
cudaError_t tc_attr() {
    return cudaFuncSetAttribute(linear_tc<BN, NCH, STAGES, NBUF>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)TcLayout<BN, STAGES>::SMEM);
}

template <int BN, int NCH, int STAGES, int NBUF>
cudaError_t tc_launch(const CUtensorMap &ta, const CUtensorMap &tb, int M, int N, int K, const Epi &e, int *status,
                      cudaStream_t st) {
    const long tiles = (long)((M + TC_BM - 1) / TC_BM) * ((N + BN - 1) / BN);
    const int grid = (int)(tiles < g_num_sms ? tiles : g_num_sms);
    launch_pdl(linear_tc<BN, NCH, STAGES, NBUF>, grid, TC_THREADS, TcLayout<BN, STAGES>::SMEM, st, ta, tb, M, N, K, e, status);
    return cudaGetLastError();
}

// cluster attribute (S, 1, 1) and programmatic dependent launch outside
// stream captures, as launch_pdl
template <int S>
cudaLaunchConfig_t sk_config(long tiles, cudaStream_t st, cudaLaunchAttribute (&attr)[2], bool pdl) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(tiles * S));
    cfg.blockDim = dim3(TC_THREADS);
    cfg.dynamicSmemBytes = SkLayout<S>::SMEM;
    cfg.stream = st;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl ? 2 : 1;
    return cfg;
}

template <int S>
cudaError_t tc_sk_init() {
    cudaError_t err = cudaFuncSetAttribute(linear_tc_sk<S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                           (int)SkLayout<S>::SMEM);
    if (err != cudaSuccess) return err;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = sk_config<S>(64, nullptr, attr, false);
    int n = 0;
    err = cudaOccupancyMaxActiveClusters(&n, linear_tc_sk<S>, &cfg);
    g_sk_clusters[S] = err == cudaSuccess ? n : 0;
    return err;
}

template <int S>
cudaError_t tc_launch_sk(const CUtensorMap &ta, const CUtensorMap &tb, int M, int N, int K, const Epi &e, int *status,
                         cudaStream_t st) {
    const long tiles = (long)((M + TC_BM - 1) / TC_BM) * ((N + SK_BN - 1) / SK_BN);
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) cs = cudaStreamCaptureStatusNone;
    cudaLaunchAttribute attr[2];
    cudaLaunchConfig_t cfg = sk_config<S>(tiles, st, attr, cs != cudaStreamCaptureStatusActive);
    return cudaLaunchKernelEx(&cfg, linear_tc_sk<S>, ta, tb, M, N, K, e, status);
}

constexpr int TC_STAGES = 6;
// 128 x 256 tiles: half the A-tile bytes per FLOP, for grids with enough
// tiles; with two K chunks the 512-column accumulator fills TMEM, so that
// variant keeps one accumulator buffer (its epilogue does not overlap)
constexpr int TC_STAGES_WIDE = 4;
// 128 x 64 tiles for grids that would leave SMs idle (a few hundred rows):
// twice the CTAs, and each streams a third fewer bytes per k-block
constexpr int TC_STAGES_NARROW = 8;

}  // namespace

cudaError_t linear_tc_init() {
    cudaDriverEntryPointQueryResult q;
    void *fn = nullptr;
    cudaError_t err = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q);
    if (err != cudaSuccess) return err;
    if (q != cudaDriverEntryPointSuccess || !fn) return cudaErrorSymbolNotFound;
    g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    int dev = 0;
    if ((err = cudaGetDevice(&dev)) != cudaSuccess) return err;
    if ((err = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return err;
    err = tc_attr<128, 1, TC_STAGES, 2>();
    if (err == cudaSuccess) err = tc_attr<128, 2, TC_STAGES, 2>();
    if (err == cudaSuccess) err = tc_attr<256, 1, TC_STAGES_WIDE, 2>();
    if (err == cudaSuccess) err = tc_attr<256, 2, TC_STAGES_WIDE, 1>();
    if (err == cudaSuccess) err = tc_attr<64, 1, TC_STAGES_NARROW, 2>();
    if (err == cudaSuccess) err = tc_attr<64, 2, TC_STAGES_NARROW, 2>();
    if (err == cudaSuccess) err = tc_sk_init<2>();
    if (err == cudaSuccess) err = tc_sk_init<4>();
    return err;
}

int device_sm_count() { return g_num_sms; }

cudaError_t launch_wait_timeout_selftest(int *status, cudaStream_t st) {
    wait_timeout_selftest_kernel<<<1, 32, 0, st>>>(status);
    return cudaGetLastError();
}

bool linear_tc_shape_ok(int M, int N, int K, int lda, int ldw, const void *A16, const void *W16) {
    return g_encode && M >= 1 && N >= 1 && K >= 8 && K <= 2 * TC_KB_PER_CHUNK * TC_BK && K % 8 == 0 && lda >= K &&
           ldw >= K && lda % 8 == 0 && ldw % 8 == 0 && ((reinterpret_cast<uintptr_t>(A16) | reinterpret_cast<uintptr_t>(W16)) & 15) == 0;
}

cudaError_t launch_linear_tc(const __half *A16, int lda, const __half *W16, int ldw, int M, int N, int K,
                             const Epi &e, int *status, cudaStream_t st) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    if (!linear_tc_shape_ok(M, N, K, lda, ldw, A16, W16)) return cudaErrorInvalidValue;
    const bool two_chunks = K > TC_KB_PER_CHUNK * TC_BK;
    const long tiles_wide = (long)((M + TC_BM - 1) / TC_BM) * ((N + 255) / 256);
    const bool wide = N >= 256 && tiles_wide >= g_num_sms;
    const long tiles_128 = (long)((M + TC_BM - 1) / TC_BM) * ((N + 127) / 128);
    const bool narrow = !wide && tiles_128 < g_num_sms;
    CUtensorMap ta, tb;
    if (!make_map(&ta, A16, K, M, lda, TC_BM) || !make_map(&tb, W16, K, N, ldw, wide ? 256 : (narrow ? 64 : 128)))
        return cudaErrorInvalidValue;
    if (narrow) {
        // split K over a cluster when the 128 x 64 tiles leave SMs idle: S CTAs
        // per tile, each with at most 16 k-blocks (one exact chunk); K of at
        // least 8 k-blocks (measured: splitting 4 k-blocks in two was slower)
        const long tiles64 = (long)((M + TC_BM - 1) / TC_BM) * ((N + SK_BN - 1) / SK_BN);
        const int nkb = (K + TC_BK - 1) / TC_BK;
        if (nkb >= 8 && tiles64 * 4 <= g_num_sms && tiles64 <= g_sk_clusters[4])
            return tc_launch_sk<4>(ta, tb, M, N, K, e, status, st);
        if (nkb >= 8 && nkb <= 32 && tiles64 * 2 <= g_num_sms && tiles64 <= g_sk_clusters[2])
            return tc_launch_sk<2>(ta, tb, M, N, K, e, status, st);
    }
    if (narrow && two_chunks) return tc_launch<64, 2, TC_STAGES_NARROW, 2>(ta, tb, M, N, K, e, status, st);
    if (narrow) return tc_launch<64, 1, TC_STAGES_NARROW, 2>(ta, tb, M, N, K, e, status, st);
    if (wide && two_chunks) return tc_launch<256, 2, TC_STAGES_WIDE, 1>(ta, tb, M, N, K, e, status, st);
    if (wide) return tc_launch<256, 1, TC_STAGES_WIDE, 2>(ta, tb, M, N, K, e, status, st);
    if (two_chunks) return tc_launch<128, 2, TC_STAGES, 2>(ta, tb, M, N, K, e, status, st);
    return tc_launch<128, 1, TC_STAGES, 2>(ta, tb, M, N, K, e, status, st);
}

cudaError_t launch_codes_to_f16(const int8_t *src, int ld_src, __half *dst, int ld_dst, int rows, int cols,
                                cudaStream_t st) {
    if (rows <= 0 || cols <= 0) return cudaSuccess;
    if (cols % 16 || ld_src % 16 || ld_dst % 8 || (reinterpret_cast<uintptr_t>(src) & 15) ||
        (reinterpret_cast<uintptr_t>(dst) & 15))
        return cudaErrorInvalidValue;
    const long units = (long)rows * (cols / 16);
    long blocks = (units + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    launch_pdl(codes_to_f16_kernel, (int)blocks, 256, 0, st, src, ld_src, dst, ld_dst, rows, cols);
    return cudaGetLastError();
}

cudaError_t launch_codes_to_f16_flat(const int8_t *src, __half *dst, size_t n, cudaStream_t st) {
    const size_t body = n & ~(size_t)15;
    cudaError_t err = cudaSuccess;
    // the body as rows of 2^20 codes (the row count stays an int)
    const size_t row = (size_t)1 << 20;
    size_t done = 0;
    if (body >= row) {
        err = launch_codes_to_f16(src, (int)row, dst, (int)row, (int)(body / row), (int)row, st);
        done = body / row * row;
    }
    if (err == cudaSuccess && body > done)
        err = launch_codes_to_f16(src + done, (int)(body - done), dst + done, (int)(body - done), 1,
                                  (int)(body - done), st);
    if (err == cudaSuccess && n > body) {
        launch_pdl(codes_to_f16_tail, 1, 32, 0, st, src, dst, body, n);
        err = cudaGetLastError();
    }
    return err;
}

}  // namespace mnmt
