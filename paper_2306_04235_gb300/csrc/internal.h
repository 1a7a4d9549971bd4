// internal.h -- types and kernel launchers shared by the translation units of
// libmnmt (host code + sm_103a kernels).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/mnmt.h"

namespace mnmt {

// Launch with programmatic stream serialisation (see pdl_grid_wait in
// common.cuh): the kernel may launch once every CTA of its predecessor has
// triggered (pdl_allow_next, issued after each kernel's main work -- the
// tensor-core kernels after their last MMA issue, LayerNorm before its store
// pass, the others at exit) and waits for the predecessor's completion before
// it reads or writes anything the predecessor touches.  Inside a stream
// capture the launch is a plain one: the decode-step graphs measured slower
// with programmatic edges between their nodes (wide batched step 711 -> 745
// us with these late triggers, 728 -> 764 us with triggers at kernel start).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                       Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) cs = cudaStreamCaptureStatusNone;
    cfg.attrs = attr;
    cfg.numAttrs = cs == cudaStreamCaptureStatusActive ? 0 : 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// Epilogue of a quantised linear (Sec. 3.3, Fig. 5).  y = fl(fl(acc *
// fl(s_x * s_w[n])) + bias[n]) then, per mode:
enum EpiMode {
    EPI_Q8 = 0,       // out[m*ldo + n] = q8(y, inv_out[n])
    EPI_RELU_Q8 = 1,  // out[m*ldo + n] = q8(max(y, 0), inv_out[n])
    EPI_RESID = 2,    // f32[m*ldf + n] = fl(fl(gamma * f32) + y)
    EPI_F32 = 3,      // f32[m*ldf + n] = y
    EPI_QKV_DEC = 4,  // n < d: out[m*ldo + n] = q8(y); n >= d: K / V cache at position *t_ptr
    EPI_KV_CROSS = 5, // row m = b*S + s: K / V -> cross cache [b][H][S][dh]
    EPI_ARGMAX = 6,   // keys[m] = max over n of pack_key(y, n)   (greedy vocabulary projection)
};

struct Epi {
    int mode;
    float s_x;
    const float *s_w;
    const float *bias;
    const float *inv_out;
    int8_t *out;
    __half *out16;  // EPI_Q8 / EPI_RELU_Q8: optional fp16 copy of out (same layout)
    int ldo;
    float *f32;
    int ldf;
    float gamma;
    // caches (EPI_QKV_DEC: [R][H][T][dh]; EPI_KV_CROSS: [B][H][S][dh])
    int8_t *kc, *vc;
    const int *t_ptr;
    int d, H, dh, T, S;
    unsigned long long *keys;
    const int *skip;  // if non-null and *skip != 0, the kernel does nothing
};

// records msg as the calling thread's mnmt_last_error() and returns code
int set_error(int code, const char *msg);

// ---- one-time kernel attribute set-up (before any launch or capture) ----
cudaError_t linear_init();
cudaError_t attention_init();
cudaError_t rows_init();

// ---- launchers (stream-ordered, no synchronisation) ----
cudaError_t launch_linear(const int8_t *A, int lda, const int8_t *W, int M, int N, int K, const Epi &e,
                          cudaStream_t st);
// row-wise 4-bit weights Wp [N][K/2] (packed runs of 32 codes); m_w: row
// offsets of the min-max form, null for symmetric rows (stored code v + 8)
cudaError_t launch_linear_w4(const int8_t *A, int lda, const uint8_t *Wp, const float *m_w, int M, int N, int K,
                             const Epi &e, cudaStream_t st);
// fake quantisation (QAT forward / backward) and the QAT forward of a linear
cudaError_t launch_fake_quant(const float *x, size_t n, float s, float r, int bits, int minmax, float *y,
                              int32_t *codes, cudaStream_t st);
cudaError_t launch_fake_quant_backward(const float *x, const float *g, size_t n, float s, float r, int bits,
                                       int minmax, float *gx, double *gs, double *gr, cudaStream_t st);
cudaError_t launch_fake_quant_linear(const float *X, const float *W, float s_x, const float *s_w, const float *bias,
                                     int M, int N, int K, int wbits, int8_t *qx, int8_t *qw, float *y,
                                     cudaStream_t st);
// symmetric 4-bit rows (codes elements) unpacked to int8 v = c - 8
cudaError_t launch_unpack_w4_sym(const uint8_t *Wp, size_t codes, int8_t *out, cudaStream_t st);

// tensor-core (tcgen05) linear over fp16 copies of the int8 codes: A16 [M][lda],
// W16 [N][ldw]; K <= 2048 and a multiple of 8; *status (device, may be null)
// receives MNMT_ETIMEOUT if a pipeline wait runs out
cudaError_t linear_tc_init();
int device_sm_count();  // SMs of the current device (read by linear_tc_init)
cudaError_t launch_wait_timeout_selftest(int *status, cudaStream_t st);
bool linear_tc_shape_ok(int M, int N, int K, int lda, int ldw, const void *A16, const void *W16);
cudaError_t launch_linear_tc(const __half *A16, int lda, const __half *W16, int ldw, int M, int N, int K,
                             const Epi &e, int *status, cudaStream_t st);
// int8 codes -> fp16 (exact): rows x cols (cols, ld_src multiples of 16), or flat
cudaError_t launch_codes_to_f16(const int8_t *src, int ld_src, __half *dst, int ld_dst, int rows, int cols,
                                cudaStream_t st);
cudaError_t launch_codes_to_f16_flat(const int8_t *src, __half *dst, size_t n, cudaStream_t st);

struct LnArgs {
    const float *r;   // [M][d] input rows (row stride d)
    float *out_f;     // optional fp32 output (may alias r)
    int8_t *out_q;    // optional int8 output
    __half *out16;    // optional fp16 copy of out_q (tensor-core operand)
    const float *g, *b;
    float inv;
    int M, d;
    int *status;
    const int *skip;
};
cudaError_t launch_layernorm(const LnArgs &a, cudaStream_t st);

struct EmbedArgs {
    const int32_t *ids;   // [M] token ids, or nullptr to use tok (decoder)
    const int32_t *tok;   // decoder tokens [M]
    int S;                // encoder: row m is position m % S; decoder: position *t_ptr
    const int *t_ptr;
    const int8_t *emb_q;
    const float *emb_s;
    const int8_t *proj_w;  // factorised E -> d (nullptr if E == d)
    const float *proj_s, *proj_b;
    float emb_scale;
    const float *pe;
    int M, d, E, V;
    float *r;              // fp32 [M][d] residual out
    int8_t *out_q;         // int8 sublayer input out
    __half *out16;         // optional fp16 copy of out_q (tensor-core operand)
    const float *ln_g, *ln_b;  // if non-null: out_q = q8(LN(x), inv) else q8(x, inv)
    float inv;
    int *status;
    const int *skip;
};
cudaError_t launch_embed(const EmbedArgs &a, cudaStream_t st);

struct AttnDecArgs {
    const int8_t *q;        // [R][d] (head h at h*dh)
    const int8_t *kc, *vc;  // self: [R][H][T][dh]; cross: [B][H][S][dh]
    int8_t *ctx;            // [R][d]
    __half *ctx16;          // optional fp16 copy of ctx (tensor-core operand)
    int R, H, dh, T;        // T = cache capacity (self) or S_pad (cross)
    int cross;              // 0 = self (keys 0..t), 1 = cross (keys < src_len[r / beam])
    int beam;
    const int *t_ptr;       // self: current step (keys 0..t)
    const int *n_keys;      // kernel-level entry: keys per row (overrides t_ptr)
    const int *src_len;     // cross
    const int *anc;         // self, beam > 1: [R][T] physical row of each position (or null)
    float sigma, rho;
    const int *skip;
};
cudaError_t launch_attention_decode(const AttnDecArgs &a, cudaStream_t st);

struct AttnEncArgs {
    const int8_t *qkv;  // [B*S][3d]: q | k | v
    int8_t *ctx;        // [B*S][d]
    __half *ctx16;      // optional fp16 copy of ctx (tensor-core operand)
    const int *len;     // [B]
    int B, S, H, dh, d;
    float sigma, rho;
};
cudaError_t launch_attention_encoder(const AttnEncArgs &a, cudaStream_t st);

// greedy: consume argmax keys, write history / next tokens / finished / done
struct GreedyArgs {
    unsigned long long *keys;  // [R], reset to 0 after reading
    int32_t *tok;              // [R] next input token
    int32_t *fin;              // [R]
    int32_t *hist;             // [T][R]
    int *t_ptr, *done;
    const int *tmax_ptr;       // steps of this translation (device)
    int R, T, eos, pad;
    // cluster step: 1 while a vocabulary kernel's maxima wait in keys for their
    // bookkeeping (done by the next step kernel, or by the greedy update as
    // the flush at the end of a run of steps, which then does nothing when 0)
    int *pending = nullptr;
};
cudaError_t launch_greedy_update(const GreedyArgs &a, cudaStream_t st);

// beam search: per-row log-softmax + top-k, then per-sentence selection
struct BeamArgs {
    const float *logits;       // [R][V]
    int32_t *tok, *fin;        // [R]
    float *cum;                // [R]
    int32_t *hist, *parents;   // [T][R]
    int32_t *anc;              // [R][T]
    unsigned long long *cand;  // [R][k] row candidates
    int *t_ptr, *done, *ticket;   // ticket[0..1]: arrival and running counters
    const int *tmax_ptr;          // steps of this translation (device)
    int B, k, V, T, eos, pad;     // T: cache / history capacity
    int *status;
};
cudaError_t launch_beam_step(const BeamArgs &a, cudaStream_t st);

struct InitArgs {
    int32_t *tok, *fin, *anc, *hist, *parents;
    float *cum;
    unsigned long long *keys;
    int *t_ptr, *done, *ticket;
    int R, k, T, bos, pad;
};
cudaError_t launch_search_init(const InitArgs &a, cudaStream_t st);

struct FinalArgs {
    const int32_t *hist, *parents;
    const float *cum;
    const int *t_ptr;
    int32_t *out_ids, *out_lens;
    float *out_scores;
    int B, k, T, max_len, eos, pad;
};
cudaError_t launch_finalize(const FinalArgs &a, cudaStream_t st);

// ---- decode step of small greedy batches on one thread-block cluster ----
constexpr int DC_RMAX = 4;   // rows (sentences) per step
constexpr int DC_LMAX = 16;  // decoder layers

struct DcLin {
    const int8_t *w;  // int8 codes, or packed 4-bit codes when bits == 4
    const float *s, *b;
    const float *m;   // 4-bit min-max rows: row offsets (else null)
    int bits;         // 8 or 4
};
struct DcLayer {
    const float *ln1_g, *ln1_b, *ln2_g, *ln2_b, *ln3_g, *ln3_b;
    float s_in1, s_ctx1, gamma1, sigma1, rho1;
    float s_in2, s_ctx2, gamma2, sigma2, rho2;
    float s_in3, s_h, gamma3;
    float inv_in1, inv_in2, inv_in3;  // fl(1 / s_in) of the three sublayer inputs
    DcLin qkv, o, q2, o2, w1, w2;
    const float *inv_qkv, *inv_q2, *inv_h;
    int8_t *self_k, *self_v;          // [R][H][T][dh]
    const int8_t *cross_k, *cross_v;  // [B][H][S][dh]
};
// weight slice table of the step's phases (phase 0: factorised embedding
// projection, then per layer qkv, o, q2, o2, w1, w2); CTA c's slice is rows
// [c * rows, (c + 1) * rows) of the [N][K] matrix
struct DcPhase {
    const int8_t *w;             // int8 codes or (bits == 4) packed 4-bit codes
    const float *s, *b, *inv;    // inv: per-column requantisation constants (or null)
    const float *m;              // 4-bit min-max rows: row offsets (else null)
    int rows, K, bits;
    // the exchange of the phase's output: 16-byte chunks per row of a slice
    // (cpr) and ceil(2^32 / d) multipliers for d = R * cpr and d = cpr
    // (quotients of chunk indices below 2^16 by one multiply-high)
    int cpr;
    uint32_t mg_rc, mg_c;
    // the slice GEMV: 2^lg lanes per weight row; the epilogue's input scale
    // and residual gain, and whether it produces fp32 residual values
    int lg, out_f32;
    float sx, gam;
    uint32_t xbytes;  // bytes a CTA receives in the phase's exchange
};
struct alignas(16) DcParams {
    int R, d, H, dh, F, E, V, T, S, n_dec, pre_ln, factorised, nc;
    const int8_t *emb_q;
    const float *emb_s;
    DcLin proj;
    float emb_scale;
    const float *pe;
    const float *fin_g, *fin_b;
    const float *ln_all;  // every LayerNorm vector of the step, contiguous: [n_dec][6][d] then final [2][d]
    float s_dout, inv_dout;  // inv_dout = fl(1 / s_dout)
    const int32_t *tok;
    const int *t_ptr, *done;
    // the previous step's greedy selection, applied by this step (CTA 0 writes)
    unsigned long long *keys;
    int32_t *tok_w, *fin, *hist;
    int *t_w, *done_w, *pending;
    const int *tmax_ptr;
    int eos, pad;
    const int32_t *src_len;
    int8_t *act_out;
    float *resid_out;
    int *status;
    // shared-memory carve-up (bytes), filled by dc_layout
    int off_r, off_a, off_qkv, off_ctx, off_q2, off_h, off_stage, off_att, off_ring, off_ln, off_red, slot_bytes,
        att_cap;
    int kv_staged, off_kvs, off_kvc;
    int stage_bytes;  // one of the two slice staging buffers
    int att_ip, att_lw;  // attention: (row, head) items per round, log2 of warps per item
    int ln_kd, ln_dodd;  // d = ln_dodd 2^ln_kd (ln_dodd odd)
    unsigned long long ln_zm;  // floor(2^64 / ln_dodd) when ln_dodd > 1  // self / cross keys and values staged in shared memory
    int off_part, off_bar;  // off_bar: mbarriers of the weight ring [DC_NB] and of the exchange [2]
    DcLayer layer[DC_LMAX];
    DcPhase phase[1 + 6 * DC_LMAX];
};
static_assert(sizeof(DcParams) % 16 == 0, "the parameter block is copied in 16-byte chunks");
int dc_cluster_size(int d, int F, int E);
size_t dc_layout(DcParams &P, size_t max_smem);
cudaError_t decode_cluster_init();
// one_row: a single-row int8 step (greedy batch 1) takes its own smaller
// kernel; flags: the model's pre-LN (bit 0), factorised-embedding (bit 1) and
// R * d > 256 (bit 2) bits, which such a kernel may have compiled in
bool decode_cluster_fits(int dh, int nc, size_t smem, bool w4, bool one_row, int flags);
cudaError_t launch_decode_cluster(const DcParams *dP, int dh, int nc, size_t smem, bool w4, bool one_row,
                                  int flags, cudaStream_t st);
// reserved_sms: SMs the step kernel that precedes the launch occupies
cudaError_t launch_vocab_greedy(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                                int M, int N, int K, unsigned long long *keys, int *ticket, const GreedyArgs &g,
                                int reserved_sms, cudaStream_t st);

}  // namespace mnmt
