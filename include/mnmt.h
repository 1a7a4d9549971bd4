/*
 * mnmt.h -- C ABI of the GB300 (sm_103a) full-INT8 encoder-decoder translation
 * path of MobileNMT (arXiv 2306.04235).
 *
 * The paper states the problem as: translate a batch of source token ids with
 * an INT8 Transformer encoder-decoder whose weights, activations and embedding
 * are 8-bit (Sec. 3.3, Table 5 "8-8-8"), decoding step by step with greedy
 * search (App. D) or beam search (Table 6).  The calls below follow that
 * statement: load quantised weights and scales, encode a source batch, run
 * decode steps, or translate end to end.
 *
 * Conventions shared by every call
 *   - Return value: MNMT_OK (0) or a negative MNMT_E* code; nothing throws or
 *     traps across the ABI.  mnmt_last_error() returns a thread-local message
 *     describing the last failure on the calling thread.
 *   - A session whose device work failed (a CUDA error or a device-side status
 *     such as MNMT_EOVERFLOW) is poisoned: every later call on it returns the
 *     same code.  Free it and create a new one.
 *   - Ownership: blob and input arrays are borrowed for the duration of the call
 *     (the blob is copied to the device); output arrays are owned by the caller.
 *   - Streams: a model is bound to one CUDA stream (cudaStream_t passed as
 *     void*, NULL = legacy default stream); all its sessions' work is issued on
 *     it.  Models and sessions are not thread-safe.
 *   - Token ids are in [0, vocab); PAD = 0, BOS = 1 (decoder start), EOS = 2
 *     (the ids the blob header carries).
 *
 * MNMT weight blob (little endian).  64-byte header: char magic[4] = "MNMT",
 * uint32 version (1 or 2), int32 config[13] in mnmt_config field order, then
 * (version 2 only) int32 wq at byte 60, zero padding.  wq is the format of the
 * attention and FFN linears (Sec. 3.3, table "quantizing weights to lower
 * bits"): 8 = int8 (version 1), 4 = 4-bit symmetric rows, 0x104 = 4-bit
 * min-max rows (App. B Eq. scale / Eq. quant); see mnmt_linear_w4 for the
 * 4-bit codes.  In a 4-bit linear the codes are packed [N][K/2] and the
 * min-max form stores f32 m[N] (row offsets) between s_w and b.  The
 * embedding table, its factorised projection and an untied output projection
 * (the embedding of W-E-A) are int8 in every format.
 * Then the arrays below in this order, each starting at a 16-byte aligned
 * offset (zero padding between arrays), the blob ending right after the last
 * array's padding.  A "linear" is {int8 W[N][K] (row n = output channel,
 * K contiguous), f32 s_w[N] (per-output-channel weight scale), f32 b[N]}.
 * d = d_model, F = d_ffn, V = vocab, E = d_embed.
 *     int8 emb_q[V][E], f32 emb_s[V]            shared src/tgt embedding codes and row scales
 *     if E != d: linear proj (N = d, K = E)     factorised embedding E -> d
 *     f32 globals[4] = {emb_scale, s_enc, s_dout, 0}
 *     f32 pe[max_pos][d]                        positional table
 *     n_enc x { self-attention block, FFN block }
 *     if pre_ln: f32 enc_ln_g[d], enc_ln_b[d]   final encoder LayerNorm
 *     n_dec x { self-attention block, cross-attention block, FFN block }
 *     if pre_ln: f32 dec_ln_g[d], dec_ln_b[d]   final decoder LayerNorm
 *     if !tied_output: int8 out_w[V][d], f32 out_s[V]
 *     f32 out_b[V]
 *   self-attention block:  f32 ln_g[d], ln_b[d];
 *                          f32 s[8] = {s_in, s_q, s_k, s_v, s_ctx, gamma, 0, 0};
 *                          linear qkv (N = 3d, rows q | k | v, K = d); linear o (N = d, K = d)
 *   cross-attention block: f32 ln_g[d], ln_b[d]; f32 s[8] (as above; s_k, s_v
 *                          quantise the cross keys/values); linear q (d x d);
 *                          linear kv (N = 2d, rows k | v, K = d; input is the
 *                          quantised encoder output at scale s_enc); linear o (d x d)
 *   FFN block:             f32 ln_g[d], ln_b[d]; f32 s[4] = {s_in, s_h, gamma, 0};
 *                          linear w1 (N = F, K = d); linear w2 (N = d, K = F)
 *   With tied_output the output projection is emb_q / emb_s (requires E = d).
 *   Scales s_* are the per-tensor activation scales of the quantisation points
 *   of Fig. 5; pre_ln = 0 selects post-LN sublayers (LayerNorm after the
 *   residual add, no final LayerNorm).  Constraints checked at load: d_model a
 *   multiple of 64 in [64, 2048], d_ffn a multiple of 64, d_embed a multiple of
 *   16, d_model / n_heads in {32, 64, 128}, at most 16 heads, vocab >= 4.
 */
#ifndef MNMT_H
#define MNMT_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    MNMT_OK = 0,
    MNMT_EINVAL = -1,    /* bad argument (size, id, pointer, flag) */
    MNMT_ENOMEM = -2,    /* device or host allocation failed */
    MNMT_ECUDA = -3,     /* a CUDA runtime call failed */
    MNMT_ETIMEOUT = -4,  /* a bounded device wait gave up */
    MNMT_EFORMAT = -5,   /* malformed weight blob */
    MNMT_EOVERFLOW = -6  /* a LayerNorm input left the fixed-point domain (|x| >= 2^32) */
};

/* flags of mnmt_encode / mnmt_translate */
#define MNMT_DEVICE_PTRS 1 /* id/length inputs and translate outputs are device pointers */

typedef struct {
    int32_t n_enc, n_dec, d_model, n_heads, d_ffn, vocab, d_embed, pre_ln, tied_output, max_pos,
        pad_id, bos_id, eos_id;
} mnmt_config;

typedef struct mnmt_model mnmt_model;     /* owns the device copy of the weights */
typedef struct mnmt_session mnmt_session; /* owns caches, workspace and search state */

/* Host-only validation of a blob (no CUDA call).  Fills *cfg_out on success.
 * Returns MNMT_EFORMAT for a malformed blob. */
int mnmt_blob_check(const void *blob, size_t bytes, mnmt_config *cfg_out);

/* Quantised weights and scales (Sec. 3.3, Fig. 5): validates the blob, copies
 * it to the device and derives the per-column requantisation constants.
 * cuda_stream: cudaStream_t the model and its sessions run on.
 * *out receives the model on success. */
int mnmt_load_weights(const void *blob, size_t bytes, void *cuda_stream, mnmt_model **out);

/* Memory-minimal operation (Sec. 4 "Memory Optimization"; the running memory
 * column of Table 2).  MNMT_LOAD_LEAN keeps only the int8 blob and the derived
 * per-column constants on the device (no fp16 copy of the weight codes): every
 * linear of the model's sessions runs on the int8 GEMV / IMMA kernels, with
 * results identical to the default load.  flags = 0 is mnmt_load_weights.
 * MNMT_EINVAL for unknown flags. */
#define MNMT_LOAD_LEAN 1
int mnmt_load_weights_ex(const void *blob, size_t bytes, void *cuda_stream, int32_t flags, mnmt_model **out);
void mnmt_model_free(mnmt_model *model);
int mnmt_model_config(const mnmt_model *model, mnmt_config *cfg_out);

/* A session sized for up to max_batch sentences of up to max_src_len tokens,
 * beam width `beam` (1 = greedy, 2..16 = beam search) and up to max_len decode
 * steps (max_len <= max_pos).  Allocates all device memory the session uses;
 * no later call allocates. */
int mnmt_session_create(mnmt_model *model, int32_t max_batch, int32_t max_src_len, int32_t beam,
                        int32_t max_len, mnmt_session **out);

/* mnmt_session_create with flags.  MNMT_SESSION_LEAN shares the activation
 * memory the way the paper's engine does (Sec. 4: operations that are never
 * live at the same time share one buffer): the encoder and the decoder step
 * use two int8 buffers -- LayerNorm output / attention context, and QKV
 * output / FFN hidden -- plus the fp32 residual stream, and no fp16 mirrors
 * (every linear on the int8 kernels).  Results are identical to the default
 * session.  MNMT_EINVAL for unknown flags. */
#define MNMT_SESSION_LEAN 1
int mnmt_session_create_ex(mnmt_model *model, int32_t max_batch, int32_t max_src_len, int32_t beam,
                           int32_t max_len, int32_t flags, mnmt_session **out);
void mnmt_session_free(mnmt_session *s);

/* Device bytes held by a model (blob, derived constants, fp16 operand copy
 * unless lean) or by a session (its one arena: caches, activations, search
 * state).  Nothing else is allocated on the device by the library after these
 * objects are created, so model + session bytes are the library's peak device
 * memory for a translation.  Negative MNMT_EINVAL for a null handle. */
int64_t mnmt_model_device_bytes(const mnmt_model *model);
int64_t mnmt_session_device_bytes(const mnmt_session *s);

/* Encoder (App. A): src_ids [B][S_pad] right-padded with PAD, src_lens [B]
 * (1 <= len <= S_pad).  Runs the encoder stack and the cross-attention key /
 * value projections of every decoder layer, then resets the search state
 * (every hypothesis starts from BOS at step 0).  Asynchronous on the model's
 * stream. */
int mnmt_encode(mnmt_session *s, const int32_t *src_ids, const int32_t *src_lens, int32_t B,
                int32_t S_pad, int32_t flags);

/* Queues n incremental decoder steps (at most the steps left before max_len)
 * on the model's stream and returns without waiting: the steps run back to
 * back with no host round trip between them, and steps after every sentence
 * has finished do nothing.  Read the outcome with mnmt_debug_tap
 * (MNMT_TAP_HISTORY / MNMT_TAP_PARENTS) or a later mnmt_decode_step.  Returns
 * the number of steps queued, or a negative error code. */
int mnmt_decode_steps(mnmt_session *s, int32_t n);

/* One incremental decoder step for every hypothesis (greedy or beam), then
 * synchronises.  Host outputs, each NULL to skip: tokens [B*beam] (token
 * chosen at this step per hypothesis), parents [B*beam] (beam index within the
 * sentence it extends), scores [B*beam] (cumulative log-probability; 0 for
 * greedy); *all_done = 1 once every sentence has finished.  Returns
 * MNMT_EINVAL after max_len steps. */
int mnmt_decode_step(mnmt_session *s, int32_t *tokens, int32_t *parents, float *scores,
                     int32_t *all_done);

/* encode + decode until every sentence has emitted EOS or max_len steps ran.
 * The beam width is the session's (fixed by mnmt_session_create): translating
 * with another width needs another session.  max_len may not exceed the
 * session's. 
 * out_ids [B][max_len]: tokens of the best hypothesis, EOS included, PAD after;
 * out_lens [B]: number of tokens up to and including EOS (max_len if none);
 * out_scores [B]: cumulative log-probability of the best beam (0 for greedy).
 * With MNMT_DEVICE_PTRS all five arrays are device pointers and the call is
 * asynchronous apart from the periodic completion check; otherwise they are
 * host pointers and the call returns after the results are copied back. */
int mnmt_translate(mnmt_session *s, const int32_t *src_ids, const int32_t *src_lens, int32_t B,
                   int32_t S_pad, int32_t max_len, int32_t flags, int32_t *out_ids,
                   int32_t *out_lens, float *out_scores);

/* Copies an intermediate tensor of the last encode / decode step to host
 * memory for parity checks.  Returns MNMT_EINVAL if `bytes` differs from the
 * tap's size (query the size with host_dst = NULL: the size is returned as
 * a positive value).
 *   MNMT_TAP_ENC_OUT    int8  [B][S_pad][d]       quantised encoder output
 *   MNMT_TAP_CROSS_K/V  int8  [B][H][S_pad][dh]   cross keys/values of decoder layer `layer`
 *   MNMT_TAP_SELF_K/V   int8  [B*beam][H][max_len][dh] self-attention cache of layer `layer`
 *                             (rows are physical cache rows; beam search reads them
 *                              through MNMT_TAP_ANCESTRY)
 *   MNMT_TAP_DEC_OUT    int8  [B*beam][d]         quantised decoder output of the last step
 *   MNMT_TAP_LOGITS     f32   [B*beam][vocab]     logits of the last step (beam search only)
 *   MNMT_TAP_RESID      f32   [rows][d]           residual stream (encoder rows after encode,
 *                                                  decoder rows after a step)
 *   MNMT_TAP_HISTORY    int32 [max_len][B*beam]   token chosen per step and hypothesis
 *   MNMT_TAP_PARENTS    int32 [max_len][B*beam]   parent beam per step and hypothesis
 *   MNMT_TAP_ANCESTRY   int32 [B*beam][max_len]   physical cache row holding each position */
enum {
    MNMT_TAP_ENC_OUT = 1,
    MNMT_TAP_CROSS_K = 2,
    MNMT_TAP_CROSS_V = 3,
    MNMT_TAP_SELF_K = 4,
    MNMT_TAP_SELF_V = 5,
    MNMT_TAP_DEC_OUT = 6,
    MNMT_TAP_LOGITS = 7,
    MNMT_TAP_RESID = 8,
    MNMT_TAP_HISTORY = 9,
    MNMT_TAP_PARENTS = 10,
    MNMT_TAP_ANCESTRY = 11
};
int64_t mnmt_debug_tap(mnmt_session *s, int32_t tap, int32_t layer, void *host_dst, size_t bytes);

/* Which decode-step implementation the session uses for the batch encoded
 * last: 1 = the single thread-block-cluster step (greedy batches of at most 4
 * sentences whose shapes fit one cluster's shared memory), 0 = the multi-kernel
 * step; negative on error.  Setting MNMT_DECODE_CLUSTER=0 in the environment
 * before the first decode of a batch forces the multi-kernel step.  Both give
 * bit-identical results. */
int mnmt_session_decode_path(mnmt_session *s);

/* Thread-local description of the last error on this thread ("" if none). */
const char *mnmt_last_error(void);

/* ---------------------------------------------------------------------------
 * Kernel-level entry points (microbenchmarks and per-kernel parity).  All
 * pointers are device pointers; work is queued on `cuda_stream` and the call
 * returns without synchronising.  They allocate nothing.
 * ------------------------------------------------------------------------- */

/* Quantised linear with a fused epilogue (Sec. 3.3, Fig. 5; Eq. 3):
 *   acc[m][n] = sum_k A[m][k] W[n][k]  (int8 x int8 -> exact int32)
 *   y = fl(fl(acc * fl(s_x * s_w[n])) + bias[n])
 *   mode MNMT_EPI_Q8:      out_q[m][n] = q8(y, inv_out[n])
 *        MNMT_EPI_RELU_Q8: out_q[m][n] = q8(max(y, 0), inv_out[n])
 *        MNMT_EPI_RESID:   out_f[m][n] = fl(fl(gamma * out_f[m][n]) + y)
 *        MNMT_EPI_F32:     out_f[m][n] = y
 * q8(x, inv) = clamp(round_half_even(fl(x * inv)), -127, 127).
 * A [M][K], W [N][K] row-major int8 with K a multiple of 64 (16 when M <= 16),
 * both 16-byte aligned; s_w, bias, inv_out [N] fp32; out_q int8 / out_f fp32
 * [M][N]. */
enum { MNMT_EPI_Q8 = 0, MNMT_EPI_RELU_Q8 = 1, MNMT_EPI_RESID = 2, MNMT_EPI_F32 = 3 };
int mnmt_linear(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                const float *inv_out, float gamma, int32_t M, int32_t N, int32_t K, int32_t mode,
                int8_t *out_q, float *out_f, void *cuda_stream);

/* Tensor-core form of mnmt_linear for layers where the batch makes the linear
 * a dense contraction: the same results bit for bit, computed on the
 * fifth-generation tensor cores (tcgen05) from fp16 copies of the int8 codes.
 * A16 [M][K] and W16 [N][K] hold fp16 bit patterns of integers in [-128, 127]
 * (mnmt_codes_to_f16 makes them); products of such integers and sums of 1024
 * of them are exact in fp32, so the kernel accumulates K in chunks of 1024 and
 * the result equals the int32 accumulator of mnmt_linear.  K a multiple of 8 in
 * [8, 2048]; A16 and W16 16-byte aligned.  mode is one of mnmt_linear's, or
 * MNMT_EPI_ARGMAX: keys[m] = max(keys[m], max over n of pack(y[m][n], n)) as in
 * mnmt_linear_argmax (keys must be initialised by the caller).  *status
 * (device int32, may be NULL) receives MNMT_ETIMEOUT if one of the kernel's
 * pipeline waits runs out (one second); the affected tiles are then not
 * written. */
enum { MNMT_EPI_ARGMAX = 4 };
int mnmt_linear_tc(const uint16_t *A16, const uint16_t *W16, const float *s_w, const float *bias, float s_x,
                   const float *inv_out, float gamma, int32_t M, int32_t N, int32_t K, int32_t mode,
                   int8_t *out_q, float *out_f, uint64_t *keys, int32_t *status, void *cuda_stream);

/* Quantised linear with row-wise 4-bit weights (Sec. 3.3: low-bit weights are
 * quantised row-wise; table "quantizing weights to lower bits", 4-8-8).
 * Wp [N][K/2] holds each row's K codes packed in runs of 32 codes per 16
 * bytes: code j of a run in the low nibble of byte j (j < 16), code 16 + j in
 * the high nibble of byte j.  m_w == NULL: symmetric rows, stored code
 * c = v + 8 for v in [-7, 7], W[n][k] = s_w[n] v, and every mode is exactly
 * mnmt_linear's on the codes v.  m_w != NULL: min-max rows (App. B Eq. scale /
 * Eq. quant), code u in [0, 15], W[n][k] = s_w[n] u + m_w[n]; with
 * A_u = sum_k A[m][k] u and A_1 = sum_k A[m][k] (exact int32)
 *   y = fl(fl(fl(A_u fl(s_x s_w[n])) + fl(A_1 fl(s_x m_w[n]))) + bias[n]),
 * then mode as in mnmt_linear, or MNMT_EPI_ARGMAX into keys (as in
 * mnmt_linear_tc).  K a multiple of 32 in [32, 3072]; A and Wp 16-byte
 * aligned; any M (rows beyond 16 are taken 16 at a time). */
int mnmt_linear_w4(const int8_t *A, const uint8_t *Wp, const float *s_w, const float *m_w, const float *bias,
                   float s_x, const float *inv_out, float gamma, int32_t M, int32_t N, int32_t K, int32_t mode,
                   int8_t *out_q, float *out_f, uint64_t *keys, void *cuda_stream);

/* Fake quantisation for quantisation-aware training (App. B "PTQ and QAT":
 * the quantiser of Eq. quant inserted into the float model; besides the
 * weights, its scale s is learnable).  Element-wise over x [n] (fp32):
 *   minmax = 0: q = clamp(rne(fl(x fl(1/s))), -(2^(bits-1)-1), 2^(bits-1)-1),
 *               y = fl(q s)
 *   minmax = 1: q = clamp(rne(fl(fl(x - r_m) fl(1/s))), 0, 2^bits - 1),
 *               y = fl(fl(q s) + r_m)            (Eq. scale / Eq. quant)
 * y [n] (fp32) and codes [n] (int32) are optional outputs (at least one).
 * 2 <= bits <= 8, s > 0 finite.  Device pointers; asynchronous on cuda_stream. */
int mnmt_fake_quant(const float *x, size_t n, float s, float r_m, int32_t bits, int32_t minmax, float *y,
                    int32_t *codes, void *cuda_stream);

/* Backward of mnmt_fake_quant for the upstream gradient g [n]: with t the
 * unrounded code and in = (qmin <= t <= qmax), gx = in ? g : 0 (straight
 * through), *gs = sum g (in ? q - t : q) (the learnable scale's gradient),
 * *gr = sum g (1 - in) (the offset's, min-max form; 0 otherwise).  gs / gr are
 * device doubles (gr may be NULL), accumulated in fp64 (summation order not
 * fixed). */
int mnmt_fake_quant_backward(const float *x, const float *g, size_t n, float s, float r_m, int32_t bits,
                             int32_t minmax, float *gx, double *gs, double *gr, void *cuda_stream);

/* QAT forward of one linear: X [M][K] fp32 fake-quantised per tensor to 8-bit
 * symmetric codes at s_x, W [N][K] fp32 per row to `wbits`-bit symmetric codes
 * at the learnable row scales s_w [N]; y [M][N] fp32 = X_q W_q^T + bias with the
 * products exact, i.e. mnmt_linear's MNMT_EPI_F32 on the two code tensors.
 * workspace: caller-allocated device scratch of at least
 * round_up(M*K, 16) + N*K bytes, 16-byte aligned, holding the codes.  K a
 * multiple of 16 (of 64 when M > 16), K <= 2048 when M <= 16. */
int mnmt_fake_quant_linear(const float *X, const float *W, float s_x, const float *s_w, const float *bias,
                           int32_t M, int32_t N, int32_t K, int32_t wbits, void *workspace, float *y,
                           void *cuda_stream);

/* dst[i] = the fp16 value of the int8 code src[i] (exact), i < n.  Device
 * pointers, src and dst 16-byte aligned. */
int mnmt_codes_to_f16(const int8_t *src, uint16_t *dst, size_t n, void *cuda_stream);

/* Diagnostic of the bounded waits of the tensor-core pipelines: one thread
 * block waits on a shared-memory transaction barrier that nothing completes.
 * The wait gives up after one second (the limit of every such wait in
 * mnmt_linear_tc), the kernel records MNMT_ETIMEOUT in *status (device int32,
 * required) and returns; no fault is raised and the context stays usable.
 * Returns once the kernel is queued. */
int mnmt_wait_timeout_selftest(int32_t *status, void *cuda_stream);

/* Output-vocabulary projection fused with greedy selection (App. D): for each
 * row m, keys[m] = max over n of pack(y[m][n], n) with y as in mnmt_linear and
 * pack(y, n) = (ord(y) << 32) | (0xFFFFFFFF - n), where ord maps fp32 to uint32
 * monotonically (-0 as +0).  The winning id is 0xFFFFFFFF - (keys[m] & 0xFFFFFFFF):
 * the largest logit, ties to the lowest id.  keys [M] (uint64) must hold 0
 * before the call (the kernel combines with atomicMax).  A [M][K], W [N][K] as
 * in mnmt_linear. */
int mnmt_linear_argmax(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                       int32_t M, int32_t N, int32_t K, uint64_t *keys, void *cuda_stream);

/* The call above without any caller-provided scratch, for callers that cannot
 * allocate device memory (their device memory is owned by another allocator or
 * a fixed budget, or they run on a latency-critical thread where cudaMalloc's
 * implicit synchronisation is not acceptable).  The paper has no counterpart:
 * this is a deployment variant of the fused vocabulary projection + argmax.
 * ids [M] (int32, device) receives the argmax id of each row, ties to the
 * lowest id; A, W, s_w, bias as in mnmt_linear_argmax.  The packed keys live in
 * a library-owned 32 KB device array (4096 rows), so M must be in [1, 4096]
 * (MNMT_EINVAL otherwise).  Nothing is allocated: the array is part of the
 * loaded library on every GPU that uses it, until the process exits.  The
 * first call on a device looks up the array's address and sets up the GEMM
 * kernels on that device; make that first call before any stream capture.
 * Every call shares the one array: calls whose GPU work overlaps (different
 * streams or threads without ordering) race and may return wrong ids. */
int mnmt_linear_argmax_ids_noalloc(const int8_t *A, const int8_t *W, const float *s_w, const float *bias,
                                   float s_x, int32_t M, int32_t N, int32_t K, int32_t *ids, void *cuda_stream);

/* Incremental attention (Eq. 1/2 per head) of R query rows over per-row
 * caches: q [R][H][dh], Kc/Vc [R][H][T][dh] int8; row r attends keys
 * j < n_keys[r] (1 <= n_keys[r] <= T <= 1024).  Scores acc_j = q.k_j (int32),
 * s_j = fl(acc_j * sigma); weights E_j = rne(exp(fl(s_j - max)) 2^24);
 * ctx[r][h][e] = q8(nearest fp32 to (sum_j E_j v_j[e]) / (sum_j E_j), rho),
 * with the sums exact integers.  dh in {32, 64, 128}. */
int mnmt_attention_decode(const int8_t *q, const int8_t *Kc, const int8_t *Vc, const int32_t *n_keys,
                          int32_t R, int32_t H, int32_t dh, int32_t T, float sigma, float rho,
                          int8_t *ctx, void *cuda_stream);

/* LayerNorm of M rows of length d (App. A / App. D) with optional fp32 output
 * out_f [M][d] and int8 output out_q = q8(LN(r), inv) (either may be NULL).
 * Mean and biased variance are exact fixed-point sums on a grid set by each
 * row's largest magnitude; eps = 1e-5.  *status (device int, may be NULL)
 * receives MNMT_EOVERFLOW if a row holds |x| >= 2^32. */
int mnmt_layernorm(const float *r, const float *g, const float *b, int32_t M, int32_t d, float inv,
                   float *out_f, int8_t *out_q, int32_t *status, void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* MNMT_H */
