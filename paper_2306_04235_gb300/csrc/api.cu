// api.cu -- host runtime and C ABI of libmnmt (include/mnmt.h).
//
// Model: the MNMT v1 blob is validated on the host, copied to the device once
// (every array keeps its 16-byte aligned blob offset, so int8 weight rows stay
// K-contiguous in HBM) and the per-column requantisation constants
// inv_out[n] = fl(1 / s_out) and the attention constants sigma, rho are derived
// on the host.
//
// Session: one device arena holds the residual stream, int8 activations, the
// int8 self- and cross-attention caches and the search state; nothing is
// allocated after mnmt_session_create.  The decoder step (embedding, every
// decoder layer, the vocabulary projection and the search update) is captured
// once per (batch, padded source length) as a CUDA graph and replayed; every
// kernel of a step reads the step counter from device memory and returns at
// once when the search is done, so extra replays are cheap.
#include <cuda_runtime.h>

#include <cmath>
#include <cstddef>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "internal.h"

using namespace mnmt;

// ---------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------
static thread_local std::string g_err;

static int fail(int code, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    g_err = buf;
    return code;
}

#define CK(call)                                                                                  \
    do {                                                                                          \
        cudaError_t e_ = (call);                                                                  \
        if (e_ != cudaSuccess)                                                                    \
            return fail(MNMT_ECUDA, "%s failed: %s (%s:%d)", #call, cudaGetErrorString(e_), __FILE__, \
                        __LINE__);                                                                \
    } while (0)

// Kernel set-up (dynamic shared-memory opt-ins, the SM count) applies to the
// device current at the time, so it runs once for every device a call is
// made on, with that device current.
static std::mutex g_init_mu;
static constexpr int MAX_INIT_DEVICES = 64;
static bool g_init_done[MAX_INIT_DEVICES] = {false};

static int lib_init() {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return fail(MNMT_ECUDA, "no usable current device: %s", cudaGetErrorString(e));
    if (dev < 0 || dev >= MAX_INIT_DEVICES) return fail(MNMT_ECUDA, "device index %d out of range", dev);
    std::lock_guard<std::mutex> lk(g_init_mu);
    if (g_init_done[dev]) return MNMT_OK;
    e = linear_init();
    if (e == cudaSuccess) e = attention_init();
    if (e == cudaSuccess) e = rows_init();
    if (e == cudaSuccess) e = decode_cluster_init();
    if (e == cudaSuccess) e = linear_tc_init();
    if (e != cudaSuccess) return fail(MNMT_ECUDA, "kernel set-up failed: %s", cudaGetErrorString(e));
    g_init_done[dev] = true;
    return MNMT_OK;
}

// ---------------------------------------------------------------------------
// blob layout (host walk over the documented MNMT v1 order)
// ---------------------------------------------------------------------------
namespace {

constexpr int WQ_MINMAX = 0x100;  // blob v2: 4-bit rows with a min-max scale and offset

struct LinOff {
    size_t w, s, b, m;
    int n, k, bits;
    bool minmax;
};
struct SelfOff {
    size_t ln_g, ln_b, sc;
    LinOff qkv, o;
};
struct CrossOff {
    size_t ln_g, ln_b, sc;
    LinOff q, kv, o;
};
struct FfnOff {
    size_t ln_g, ln_b, sc;
    LinOff w1, w2;
};
struct Layout {
    mnmt_config c;
    int wq;  // weight format of the attention / FFN linears: 8, 4, or 4 | WQ_MINMAX
    size_t emb_q, emb_s, globals, pe, enc_ln_g, enc_ln_b, dec_ln_g, dec_ln_b, out_w, out_s, out_b;
    LinOff proj;
    std::vector<SelfOff> enc_self, dec_self;
    std::vector<FfnOff> enc_ffn, dec_ffn;
    std::vector<CrossOff> dec_cross;
};

struct Walker {
    size_t off, size;
    bool bad;
    size_t take(size_t n) {
        if (bad || n > size || off > size - n) {
            bad = true;
            return 0;
        }
        size_t at = off;
        off = (off + n + 15) & ~(size_t)15;
        if (off > size) off = size;
        return at;
    }
    // a linear of format wq: codes (int8 [n][k], or 4-bit packed [n][k/2]),
    // row scales, row offsets (min-max form only), biases
    LinOff lin(int n, int k, int wq = 8) {
        LinOff l;
        l.n = n;
        l.k = k;
        l.bits = wq & 0xFF;
        l.minmax = (wq & WQ_MINMAX) != 0;
        l.w = take(l.bits == 4 ? (size_t)n * k / 2 : (size_t)n * k);
        l.s = take((size_t)n * 4);
        l.m = l.minmax ? take((size_t)n * 4) : 0;
        l.b = take((size_t)n * 4);
        return l;
    }
};

bool pow2_in(int v, int lo, int hi) { return v >= lo && v <= hi && (v & (v - 1)) == 0; }

int parse_layout(const void *blob, size_t bytes, Layout *L) {
    if (!blob || bytes < 64) return fail(MNMT_EFORMAT, "blob shorter than its 64-byte header");
    const uint8_t *p = static_cast<const uint8_t *>(blob);
    if (std::memcmp(p, "MNMT", 4) != 0) return fail(MNMT_EFORMAT, "bad magic");
    uint32_t ver;
    std::memcpy(&ver, p + 4, 4);
    if (ver != 1 && ver != 2) return fail(MNMT_EFORMAT, "unsupported blob version %u", ver);
    L->wq = 8;
    if (ver == 2) std::memcpy(&L->wq, p + 60, 4);
    if (L->wq != 8 && L->wq != 4 && L->wq != (4 | WQ_MINMAX))
        return fail(MNMT_EFORMAT, "unsupported weight format 0x%x", L->wq);
    int32_t h[13];
    std::memcpy(h, p + 8, sizeof(h));
    mnmt_config &c = L->c;
    c.n_enc = h[0]; c.n_dec = h[1]; c.d_model = h[2]; c.n_heads = h[3]; c.d_ffn = h[4];
    c.vocab = h[5]; c.d_embed = h[6]; c.pre_ln = h[7]; c.tied_output = h[8]; c.max_pos = h[9];
    c.pad_id = h[10]; c.bos_id = h[11]; c.eos_id = h[12];
    const int d = c.d_model, F = c.d_ffn, V = c.vocab, E = c.d_embed;
    if (c.n_enc < 1 || c.n_enc > 64 || c.n_dec < 1 || c.n_dec > 64) return fail(MNMT_EFORMAT, "layer counts out of range");
    if (d < 64 || d > 2048 || d % 64 || c.n_heads < 1 || d % c.n_heads)
        return fail(MNMT_EFORMAT, "d_model %d / heads %d unsupported (d_model: a multiple of 64 in [64, 2048])", d,
                    c.n_heads);
    if (!pow2_in(d / c.n_heads, 32, 128)) return fail(MNMT_EFORMAT, "head dim %d not in {32,64,128}", d / c.n_heads);
    if (c.n_heads > 16) return fail(MNMT_EFORMAT, "more than 16 heads");
    if (F < 64 || F % 64 || F > 8192) return fail(MNMT_EFORMAT, "d_ffn %d unsupported", F);
    if (V < 4 || E < 16 || E % 16 || E > d) return fail(MNMT_EFORMAT, "vocab / d_embed out of range");
    if (c.tied_output && E != d) return fail(MNMT_EFORMAT, "tied output needs d_embed == d_model");
    if (c.max_pos < 1 || c.max_pos > 1024) return fail(MNMT_EFORMAT, "max_pos out of range");
    for (int id : {c.pad_id, c.bos_id, c.eos_id})
        if (id < 0 || id >= V) return fail(MNMT_EFORMAT, "special id out of range");
    Walker w{64, bytes, false};
    L->emb_q = w.take((size_t)V * E);
    L->emb_s = w.take((size_t)V * 4);
    if (E != d) L->proj = w.lin(d, E);
    L->globals = w.take(16);
    L->pe = w.take((size_t)c.max_pos * d * 4);
    auto self_blk = [&]() {
        SelfOff s;
        s.ln_g = w.take((size_t)d * 4);
        s.ln_b = w.take((size_t)d * 4);
        s.sc = w.take(32);
        s.qkv = w.lin(3 * d, d, L->wq);
        s.o = w.lin(d, d, L->wq);
        return s;
    };
    auto ffn_blk = [&]() {
        FfnOff f;
        f.ln_g = w.take((size_t)d * 4);
        f.ln_b = w.take((size_t)d * 4);
        f.sc = w.take(16);
        f.w1 = w.lin(F, d, L->wq);
        f.w2 = w.lin(d, F, L->wq);
        return f;
    };
    for (int l = 0; l < c.n_enc; l++) {
        L->enc_self.push_back(self_blk());
        L->enc_ffn.push_back(ffn_blk());
    }
    if (c.pre_ln) {
        L->enc_ln_g = w.take((size_t)d * 4);
        L->enc_ln_b = w.take((size_t)d * 4);
    }
    for (int l = 0; l < c.n_dec; l++) {
        L->dec_self.push_back(self_blk());
        CrossOff x;
        x.ln_g = w.take((size_t)d * 4);
        x.ln_b = w.take((size_t)d * 4);
        x.sc = w.take(32);
        x.q = w.lin(d, d, L->wq);
        x.kv = w.lin(2 * d, d, L->wq);
        x.o = w.lin(d, d, L->wq);
        L->dec_cross.push_back(x);
        L->dec_ffn.push_back(ffn_blk());
    }
    if (c.pre_ln) {
        L->dec_ln_g = w.take((size_t)d * 4);
        L->dec_ln_b = w.take((size_t)d * 4);
    }
    if (!c.tied_output) {
        L->out_w = w.take((size_t)V * d);
        L->out_s = w.take((size_t)V * 4);
    } else {
        L->out_w = L->emb_q;
        L->out_s = L->emb_s;
    }
    L->out_b = w.take((size_t)V * 4);
    if (w.bad || w.off != bytes) return fail(MNMT_EFORMAT, "blob size does not match its config");
    return MNMT_OK;
}

}  // namespace

// ---------------------------------------------------------------------------
// model
// ---------------------------------------------------------------------------
namespace {
struct Lin {
    const int8_t *w;  // int8 codes [n][k] (4-bit symmetric rows: the unpacked copy, or null when lean)
    const float *s, *b;
    int n, k;
    int bits;                 // 8 or 4
    const uint8_t *wp;        // 4-bit: packed codes [n][k/2]
    const float *m;           // 4-bit min-max rows: row offsets (null: symmetric)
};
struct LnP {
    const float *g, *b;
};
struct SelfBlk {
    LnP ln;
    float s_in, s_q, s_k, s_v, s_ctx, gamma, sigma, rho;
    Lin qkv, o;
    const float *inv_qkv;
};
struct CrossBlk {
    LnP ln;
    float s_in, s_q, s_k, s_v, s_ctx, gamma, sigma, rho;
    Lin q, kv, o;
    const float *inv_q, *inv_kv;
};
struct FfnBlk {
    LnP ln;
    float s_in, s_h, gamma;
    Lin w1, w2;
    const float *inv_h;
};
}  // namespace

struct mnmt_model {
    mnmt_config c;
    cudaStream_t stream;
    bool own_stream;
    uint8_t *d_blob;
    __half *d_blob16;  // fp16 copy of every blob byte read as an int8 code (tensor-core operands); null when lean
    int wq;            // weight format of the attention / FFN linears (8, 4, 4 | WQ_MINMAX)
    int8_t *d_w8;      // symmetric 4-bit linears unpacked to int8 (the IMMA / tensor-core operands); null when lean
    __half *d_w8_16;   // its fp16 copy
    size_t w8_codes;
    float *d_aux;
    size_t bytes;
    size_t device_bytes;  // every byte of device memory the model holds
    bool lean;            // loaded with MNMT_LOAD_LEAN: int8 blob only, no fp16 operand copy
    const int8_t *emb_q;
    const float *emb_s;
    bool factorised;
    Lin proj;
    float emb_scale, s_enc, s_dout;
    const float *pe;
    std::vector<SelfBlk> enc_self, dec_self;
    std::vector<CrossBlk> dec_cross;
    std::vector<FfnBlk> enc_ffn, dec_ffn;
    LnP enc_final, dec_final;
    Lin out;
};

static float host_sigma(float s_q, float s_k, int dh) {
    return (float)((double)s_q * (double)s_k / std::sqrt((double)dh));
}

extern "C" int mnmt_blob_check(const void *blob, size_t bytes, mnmt_config *cfg_out) {
    Layout L;
    int st = parse_layout(blob, bytes, &L);
    if (st) return st;
    if (cfg_out) *cfg_out = L.c;
    return MNMT_OK;
}

extern "C" int mnmt_model_config(const mnmt_model *m, mnmt_config *cfg_out) {
    if (!m || !cfg_out) return fail(MNMT_EINVAL, "null argument");
    *cfg_out = m->c;
    return MNMT_OK;
}

extern "C" int mnmt_load_weights(const void *blob, size_t bytes, void *cuda_stream, mnmt_model **out) {
    return mnmt_load_weights_ex(blob, bytes, cuda_stream, 0, out);
}

extern "C" int mnmt_load_weights_ex(const void *blob, size_t bytes, void *cuda_stream, int32_t flags,
                                    mnmt_model **out) {
    if (!out) return fail(MNMT_EINVAL, "out is null");
    *out = nullptr;
    if (flags & ~MNMT_LOAD_LEAN) return fail(MNMT_EINVAL, "unknown load flags 0x%x", flags);
    Layout L;
    int st = parse_layout(blob, bytes, &L);
    if (st) return st;
    if ((st = lib_init())) return st;
    mnmt_model *m = new (std::nothrow) mnmt_model();
    if (!m) return fail(MNMT_ENOMEM, "host allocation failed");
    m->c = L.c;
    m->bytes = bytes;
    m->lean = (flags & MNMT_LOAD_LEAN) != 0;
    if (cuda_stream) {
        m->stream = static_cast<cudaStream_t>(cuda_stream);
        m->own_stream = false;
    } else {
        // the legacy default stream cannot be captured into a graph: use a
        // blocking stream of our own, ordered with the legacy stream
        if (cudaStreamCreate(&m->stream) != cudaSuccess) {
            delete m;
            return fail(MNMT_ECUDA, "cudaStreamCreate failed");
        }
        m->own_stream = true;
    }
    const uint8_t *hb = static_cast<const uint8_t *>(blob);
    const mnmt_config &c = m->c;
    const int d = c.d_model, F = c.d_ffn, dh = d / c.n_heads;
    if (cudaMalloc(&m->d_blob, bytes) != cudaSuccess) {
        mnmt_model_free(m);
        return fail(MNMT_ENOMEM, "cudaMalloc of %zu weight bytes failed", bytes);
    }
    if (cudaMemcpyAsync(m->d_blob, blob, bytes, cudaMemcpyHostToDevice, m->stream) != cudaSuccess) {
        mnmt_model_free(m);
        return fail(MNMT_ECUDA, "weight upload failed");
    }
    auto hf = [&](size_t off, int i) {
        float v;
        std::memcpy(&v, hb + off + 4 * i, 4);
        return v;
    };
    // 4-bit linears: rows of at most 16 (and min-max rows always) run on the
    // 4-bit GEMV kernel; for more rows symmetric linears use an int8 copy of
    // their codes on the IMMA / tensor-core kernels (not kept when lean)
    m->wq = L.wq;
    if (L.wq == 4 && !m->lean) {
        size_t codes = 0;
        auto add = [&](const LinOff &o) { codes += (size_t)o.n * o.k; };
        for (const auto &x : L.enc_self) { add(x.qkv); add(x.o); }
        for (const auto &x : L.enc_ffn) { add(x.w1); add(x.w2); }
        for (const auto &x : L.dec_self) { add(x.qkv); add(x.o); }
        for (const auto &x : L.dec_cross) { add(x.q); add(x.kv); add(x.o); }
        for (const auto &x : L.dec_ffn) { add(x.w1); add(x.w2); }
        if (cudaMalloc(&m->d_w8, codes) != cudaSuccess) {
            mnmt_model_free(m);
            return fail(MNMT_ENOMEM, "cudaMalloc of %zu unpacked weight codes failed", codes);
        }
        m->w8_codes = codes;
    }
    size_t w8_at = 0;
    cudaError_t unpack_err = cudaSuccess;
    auto dlin = [&](const LinOff &o) {
        Lin l;
        l.s = reinterpret_cast<const float *>(m->d_blob + o.s);
        l.b = reinterpret_cast<const float *>(m->d_blob + o.b);
        l.n = o.n;
        l.k = o.k;
        l.bits = o.bits;
        l.wp = nullptr;
        l.m = nullptr;
        if (o.bits == 4) {
            l.wp = m->d_blob + o.w;
            l.m = o.minmax ? reinterpret_cast<const float *>(m->d_blob + o.m) : nullptr;
            l.w = nullptr;
            if (m->d_w8 && !o.minmax) {
                int8_t *dst = m->d_w8 + w8_at;
                w8_at += (size_t)o.n * o.k;
                if (unpack_err == cudaSuccess)
                    unpack_err = launch_unpack_w4_sym(l.wp, (size_t)o.n * o.k, dst, m->stream);
                l.w = dst;
            }
        } else {
            l.w = reinterpret_cast<const int8_t *>(m->d_blob + o.w);
        }
        return l;
    };
    auto dln = [&](size_t g, size_t b) {
        return LnP{reinterpret_cast<const float *>(m->d_blob + g), reinterpret_cast<const float *>(m->d_blob + b)};
    };
    // derived per-column requantisation constants: inv = fl(1 / s)
    std::vector<float> aux;
    std::vector<size_t> aux_at;
    auto push_inv = [&](std::initializer_list<std::pair<float, int>> segs) {
        aux_at.push_back(aux.size());
        for (auto &sg : segs)
            for (int i = 0; i < sg.second; i++) aux.push_back(1.0f / sg.first);
        while (aux.size() % 4) aux.push_back(0.0f);
        return aux_at.size() - 1;
    };
    struct Pend {
        const float **dst;
        size_t idx;
    };
    std::vector<Pend> pend;
    m->emb_q = reinterpret_cast<const int8_t *>(m->d_blob + L.emb_q);
    m->emb_s = reinterpret_cast<const float *>(m->d_blob + L.emb_s);
    m->factorised = c.d_embed != d;
    if (m->factorised) m->proj = dlin(L.proj);
    m->emb_scale = hf(L.globals, 0);
    m->s_enc = hf(L.globals, 1);
    m->s_dout = hf(L.globals, 2);
    m->pe = reinterpret_cast<const float *>(m->d_blob + L.pe);
    auto mk_self = [&](const SelfOff &o) {
        SelfBlk s;
        s.ln = dln(o.ln_g, o.ln_b);
        s.s_in = hf(o.sc, 0); s.s_q = hf(o.sc, 1); s.s_k = hf(o.sc, 2); s.s_v = hf(o.sc, 3);
        s.s_ctx = hf(o.sc, 4); s.gamma = hf(o.sc, 5);
        s.sigma = host_sigma(s.s_q, s.s_k, dh);
        s.rho = s.s_v / s.s_ctx;
        s.qkv = dlin(o.qkv);
        s.o = dlin(o.o);
        s.inv_qkv = nullptr;
        return s;
    };
    auto mk_ffn = [&](const FfnOff &o) {
        FfnBlk f;
        f.ln = dln(o.ln_g, o.ln_b);
        f.s_in = hf(o.sc, 0); f.s_h = hf(o.sc, 1); f.gamma = hf(o.sc, 2);
        f.w1 = dlin(o.w1);
        f.w2 = dlin(o.w2);
        f.inv_h = nullptr;
        return f;
    };
    for (int l = 0; l < c.n_enc; l++) {
        m->enc_self.push_back(mk_self(L.enc_self[l]));
        m->enc_ffn.push_back(mk_ffn(L.enc_ffn[l]));
    }
    for (int l = 0; l < c.n_dec; l++) {
        m->dec_self.push_back(mk_self(L.dec_self[l]));
        const CrossOff &o = L.dec_cross[l];
        CrossBlk x;
        x.ln = dln(o.ln_g, o.ln_b);
        x.s_in = hf(o.sc, 0); x.s_q = hf(o.sc, 1); x.s_k = hf(o.sc, 2); x.s_v = hf(o.sc, 3);
        x.s_ctx = hf(o.sc, 4); x.gamma = hf(o.sc, 5);
        x.sigma = host_sigma(x.s_q, x.s_k, dh);
        x.rho = x.s_v / x.s_ctx;
        x.q = dlin(o.q);
        x.kv = dlin(o.kv);
        x.o = dlin(o.o);
        m->dec_cross.push_back(x);
        m->dec_ffn.push_back(mk_ffn(L.dec_ffn[l]));
    }
    // vectors are final now: record pointer slots to patch after the aux upload
    for (auto &s : m->enc_self) pend.push_back({&s.inv_qkv, push_inv({{s.s_q, d}, {s.s_k, d}, {s.s_v, d}})});
    for (auto &s : m->dec_self) pend.push_back({&s.inv_qkv, push_inv({{s.s_q, d}, {s.s_k, d}, {s.s_v, d}})});
    for (auto &f : m->enc_ffn) pend.push_back({&f.inv_h, push_inv({{f.s_h, F}})});
    for (auto &f : m->dec_ffn) pend.push_back({&f.inv_h, push_inv({{f.s_h, F}})});
    for (auto &x : m->dec_cross) {
        pend.push_back({&x.inv_q, push_inv({{x.s_q, d}})});
        pend.push_back({&x.inv_kv, push_inv({{x.s_k, d}, {x.s_v, d}})});
    }
    if (c.pre_ln) {
        m->enc_final = dln(L.enc_ln_g, L.enc_ln_b);
        m->dec_final = dln(L.dec_ln_g, L.dec_ln_b);
    }
    m->out.w = reinterpret_cast<const int8_t *>(m->d_blob + L.out_w);
    m->out.s = reinterpret_cast<const float *>(m->d_blob + L.out_s);
    m->out.b = reinterpret_cast<const float *>(m->d_blob + L.out_b);
    m->out.n = c.vocab;
    m->out.k = d;
    // the tensor-core linears read the weight codes as fp16: convert the whole
    // blob once (the fp32 regions become unused garbage); offsets stay 16-byte
    // aligned, so W16 = d_blob16 + (W - d_blob) is 32-byte aligned.  A lean
    // model keeps the int8 blob only and runs every linear on the int8 kernels.
    if (unpack_err != cudaSuccess) {
        mnmt_model_free(m);
        return fail(MNMT_ECUDA, "unpacking the 4-bit weights failed");
    }
    m->device_bytes = bytes + aux.size() * 4 + m->w8_codes;
    if (m->d_w8) {
        if (cudaMalloc(&m->d_w8_16, m->w8_codes * 2) != cudaSuccess) {
            mnmt_model_free(m);
            return fail(MNMT_ENOMEM, "cudaMalloc of %zu fp16 weight bytes failed", m->w8_codes * 2);
        }
        m->device_bytes += m->w8_codes * 2;
        if (launch_codes_to_f16_flat(m->d_w8, m->d_w8_16, m->w8_codes, m->stream) != cudaSuccess) {
            mnmt_model_free(m);
            return fail(MNMT_ECUDA, "fp16 weight conversion failed");
        }
    }
    if (!m->lean) {
        if (cudaMalloc(&m->d_blob16, bytes * 2) != cudaSuccess) {
            mnmt_model_free(m);
            return fail(MNMT_ENOMEM, "cudaMalloc of %zu fp16 weight bytes failed", bytes * 2);
        }
        m->device_bytes += bytes * 2;
        if (launch_codes_to_f16_flat(reinterpret_cast<const int8_t *>(m->d_blob), m->d_blob16, bytes, m->stream) !=
            cudaSuccess) {
            mnmt_model_free(m);
            return fail(MNMT_ECUDA, "fp16 weight conversion failed");
        }
    }
    if (cudaMalloc(&m->d_aux, aux.size() * 4) != cudaSuccess) {
        mnmt_model_free(m);
        return fail(MNMT_ENOMEM, "cudaMalloc of derived constants failed");
    }
    if (cudaMemcpyAsync(m->d_aux, aux.data(), aux.size() * 4, cudaMemcpyHostToDevice, m->stream) != cudaSuccess ||
        cudaStreamSynchronize(m->stream) != cudaSuccess) {
        mnmt_model_free(m);
        return fail(MNMT_ECUDA, "upload of derived constants failed");
    }
    for (auto &pd : pend) *pd.dst = m->d_aux + aux_at[pd.idx];
    *out = m;
    return MNMT_OK;
}

extern "C" void mnmt_model_free(mnmt_model *m) {
    if (!m) return;
    if (m->stream) cudaStreamSynchronize(m->stream);
    if (m->d_blob) cudaFree(m->d_blob);
    if (m->d_blob16) cudaFree(m->d_blob16);
    if (m->d_w8) cudaFree(m->d_w8);
    if (m->d_w8_16) cudaFree(m->d_w8_16);
    if (m->d_aux) cudaFree(m->d_aux);
    if (m->own_stream && m->stream) cudaStreamDestroy(m->stream);
    delete m;
}

// ---------------------------------------------------------------------------
// session
// ---------------------------------------------------------------------------
// state words: step counter, done flag, step limit, beam tickets [3..4] (the
// cluster step's pending greedy selection shares [4]: search init clears
// both), status
enum { ST_T = 0, ST_DONE = 1, ST_TMAX = 2, ST_TICKET = 3, ST_PENDING = 4, ST_STATUS = 5, ST_N = 8 };
// layers of more rows than the GEMV kernel takes (16) run on the tensor cores
constexpr size_t TC_MIN_ROWS = 17;
// steps per multi-step decode graph (and per completion check of translate)
constexpr int GRAPH_STEPS = 16;

struct mnmt_session {
    mnmt_model *m;
    int Bmax, Smax, k, Tcap;
    int B = 0, S = 0, max_len = 0;
    int steps = 0;      // decode steps launched since the last encode
    int poisoned = 0;
    uint8_t *arena = nullptr;
    size_t arena_bytes = 0;
    float *resid, *cum, *logits;
    int8_t *act, *qkv, *ctx, *hid, *qbuf, *enc_q, *ck, *cv, *sk, *sv;
    __half *a16;        // fp16 copy of a tensor-core linear's input rows (other buffers)
    // fp16 mirrors of the int8 activation buffers, written by their producers
    // when the consumer is a tensor-core linear
    __half *act16 = nullptr, *ctx16 = nullptr, *hid16 = nullptr, *encq16 = nullptr;
    bool use_tc = true;  // tensor-core linears for layers of >= TC_MIN_ROWS rows
    int32_t *src_ids, *src_lens, *tok, *fin, *hist, *parents, *anc, *out_ids, *out_lens;
    float *out_scores;
    unsigned long long *keys, *cand;
    int *state;
    int *h_state = nullptr;  // pinned mirror of state, then a second slot for the look-ahead copy
    cudaEvent_t ev_look = nullptr;  // marks the look-ahead copy of translate's decode loop
    size_t ck_layer, sk_layer;  // per-layer strides of the caches (elements)
    cudaGraphExec_t gexec = nullptr;
    cudaGraphExec_t gexec_n = nullptr;  // GRAPH_STEPS consecutive steps (cluster path)
    int graph_B = -1, graph_S = -1;
    // cluster decode step (small greedy batches)
    DcParams *d_dc = nullptr;
    float *dc_ln = nullptr;  // the cluster step's LayerNorm vectors, contiguous
    bool use_cluster = false;
    int dc_S = 0;  // host source of the parameter block's S when it is updated
    int dc_nc = 0;
    size_t dc_smem = 0;
    int dc_flags = -1;  // the compiled-in model bits of its step kernel (dc_flags)
};

static int poison(mnmt_session *s, int code) {
    if (!s->poisoned) s->poisoned = code;
    return code;
}

extern "C" int mnmt_session_create(mnmt_model *m, int32_t max_batch, int32_t max_src_len, int32_t beam,
                                   int32_t max_len, mnmt_session **out) {
    return mnmt_session_create_ex(m, max_batch, max_src_len, beam, max_len, 0, out);
}

extern "C" int mnmt_session_create_ex(mnmt_model *m, int32_t max_batch, int32_t max_src_len, int32_t beam,
                                      int32_t max_len, int32_t flags, mnmt_session **out) {
    if (!out) return fail(MNMT_EINVAL, "out is null");
    *out = nullptr;
    if (!m) return fail(MNMT_EINVAL, "model is null");
    if (flags & ~MNMT_SESSION_LEAN) return fail(MNMT_EINVAL, "unknown session flags 0x%x", flags);
    // lean: the encoder and decoder share two int8 activation buffers and the
    // fp32 residual (the context aliases the LayerNorm output, the FFN hidden
    // aliases the QKV output: never live at the same time), no fp16 mirrors;
    // a lean model's sessions run every linear on the int8 kernels
    const bool lean = (flags & MNMT_SESSION_LEAN) != 0;
    const bool tc_ok = !lean && !m->lean;
    const mnmt_config &c = m->c;
    if (max_batch < 1 || max_src_len < 1 || max_src_len > 512 || max_src_len > c.max_pos || beam < 1 ||
        beam > 16 || beam > c.vocab || max_len < 1 || max_len > c.max_pos || max_len > 1024)
        return fail(MNMT_EINVAL, "session sizes out of range (batch %d, src %d, beam %d, len %d)", max_batch,
                    max_src_len, beam, max_len);
    mnmt_session *s = new (std::nothrow) mnmt_session();
    if (!s) return fail(MNMT_ENOMEM, "host allocation failed");
    s->m = m;
    s->Bmax = max_batch;
    s->Smax = max_src_len;
    s->k = beam;
    s->Tcap = max_len;
    const size_t d = c.d_model, F = c.d_ffn, V = c.vocab, L = c.n_dec;
    const size_t R = (size_t)max_batch * beam, ME = (size_t)max_batch * max_src_len;
    const size_t rows = ME > R ? ME : R;
    s->ck_layer = (size_t)max_batch * max_src_len * d;
    s->sk_layer = R * max_len * d;
    // arena layout (256-byte aligned pieces)
    size_t off = 0;
    auto piece = [&](size_t bytes) {
        size_t at = off;
        off += (bytes + 255) & ~(size_t)255;
        return at;
    };
    const size_t qkv_bytes = lean ? std::max(ME * 3 * d, rows * F) : ME * 3 * d;
    size_t o_resid = piece(rows * d * 4), o_act = piece(rows * (d > F ? d : F)), o_qkv = piece(qkv_bytes),
           o_ctx = lean ? o_act : piece(rows * d), o_hid = lean ? o_qkv : piece(rows * F), o_qbuf = piece(R * d),
           o_encq = piece(ME * d),
           o_ck = piece(L * s->ck_layer), o_cv = piece(L * s->ck_layer), o_sk = piece(L * s->sk_layer),
           o_sv = piece(L * s->sk_layer), o_ids = piece(ME * 4), o_lens = piece((size_t)max_batch * 4),
           o_tok = piece(R * 4), o_fin = piece(R * 4), o_cum = piece(R * 4),
           o_hist = piece((size_t)max_len * R * 4), o_par = piece((size_t)max_len * R * 4),
           o_anc = piece(R * max_len * 4), o_keys = piece(R * 8), o_cand = piece(R * beam * 8),
           o_logits = piece(beam > 1 ? R * V * 4 : 256), o_outids = piece((size_t)max_batch * max_len * 4),
           o_outlens = piece((size_t)max_batch * 4), o_outsc = piece((size_t)max_batch * 4),
           o_state = piece(ST_N * 4), o_dc = piece(sizeof(DcParams)), o_dcln = piece((6 * L + 2) * d * 4);
    const size_t kmax = std::max(d, std::max(F, (size_t)c.d_embed));
    const bool tc_any = tc_ok && rows >= TC_MIN_ROWS;
    size_t o_a16 = piece(tc_any ? rows * kmax * 2 : 256);
    size_t o_act16 = piece(tc_any ? rows * kmax * 2 : 256), o_ctx16 = piece(tc_any ? rows * d * 2 : 256),
           o_hid16 = piece(tc_any ? rows * F * 2 : 256), o_encq16 = piece(tc_any ? ME * d * 2 : 256);
    s->arena_bytes = off;
    if (cudaMalloc(&s->arena, off) != cudaSuccess) {
        delete s;
        return fail(MNMT_ENOMEM, "cudaMalloc of %zu session bytes failed", off);
    }
    if (cudaMallocHost(&s->h_state, 2 * ST_N * 4) != cudaSuccess) {
        cudaFree(s->arena);
        delete s;
        return fail(MNMT_ENOMEM, "pinned host allocation failed");
    }
    if (cudaEventCreateWithFlags(&s->ev_look, cudaEventDisableTiming) != cudaSuccess) {
        cudaFreeHost(s->h_state);
        cudaFree(s->arena);
        delete s;
        return fail(MNMT_ECUDA, "event creation failed");
    }
    uint8_t *a = s->arena;
    s->resid = reinterpret_cast<float *>(a + o_resid);
    s->act = reinterpret_cast<int8_t *>(a + o_act);
    s->qkv = reinterpret_cast<int8_t *>(a + o_qkv);
    s->ctx = reinterpret_cast<int8_t *>(a + o_ctx);
    s->hid = reinterpret_cast<int8_t *>(a + o_hid);
    s->qbuf = reinterpret_cast<int8_t *>(a + o_qbuf);
    s->enc_q = reinterpret_cast<int8_t *>(a + o_encq);
    s->ck = reinterpret_cast<int8_t *>(a + o_ck);
    s->cv = reinterpret_cast<int8_t *>(a + o_cv);
    s->sk = reinterpret_cast<int8_t *>(a + o_sk);
    s->sv = reinterpret_cast<int8_t *>(a + o_sv);
    s->src_ids = reinterpret_cast<int32_t *>(a + o_ids);
    s->src_lens = reinterpret_cast<int32_t *>(a + o_lens);
    s->tok = reinterpret_cast<int32_t *>(a + o_tok);
    s->fin = reinterpret_cast<int32_t *>(a + o_fin);
    s->cum = reinterpret_cast<float *>(a + o_cum);
    s->hist = reinterpret_cast<int32_t *>(a + o_hist);
    s->parents = reinterpret_cast<int32_t *>(a + o_par);
    s->anc = reinterpret_cast<int32_t *>(a + o_anc);
    s->keys = reinterpret_cast<unsigned long long *>(a + o_keys);
    s->cand = reinterpret_cast<unsigned long long *>(a + o_cand);
    s->logits = reinterpret_cast<float *>(a + o_logits);
    s->out_ids = reinterpret_cast<int32_t *>(a + o_outids);
    s->out_lens = reinterpret_cast<int32_t *>(a + o_outlens);
    s->out_scores = reinterpret_cast<float *>(a + o_outsc);
    s->state = reinterpret_cast<int *>(a + o_state);
    s->d_dc = reinterpret_cast<DcParams *>(a + o_dc);
    s->dc_ln = reinterpret_cast<float *>(a + o_dcln);
    s->a16 = reinterpret_cast<__half *>(a + o_a16);
    s->act16 = reinterpret_cast<__half *>(a + o_act16);
    s->ctx16 = reinterpret_cast<__half *>(a + o_ctx16);
    s->hid16 = reinterpret_cast<__half *>(a + o_hid16);
    s->encq16 = reinterpret_cast<__half *>(a + o_encq16);
    {
        const char *v = std::getenv("MNMT_TC");
        s->use_tc = tc_ok && !(v && v[0] == '0') && rows >= TC_MIN_ROWS;
    }
    if (cudaMemsetAsync(s->arena, 0, off, m->stream) != cudaSuccess ||
        cudaStreamSynchronize(m->stream) != cudaSuccess) {
        mnmt_session_free(s);
        return fail(MNMT_ECUDA, "arena initialisation failed");
    }
    *out = s;
    return MNMT_OK;
}

extern "C" void mnmt_session_free(mnmt_session *s) {
    if (!s) return;
    if (s->m && s->m->stream) cudaStreamSynchronize(s->m->stream);
    if (s->gexec) cudaGraphExecDestroy(s->gexec);
    if (s->gexec_n) cudaGraphExecDestroy(s->gexec_n);
    if (s->arena) cudaFree(s->arena);
    if (s->h_state) cudaFreeHost(s->h_state);
    if (s->ev_look) cudaEventDestroy(s->ev_look);
    delete s;
}

// ---------------------------------------------------------------------------
// launch sequences
// ---------------------------------------------------------------------------
namespace {

Epi base_epi(int mode, float s_x, const Lin &l) {
    Epi e;
    std::memset(&e, 0, sizeof(e));
    e.mode = mode;
    e.s_x = s_x;
    e.s_w = l.s;
    e.bias = l.b;
    return e;
}

// fp16 copy of the codes of weight w (tensor-core operand)
const __half *w16_of(const mnmt_model *m, const int8_t *w) {
    if (m->d_w8 && w >= m->d_w8 && w < m->d_w8 + m->w8_codes) return m->d_w8_16 + (w - m->d_w8);
    return m->d_blob16 + (w - reinterpret_cast<const int8_t *>(m->d_blob));
}

// does a linear of M rows run on the tensor cores (then its input comes from
// the fp16 mirror its producer wrote)
bool tc_rows(const mnmt_session *s, int M) { return s->use_tc && (size_t)M >= TC_MIN_ROWS; }

// fp16 mirror of one of the session's int8 activation buffers
__half *mirror16(mnmt_session *s, const int8_t *buf) {
    if (buf == s->act) return s->act16;
    if (buf == s->ctx) return s->ctx16;
    if (buf == s->hid) return s->hid16;
    if (buf == s->enc_q) return s->encq16;
    return nullptr;
}

// the fp16 copy a producer of buf (M rows) must also write, or null
__half *out16_for(mnmt_session *s, const int8_t *buf, int M) { return tc_rows(s, M) ? mirror16(s, buf) : nullptr; }

// The quantised linear of rows A [M][lda] (Eq. 3 + epilogue e): on the
// tensor cores when the layer is a dense contraction (M >= TC_MIN_ROWS),
// reading the fp16 mirror of A that A's producer wrote; else on the IMMA /
// GEMV kernels.
cudaError_t run_linear(mnmt_session *s, const int8_t *A, int lda, const Lin &l, int M, const Epi &e,
                       cudaStream_t st) {
    const mnmt_model *m = s->m;
    if (l.bits == 4 && ((size_t)M <= 16 || !l.w)) return launch_linear_w4(A, lda, l.wp, l.m, M, l.n, l.k, e, st);
    if (tc_rows(s, M) && l.k % 16 == 0) {
        const __half *w16 = w16_of(m, l.w);
        const __half *a16 = mirror16(s, A);
        int lda16 = lda;
        if (!a16) {  // not a mirrored buffer: convert here
            a16 = s->a16;
            lda16 = l.k;
        }
        if (linear_tc_shape_ok(M, l.n, l.k, lda16, l.k, a16, w16)) {
            cudaError_t err = cudaSuccess;
            if (a16 == s->a16) err = launch_codes_to_f16(A, lda, s->a16, l.k, M, l.k, st);
            if (err == cudaSuccess)
                err = launch_linear_tc(a16, lda16, w16, l.k, M, l.n, l.k, e, s->state + ST_STATUS, st);
            return err;
        }
    }
    return launch_linear(A, lda, l.w, M, l.n, l.k, e, st);
}

#define LK(call)                                                                                   \
    do {                                                                                           \
        cudaError_t e_ = (call);                                                                   \
        if (e_ != cudaSuccess) return fail(MNMT_ECUDA, "%s: %s", #call, cudaGetErrorString(e_));   \
    } while (0)

// LayerNorm after a residual update.  Pre-LN: q8(LN_next(r)) into act (r kept).
// Post-LN: r = LN_this(r) in place, act = q8(r).
int ln_after_residual(mnmt_session *s, int M, const LnP &ln_pre_next, const LnP &ln_post_this, float s_next,
                      int8_t *act_out, const int *skip) {
    mnmt_model *m = s->m;
    LnArgs a;
    std::memset(&a, 0, sizeof(a));
    a.r = s->resid;
    a.M = M;
    a.d = m->c.d_model;
    a.inv = 1.0f / s_next;
    a.out_q = act_out;
    a.out16 = out16_for(s, act_out, M);
    a.status = s->state + ST_STATUS;
    a.skip = skip;
    if (m->c.pre_ln) {
        a.g = ln_pre_next.g;
        a.b = ln_pre_next.b;
    } else {
        a.g = ln_post_this.g;
        a.b = ln_post_this.b;
        a.out_f = s->resid;
    }
    LK(launch_layernorm(a, m->stream));
    return MNMT_OK;
}

int run_encoder(mnmt_session *s, int B, int S) {
    mnmt_model *m = s->m;
    const mnmt_config &c = m->c;
    const int d = c.d_model, F = c.d_ffn, H = c.n_heads, dh = d / H, M = B * S;
    cudaStream_t st = m->stream;
    int *status = s->state + ST_STATUS;
    {
        EmbedArgs e;
        std::memset(&e, 0, sizeof(e));
        e.ids = s->src_ids;
        e.S = S;
        e.emb_q = m->emb_q;
        e.emb_s = m->emb_s;
        if (m->factorised) {
            e.proj_w = m->proj.w;
            e.proj_s = m->proj.s;
            e.proj_b = m->proj.b;
        }
        e.emb_scale = m->emb_scale;
        e.pe = m->pe;
        e.M = M;
        e.d = d;
        e.E = c.d_embed;
        e.V = c.vocab;
        e.r = s->resid;
        e.out_q = s->act;
        e.out16 = out16_for(s, s->act, M);
        if (c.pre_ln) {
            e.ln_g = m->enc_self[0].ln.g;
            e.ln_b = m->enc_self[0].ln.b;
        }
        e.inv = 1.0f / m->enc_self[0].s_in;
        e.status = status;
        LK(launch_embed(e, st));
    }
    for (int l = 0; l < c.n_enc; l++) {
        const SelfBlk &A = m->enc_self[l];
        const FfnBlk &Fb = m->enc_ffn[l];
        Epi e = base_epi(EPI_Q8, A.s_in, A.qkv);
        e.inv_out = A.inv_qkv;
        e.out = s->qkv;
        e.ldo = 3 * d;
        LK(run_linear(s, s->act, d, A.qkv, M, e, st));  // N = 3 * d, K = d
        AttnEncArgs at;
        std::memset(&at, 0, sizeof(at));
        at.qkv = s->qkv;
        at.ctx = s->ctx;
        at.ctx16 = out16_for(s, s->ctx, M);
        at.len = s->src_lens;
        at.B = B;
        at.S = S;
        at.H = H;
        at.dh = dh;
        at.d = d;
        at.sigma = A.sigma;
        at.rho = A.rho;
        LK(launch_attention_encoder(at, st));
        e = base_epi(EPI_RESID, A.s_ctx, A.o);
        e.f32 = s->resid;
        e.ldf = d;
        e.gamma = A.gamma;
        LK(run_linear(s, s->ctx, d, A.o, M, e, st));  // N = d, K = d
        int rc = ln_after_residual(s, M, Fb.ln, A.ln, Fb.s_in, s->act, nullptr);
        if (rc) return rc;
        e = base_epi(EPI_RELU_Q8, Fb.s_in, Fb.w1);
        e.inv_out = Fb.inv_h;
        e.out = s->hid;
        e.out16 = out16_for(s, s->hid, M);
        e.ldo = F;
        LK(run_linear(s, s->act, d, Fb.w1, M, e, st));  // N = F, K = d
        e = base_epi(EPI_RESID, Fb.s_h, Fb.w2);
        e.f32 = s->resid;
        e.ldf = d;
        e.gamma = Fb.gamma;
        LK(run_linear(s, s->hid, F, Fb.w2, M, e, st));  // N = d, K = F
        if (l + 1 < c.n_enc) {
            const SelfBlk &An = m->enc_self[l + 1];
            rc = ln_after_residual(s, M, An.ln, Fb.ln, An.s_in, s->act, nullptr);
        } else {
            rc = ln_after_residual(s, M, m->enc_final, Fb.ln, m->s_enc, s->enc_q, nullptr);
        }
        if (rc) return rc;
    }
    for (int l = 0; l < c.n_dec; l++) {
        const CrossBlk &X = m->dec_cross[l];
        Epi e = base_epi(EPI_KV_CROSS, m->s_enc, X.kv);
        e.inv_out = X.inv_kv;
        e.kc = s->ck + l * s->ck_layer;
        e.vc = s->cv + l * s->ck_layer;
        e.d = d;
        e.H = H;
        e.dh = dh;
        e.S = S;
        LK(run_linear(s, s->enc_q, d, X.kv, M, e, st));  // N = 2 * d, K = d
    }
    return MNMT_OK;
}

// the model bits the single-row step kernels may have compiled in: pre-LN,
// factorised embedding, R * d above 256, log2 of the attention's warps per
// item (bits 3-4, from the parameter block's layout)
static int dc_flags(const mnmt_config &c, const mnmt_model *m, int R, int att_lw) {
    return (c.pre_ln ? 1 : 0) | (m->factorised ? 2 : 0) | (R * c.d_model > 256 ? 4 : 0) | (att_lw << 3);
}

// one decoder step for all B*k hypotheses (captured into a graph)
int issue_decode_step(mnmt_session *s) {
    mnmt_model *m = s->m;
    const mnmt_config &c = m->c;
    const int d = c.d_model, F = c.d_ffn, H = c.n_heads, dh = d / H;
    const int R = s->B * s->k;
    cudaStream_t st = m->stream;
    const int *done = s->state + ST_DONE;
    int *t_ptr = s->state + ST_T;
    int *status = s->state + ST_STATUS;
    if (s->use_cluster) {
        LK(launch_decode_cluster(s->d_dc, dh, s->dc_nc, s->dc_smem, m->wq != 8, R == 1, s->dc_flags, st));
        GreedyArgs g;
        g.keys = s->keys;
        g.tok = s->tok;
        g.fin = s->fin;
        g.hist = s->hist;
        g.t_ptr = t_ptr;
        g.done = s->state + ST_DONE;
        g.tmax_ptr = s->state + ST_TMAX;
        g.R = R;
        g.T = s->Tcap;
        g.eos = c.eos_id;
        g.pad = c.pad_id;
        g.pending = s->state + ST_PENDING;
        LK(launch_vocab_greedy(s->act, m->out.w, m->out.s, m->out.b, m->s_dout, R, c.vocab, d, s->keys,
                               s->state + ST_TICKET, g, s->dc_nc, st));
        return MNMT_OK;
    }
    {
        EmbedArgs e;
        std::memset(&e, 0, sizeof(e));
        e.tok = s->tok;
        e.t_ptr = t_ptr;
        e.emb_q = m->emb_q;
        e.emb_s = m->emb_s;
        if (m->factorised) {
            e.proj_w = m->proj.w;
            e.proj_s = m->proj.s;
            e.proj_b = m->proj.b;
        }
        e.emb_scale = m->emb_scale;
        e.pe = m->pe;
        e.M = R;
        e.d = d;
        e.E = c.d_embed;
        e.V = c.vocab;
        e.r = s->resid;
        e.out_q = s->act;
        e.out16 = out16_for(s, s->act, R);
        if (c.pre_ln) {
            e.ln_g = m->dec_self[0].ln.g;
            e.ln_b = m->dec_self[0].ln.b;
        }
        e.inv = 1.0f / m->dec_self[0].s_in;
        e.status = status;
        e.skip = done;
        LK(launch_embed(e, st));
    }
    for (int l = 0; l < c.n_dec; l++) {
        const SelfBlk &A = m->dec_self[l];
        const CrossBlk &X = m->dec_cross[l];
        const FfnBlk &Fb = m->dec_ffn[l];
        Epi e = base_epi(EPI_QKV_DEC, A.s_in, A.qkv);
        e.inv_out = A.inv_qkv;
        e.out = s->qbuf;
        e.ldo = d;
        e.kc = s->sk + l * s->sk_layer;
        e.vc = s->sv + l * s->sk_layer;
        e.t_ptr = t_ptr;
        e.d = d;
        e.H = H;
        e.dh = dh;
        e.T = s->Tcap;
        e.skip = done;
        LK(run_linear(s, s->act, d, A.qkv, R, e, st));  // N = 3 * d, K = d
        AttnDecArgs at;
        std::memset(&at, 0, sizeof(at));
        at.q = s->qbuf;
        at.kc = s->sk + l * s->sk_layer;
        at.vc = s->sv + l * s->sk_layer;
        at.ctx = s->ctx;
        at.ctx16 = out16_for(s, s->ctx, R);
        at.R = R;
        at.H = H;
        at.dh = dh;
        at.T = s->Tcap;
        at.cross = 0;
        at.beam = s->k;
        at.t_ptr = t_ptr;
        at.anc = s->k > 1 ? s->anc : nullptr;
        at.sigma = A.sigma;
        at.rho = A.rho;
        at.skip = done;
        LK(launch_attention_decode(at, st));
        e = base_epi(EPI_RESID, A.s_ctx, A.o);
        e.f32 = s->resid;
        e.ldf = d;
        e.gamma = A.gamma;
        e.skip = done;
        LK(run_linear(s, s->ctx, d, A.o, R, e, st));  // N = d, K = d
        int rc = ln_after_residual(s, R, X.ln, A.ln, X.s_in, s->act, done);
        if (rc) return rc;
        e = base_epi(EPI_Q8, X.s_in, X.q);
        e.inv_out = X.inv_q;
        e.out = s->qbuf;
        e.ldo = d;
        e.skip = done;
        LK(run_linear(s, s->act, d, X.q, R, e, st));  // N = d, K = d
        at.kc = s->ck + l * s->ck_layer;
        at.vc = s->cv + l * s->ck_layer;
        at.T = s->S;
        at.cross = 1;
        at.src_len = s->src_lens;
        at.anc = nullptr;
        at.sigma = X.sigma;
        at.rho = X.rho;
        LK(launch_attention_decode(at, st));
        e = base_epi(EPI_RESID, X.s_ctx, X.o);
        e.f32 = s->resid;
        e.ldf = d;
        e.gamma = X.gamma;
        e.skip = done;
        LK(run_linear(s, s->ctx, d, X.o, R, e, st));  // N = d, K = d
        rc = ln_after_residual(s, R, Fb.ln, X.ln, Fb.s_in, s->act, done);
        if (rc) return rc;
        e = base_epi(EPI_RELU_Q8, Fb.s_in, Fb.w1);
        e.inv_out = Fb.inv_h;
        e.out = s->hid;
        e.out16 = out16_for(s, s->hid, R);
        e.ldo = F;
        e.skip = done;
        LK(run_linear(s, s->act, d, Fb.w1, R, e, st));  // N = F, K = d
        e = base_epi(EPI_RESID, Fb.s_h, Fb.w2);
        e.f32 = s->resid;
        e.ldf = d;
        e.gamma = Fb.gamma;
        e.skip = done;
        LK(run_linear(s, s->hid, F, Fb.w2, R, e, st));  // N = d, K = F
        if (l + 1 < c.n_dec) {
            const SelfBlk &An = m->dec_self[l + 1];
            rc = ln_after_residual(s, R, An.ln, Fb.ln, An.s_in, s->act, done);
        } else {
            rc = ln_after_residual(s, R, m->dec_final, Fb.ln, m->s_dout, s->act, done);
        }
        if (rc) return rc;
    }
    if (s->k == 1) {
        Epi e = base_epi(EPI_ARGMAX, m->s_dout, m->out);
        e.keys = s->keys;
        e.skip = done;
        LK(run_linear(s, s->act, d, m->out, R, e, st));  // N = c.vocab, K = d
        GreedyArgs g;
        g.keys = s->keys;
        g.tok = s->tok;
        g.fin = s->fin;
        g.hist = s->hist;
        g.t_ptr = t_ptr;
        g.done = s->state + ST_DONE;
        g.tmax_ptr = s->state + ST_TMAX;
        g.R = R;
        g.T = s->Tcap;
        g.eos = c.eos_id;
        g.pad = c.pad_id;
        LK(launch_greedy_update(g, st));
    } else {
        Epi e = base_epi(EPI_F32, m->s_dout, m->out);
        e.f32 = s->logits;
        e.ldf = c.vocab;
        e.skip = done;
        LK(run_linear(s, s->act, d, m->out, R, e, st));  // N = c.vocab, K = d
        BeamArgs b;
        b.logits = s->logits;
        b.tok = s->tok;
        b.fin = s->fin;
        b.cum = s->cum;
        b.hist = s->hist;
        b.parents = s->parents;
        b.anc = s->anc;
        b.cand = s->cand;
        b.t_ptr = t_ptr;
        b.done = s->state + ST_DONE;
        b.ticket = s->state + ST_TICKET;
        b.tmax_ptr = s->state + ST_TMAX;
        b.B = s->B;
        b.k = s->k;
        b.V = c.vocab;
        b.T = s->Tcap;
        b.eos = c.eos_id;
        b.pad = c.pad_id;
        b.status = status;
        LK(launch_beam_step(b, st));
    }
    return MNMT_OK;
}

// Chooses the decode-step implementation for the current batch: the
// single-cluster step for greedy batches of at most DC_RMAX sentences whose
// shapes fit one cluster's shared memory, else the multi-kernel step.
// MNMT_DECODE_CLUSTER=0 in the environment forces the multi-kernel step.
int setup_cluster_step(mnmt_session *s) {
    mnmt_model *m = s->m;
    const mnmt_config &c = m->c;
    s->use_cluster = false;
    const char *env = getenv("MNMT_DECODE_CLUSTER");
    if (env && env[0] == '0') return MNMT_OK;
    const int d = c.d_model, F = c.d_ffn, H = c.n_heads, dh = d / H;
    const int R = s->B * s->k;
    const int E = c.d_embed;
    const int nc = dc_cluster_size(d, F, E);
    if (s->k != 1 || R > DC_RMAX || c.n_dec > DC_LMAX || nc == 0 || d > 512 || F > 2048 || d % (16 * nc) ||
        F % (16 * nc) || (3 * d) % (16 * nc))
        return MNMT_OK;
    DcParams P;
    std::memset(&P, 0, sizeof(P));
    P.R = R; P.d = d; P.H = H; P.dh = dh; P.F = F; P.E = c.d_embed; P.V = c.vocab; P.T = s->Tcap; P.S = s->S;
    P.n_dec = c.n_dec; P.pre_ln = c.pre_ln; P.factorised = m->factorised; P.nc = nc;
    P.emb_q = m->emb_q; P.emb_s = m->emb_s;
    if (m->factorised) P.proj = DcLin{m->proj.w, m->proj.s, m->proj.b, nullptr, 8};
    P.emb_scale = m->emb_scale; P.pe = m->pe;
    P.fin_g = m->dec_final.g; P.fin_b = m->dec_final.b; P.s_dout = m->s_dout; P.inv_dout = 1.0f / m->s_dout;
    P.tok = s->tok; P.t_ptr = s->state + ST_T; P.done = s->state + ST_DONE; P.src_len = s->src_lens;
    P.keys = s->keys; P.tok_w = s->tok; P.fin = s->fin; P.hist = s->hist; P.t_w = s->state + ST_T;
    P.done_w = s->state + ST_DONE; P.pending = s->state + ST_PENDING; P.tmax_ptr = s->state + ST_TMAX;
    P.eos = c.eos_id; P.pad = c.pad_id;
    P.act_out = s->act; P.resid_out = s->resid; P.status = s->state + ST_STATUS;
    for (int l = 0; l < c.n_dec; l++) {
        const SelfBlk &A = m->dec_self[l];
        const CrossBlk &X = m->dec_cross[l];
        const FfnBlk &Fb = m->dec_ffn[l];
        DcLayer &Y = P.layer[l];
        Y.ln1_g = A.ln.g; Y.ln1_b = A.ln.b; Y.ln2_g = X.ln.g; Y.ln2_b = X.ln.b; Y.ln3_g = Fb.ln.g; Y.ln3_b = Fb.ln.b;
        Y.s_in1 = A.s_in; Y.s_ctx1 = A.s_ctx; Y.gamma1 = A.gamma; Y.sigma1 = A.sigma; Y.rho1 = A.rho;
        Y.s_in2 = X.s_in; Y.s_ctx2 = X.s_ctx; Y.gamma2 = X.gamma; Y.sigma2 = X.sigma; Y.rho2 = X.rho;
        Y.s_in3 = Fb.s_in; Y.s_h = Fb.s_h; Y.gamma3 = Fb.gamma;
        Y.inv_in1 = 1.0f / A.s_in; Y.inv_in2 = 1.0f / X.s_in; Y.inv_in3 = 1.0f / Fb.s_in;
        // 4-bit linears stream their packed codes (half the ring bytes)
        auto dl = [](const Lin &x) {
            if (x.bits == 4) return DcLin{reinterpret_cast<const int8_t *>(x.wp), x.s, x.b, x.m, 4};
            return DcLin{x.w, x.s, x.b, nullptr, 8};
        };
        Y.qkv = dl(A.qkv); Y.o = dl(A.o);
        Y.q2 = dl(X.q); Y.o2 = dl(X.o);
        Y.w1 = dl(Fb.w1); Y.w2 = dl(Fb.w2);
        Y.inv_qkv = A.inv_qkv; Y.inv_q2 = X.inv_q; Y.inv_h = Fb.inv_h;
        Y.self_k = s->sk + l * s->sk_layer; Y.self_v = s->sv + l * s->sk_layer;
        Y.cross_k = s->ck + l * s->ck_layer; Y.cross_v = s->cv + l * s->ck_layer;
    }
    // the LayerNorm vectors in one contiguous array (one copy per step)
    {
        const size_t vb = (size_t)d * 4;
        CK(cudaMemsetAsync(s->dc_ln, 0, (6 * c.n_dec + 2) * vb, m->stream));
        for (int l = 0; l < c.n_dec; l++) {
            const DcLayer &Y = P.layer[l];
            const float *src[6] = {Y.ln1_g, Y.ln1_b, Y.ln2_g, Y.ln2_b, Y.ln3_g, Y.ln3_b};
            for (int w = 0; w < 6; w++)
                if (src[w])
                    CK(cudaMemcpyAsync(s->dc_ln + (size_t)(6 * l + w) * d, src[w], vb, cudaMemcpyDeviceToDevice,
                                       m->stream));
        }
        if (P.fin_g) CK(cudaMemcpyAsync(s->dc_ln + (size_t)6 * c.n_dec * d, P.fin_g, vb, cudaMemcpyDeviceToDevice, m->stream));
        if (P.fin_b)
            CK(cudaMemcpyAsync(s->dc_ln + (size_t)(6 * c.n_dec + 1) * d, P.fin_b, vb, cudaMemcpyDeviceToDevice, m->stream));
        P.ln_all = s->dc_ln;
    }
    // lay shared memory out for the session's longest source, so that the
    // captured step serves every padded length (only P.S changes per batch)
    P.S = s->Smax;
    size_t smem = dc_layout(P, 227 * 1024);
    P.S = s->S;
    const int flags = dc_flags(c, m, R, P.att_lw);
    if (!decode_cluster_fits(dh, nc, smem, m->wq != 8, R == 1, flags)) return MNMT_OK;
    CK(cudaMemcpyAsync(s->d_dc, &P, sizeof(P), cudaMemcpyHostToDevice, m->stream));
    CK(cudaStreamSynchronize(m->stream));  // P lives on this stack frame
    s->use_cluster = true;
    s->dc_nc = nc;
    s->dc_smem = smem;
    s->dc_flags = flags;
    return MNMT_OK;
}

// capture `steps` consecutive decode steps into one executable graph
int capture_steps(mnmt_session *s, int steps, cudaGraphExec_t *out) {
    cudaStream_t st = s->m->stream;
    cudaGraph_t g = nullptr;
    CK(cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal));
    int rc = MNMT_OK;
    for (int i = 0; i < steps && !rc; i++) rc = issue_decode_step(s);
    if (!rc && s->use_cluster) {
        // the last step's greedy selection is still pending: apply it, so the
        // step counter, done flag and history are current when the graph ends
        GreedyArgs ga;
        ga.keys = s->keys;
        ga.tok = s->tok;
        ga.fin = s->fin;
        ga.hist = s->hist;
        ga.t_ptr = s->state + ST_T;
        ga.done = s->state + ST_DONE;
        ga.tmax_ptr = s->state + ST_TMAX;
        ga.R = s->B * s->k;
        ga.T = s->Tcap;
        ga.eos = s->m->c.eos_id;
        ga.pad = s->m->c.pad_id;
        ga.pending = s->state + ST_PENDING;
        cudaError_t le = launch_greedy_update(ga, st);
        if (le != cudaSuccess) rc = fail(MNMT_ECUDA, "greedy update launch failed: %s", cudaGetErrorString(le));
    }
    cudaError_t ce = cudaStreamEndCapture(st, &g);
    if (rc) {
        if (g) cudaGraphDestroy(g);
        return rc;
    }
    if (ce != cudaSuccess) return fail(MNMT_ECUDA, "graph capture failed: %s", cudaGetErrorString(ce));
    ce = cudaGraphInstantiate(out, g, 0);
    cudaGraphDestroy(g);
    if (ce != cudaSuccess) {
        *out = nullptr;
        return fail(MNMT_ECUDA, "graph instantiation failed: %s", cudaGetErrorString(ce));
    }
    return MNMT_OK;
}

int ensure_graph(mnmt_session *s) {
    if (s->gexec && s->graph_B == s->B && s->graph_S == s->S) return MNMT_OK;
    if (s->gexec && s->graph_B == s->B && s->use_cluster) {
        // the cluster step reads the padded source length from its parameter
        // block: update it in stream order and keep the captured graphs
        s->dc_S = s->S;
        CK(cudaMemcpyAsync(reinterpret_cast<uint8_t *>(s->d_dc) + offsetof(DcParams, S), &s->dc_S, sizeof(int),
                           cudaMemcpyHostToDevice, s->m->stream));
        s->graph_S = s->S;
        return MNMT_OK;
    }
    for (cudaGraphExec_t *ge : {&s->gexec, &s->gexec_n})
        if (*ge) {
            cudaGraphExecDestroy(*ge);
            *ge = nullptr;
        }
    int rc = setup_cluster_step(s);
    if (rc) return rc;
    if ((rc = capture_steps(s, 1, &s->gexec))) return rc;
    // the cluster step also gets a graph of GRAPH_STEPS steps, inside which
    // each step's kernel starts while the previous step's vocabulary kernel
    // runs (programmatic dependent launch)
    if (s->use_cluster && (rc = capture_steps(s, GRAPH_STEPS, &s->gexec_n))) return rc;
    s->graph_B = s->B;
    s->graph_S = s->S;
    return MNMT_OK;
}

// queue n decode steps (graph launches, no synchronisation)
int launch_steps(mnmt_session *s, int n) {
    cudaStream_t st = s->m->stream;
    while (n > 0) {
        if (s->gexec_n && n >= GRAPH_STEPS) {
            CK(cudaGraphLaunch(s->gexec_n, st));
            n -= GRAPH_STEPS;
        } else {
            CK(cudaGraphLaunch(s->gexec, st));
            n--;
        }
    }
    return MNMT_OK;
}

int check_device_status(mnmt_session *s) {
    // called after a synchronisation that covered a copy of state into h_state
    int code = s->h_state[ST_STATUS];
    if (code) return poison(s, fail(code, "device reported status %d", code));
    return MNMT_OK;
}

int sync_state(mnmt_session *s) {
    cudaStream_t st = s->m->stream;
    cudaError_t e = cudaMemcpyAsync(s->h_state, s->state, ST_N * 4, cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return poison(s, fail(MNMT_ECUDA, "device work failed: %s", cudaGetErrorString(e)));
    return check_device_status(s);
}

}  // namespace

extern "C" int mnmt_encode(mnmt_session *s, const int32_t *src_ids, const int32_t *src_lens, int32_t B,
                           int32_t S_pad, int32_t flags) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    if (s->poisoned) return fail(s->poisoned, "session poisoned by an earlier failure");
    if (!src_ids || !src_lens || B < 1 || B > s->Bmax || S_pad < 1 || S_pad > s->Smax)
        return fail(MNMT_EINVAL, "encode: bad batch %d / padded length %d (capacity %d / %d)", B, S_pad, s->Bmax,
                    s->Smax);
    mnmt_model *m = s->m;
    cudaStream_t st = m->stream;
    const bool dev = flags & MNMT_DEVICE_PTRS;
    if (!dev) {
        for (int b = 0; b < B; b++)
            if (src_lens[b] < 1 || src_lens[b] > S_pad) return fail(MNMT_EINVAL, "source length %d out of range", src_lens[b]);
        for (long i = 0; i < (long)B * S_pad; i++)
            if (src_ids[i] < 0 || src_ids[i] >= m->c.vocab) return fail(MNMT_EINVAL, "source id out of range");
    }
    cudaMemcpyKind kind = dev ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;
    CK(cudaMemcpyAsync(s->src_ids, src_ids, (size_t)B * S_pad * 4, kind, st));
    CK(cudaMemcpyAsync(s->src_lens, src_lens, (size_t)B * 4, kind, st));
    s->B = B;
    s->S = S_pad;
    int rc = run_encoder(s, B, S_pad);
    if (rc) return poison(s, rc);
    InitArgs ia;
    ia.tok = s->tok;
    ia.fin = s->fin;
    ia.anc = s->anc;
    ia.hist = s->hist;
    ia.parents = s->parents;
    ia.cum = s->cum;
    ia.keys = s->keys;
    ia.t_ptr = s->state + ST_T;
    ia.done = s->state + ST_DONE;
    ia.ticket = s->state + ST_TICKET;
    ia.R = B * s->k;
    ia.k = s->k;
    ia.T = s->Tcap;
    ia.bos = m->c.bos_id;
    ia.pad = m->c.pad_id;
    CK(launch_search_init(ia, st));
    s->max_len = s->Tcap;
    s->h_state[ST_TMAX] = s->Tcap;
    CK(cudaMemcpyAsync(s->state + ST_TMAX, s->h_state + ST_TMAX, 4, cudaMemcpyHostToDevice, st));
    s->steps = 0;
    return MNMT_OK;
}

extern "C" int mnmt_decode_steps(mnmt_session *s, int32_t n) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    if (s->poisoned) return fail(s->poisoned, "session poisoned by an earlier failure");
    if (s->B < 1) return fail(MNMT_EINVAL, "decode_steps before encode");
    if (n < 0) return fail(MNMT_EINVAL, "negative step count");
    const int left = s->max_len - s->steps;
    if (n > left) n = left;
    if (n == 0) return 0;
    int rc = ensure_graph(s);
    if (rc) return poison(s, rc);
    if ((rc = launch_steps(s, n))) return poison(s, rc);
    s->steps += n;
    return n;
}

extern "C" int mnmt_decode_step(mnmt_session *s, int32_t *tokens, int32_t *parents, float *scores,
                                int32_t *all_done) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    if (s->poisoned) return fail(s->poisoned, "session poisoned by an earlier failure");
    if (s->B < 1) return fail(MNMT_EINVAL, "decode_step before encode");
    if (s->steps >= s->max_len) return fail(MNMT_EINVAL, "all %d steps already ran", s->max_len);
    int rc = ensure_graph(s);
    if (rc) return poison(s, rc);
    cudaStream_t st = s->m->stream;
    CK(cudaGraphLaunch(s->gexec, st));
    const int t = s->steps++;
    const int R = s->B * s->k;
    if (tokens) CK(cudaMemcpyAsync(tokens, s->hist + (size_t)t * R, R * 4, cudaMemcpyDeviceToHost, st));
    if (parents) CK(cudaMemcpyAsync(parents, s->parents + (size_t)t * R, R * 4, cudaMemcpyDeviceToHost, st));
    if (scores) CK(cudaMemcpyAsync(scores, s->cum, R * 4, cudaMemcpyDeviceToHost, st));
    if ((rc = sync_state(s))) return rc;
    if (scores && s->k == 1)
        for (int i = 0; i < R; i++) scores[i] = 0.0f;
    if (all_done) *all_done = s->h_state[ST_DONE];
    return MNMT_OK;
}

extern "C" int mnmt_translate(mnmt_session *s, const int32_t *src_ids, const int32_t *src_lens, int32_t B,
                              int32_t S_pad, int32_t max_len, int32_t flags, int32_t *out_ids,
                              int32_t *out_lens, float *out_scores) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    if (max_len < 1 || max_len > s->Tcap) return fail(MNMT_EINVAL, "max_len %d outside [1, %d]", max_len, s->Tcap);
    if (!out_ids || !out_lens || !out_scores) return fail(MNMT_EINVAL, "null output");
    int rc = mnmt_encode(s, src_ids, src_lens, B, S_pad, flags);
    if (rc) return rc;
    cudaStream_t st = s->m->stream;
    s->max_len = max_len;
    s->h_state[ST_TMAX] = max_len;
    CK(cudaMemcpyAsync(s->state + ST_TMAX, s->h_state + ST_TMAX, 4, cudaMemcpyHostToDevice, st));
    if ((rc = ensure_graph(s))) return poison(s, rc);
    // Chunks of GRAPH_STEPS steps with one chunk of look-ahead: a copy of the
    // state after the chunks queued so far is taken, the next chunk is queued,
    // and only then is the copy read, so the device never waits for the host.
    // Steps queued after every hypothesis finished are no-ops (each step
    // kernel tests the done flag).
    const int CHECK = GRAPH_STEPS;
    int steps = max_len < CHECK ? max_len : CHECK;
    if ((rc = launch_steps(s, steps))) return poison(s, rc);
    int *look = s->h_state + ST_N;
    while (steps < max_len) {
        CK(cudaMemcpyAsync(look, s->state, ST_N * 4, cudaMemcpyDeviceToHost, st));
        CK(cudaEventRecord(s->ev_look, st));
        const int n = max_len - steps < CHECK ? max_len - steps : CHECK;
        if ((rc = launch_steps(s, n))) return poison(s, rc);
        steps += n;
        const cudaError_t e = cudaEventSynchronize(s->ev_look);
        if (e != cudaSuccess) return poison(s, fail(MNMT_ECUDA, "device work failed: %s", cudaGetErrorString(e)));
        if (look[ST_STATUS]) return poison(s, fail(look[ST_STATUS], "device reported status %d", look[ST_STATUS]));
        if (look[ST_DONE]) break;
    }
    s->steps = steps;
    const bool dev = flags & MNMT_DEVICE_PTRS;
    FinalArgs fa;
    fa.hist = s->hist;
    fa.parents = s->parents;
    fa.cum = s->cum;
    fa.t_ptr = s->state + ST_T;
    fa.out_ids = dev ? out_ids : s->out_ids;
    fa.out_lens = dev ? out_lens : s->out_lens;
    fa.out_scores = dev ? out_scores : s->out_scores;
    fa.B = B;
    fa.k = s->k;
    fa.T = s->Tcap;
    fa.max_len = max_len;
    fa.eos = s->m->c.eos_id;
    fa.pad = s->m->c.pad_id;
    CK(launch_finalize(fa, st));
    if (!dev) {
        CK(cudaMemcpyAsync(out_ids, s->out_ids, (size_t)B * max_len * 4, cudaMemcpyDeviceToHost, st));
        CK(cudaMemcpyAsync(out_lens, s->out_lens, (size_t)B * 4, cudaMemcpyDeviceToHost, st));
        CK(cudaMemcpyAsync(out_scores, s->out_scores, (size_t)B * 4, cudaMemcpyDeviceToHost, st));
        return sync_state(s);
    }
    // device outputs: report asynchronous failures at the next synchronising call
    cudaError_t e = cudaMemcpyAsync(s->h_state, s->state, ST_N * 4, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return poison(s, fail(MNMT_ECUDA, "state copy failed: %s", cudaGetErrorString(e)));
    return MNMT_OK;
}

extern "C" int64_t mnmt_debug_tap(mnmt_session *s, int32_t tap, int32_t layer, void *host_dst, size_t bytes) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    const mnmt_config &c = s->m->c;
    const size_t d = c.d_model, H = c.n_heads, dh = d / H, R = (size_t)s->B * s->k;
    const void *src = nullptr;
    size_t n = 0;
    auto need_layer = [&]() { return layer >= 0 && layer < c.n_dec; };
    switch (tap) {
        case MNMT_TAP_ENC_OUT:
            src = s->enc_q;
            n = (size_t)s->B * s->S * d;
            break;
        case MNMT_TAP_CROSS_K:
        case MNMT_TAP_CROSS_V:
            if (!need_layer()) return fail(MNMT_EINVAL, "layer out of range");
            src = (tap == MNMT_TAP_CROSS_K ? s->ck : s->cv) + layer * s->ck_layer;
            n = (size_t)s->B * H * s->S * dh;
            break;
        case MNMT_TAP_SELF_K:
        case MNMT_TAP_SELF_V:
            if (!need_layer()) return fail(MNMT_EINVAL, "layer out of range");
            src = (tap == MNMT_TAP_SELF_K ? s->sk : s->sv) + layer * s->sk_layer;
            n = R * H * s->Tcap * dh;
            break;
        case MNMT_TAP_DEC_OUT:
            src = s->act;
            n = R * d;
            break;
        case MNMT_TAP_LOGITS:
            if (s->k == 1) return fail(MNMT_EINVAL, "logits are kept only for beam search");
            src = s->logits;
            n = R * c.vocab * 4;
            break;
        case MNMT_TAP_RESID:
            src = s->resid;
            n = (s->steps > 0 ? R : (size_t)s->B * s->S) * d * 4;
            break;
        case MNMT_TAP_HISTORY:
            src = s->hist;
            n = (size_t)s->Tcap * R * 4;
            break;
        case MNMT_TAP_PARENTS:
            src = s->parents;
            n = (size_t)s->Tcap * R * 4;
            break;
        case MNMT_TAP_ANCESTRY:
            src = s->anc;
            n = R * s->Tcap * 4;
            break;
        default:
            return fail(MNMT_EINVAL, "unknown tap %d", tap);
    }
    if (!host_dst) return (int64_t)n;
    if (bytes != n) return fail(MNMT_EINVAL, "tap %d holds %zu bytes, not %zu", tap, n, bytes);
    cudaStream_t st = s->m->stream;
    CK(cudaMemcpyAsync(host_dst, src, n, cudaMemcpyDeviceToHost, st));
    CK(cudaStreamSynchronize(st));
    return MNMT_OK;
}

extern "C" const char *mnmt_last_error(void) { return g_err.c_str(); }

extern "C" int64_t mnmt_model_device_bytes(const mnmt_model *m) {
    if (!m) return fail(MNMT_EINVAL, "model is null");
    return (int64_t)m->device_bytes;
}

extern "C" int64_t mnmt_session_device_bytes(const mnmt_session *s) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    return (int64_t)s->arena_bytes;
}

extern "C" int mnmt_session_decode_path(mnmt_session *s) {
    if (!s) return fail(MNMT_EINVAL, "session is null");
    if (s->B < 1) return fail(MNMT_EINVAL, "no batch encoded yet");
    int rc = ensure_graph(s);
    if (rc) return rc;
    return s->use_cluster ? 1 : 0;
}

int mnmt::set_error(int code, const char *msg) { return fail(code, "%s", msg); }

// ---------------------------------------------------------------------------
// kernel-level entry points
// ---------------------------------------------------------------------------
extern "C" int mnmt_linear(const int8_t *A, const int8_t *W, const float *s_w, const float *bias, float s_x,
                           const float *inv_out, float gamma, int32_t M, int32_t N, int32_t K, int32_t mode,
                           int8_t *out_q, float *out_f, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!A || !W || !s_w || !bias || M < 1 || N < 1 || K < 16 || K % 16 || (M > 16 && K % 64))
        return fail(MNMT_EINVAL, "linear: bad shape M=%d N=%d K=%d", M, N, K);
    if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(W)) & 15)
        return fail(MNMT_EINVAL, "linear: A and W must be 16-byte aligned");
    if (M <= 16 && K > 2048) return fail(MNMT_EINVAL, "linear: K > 2048 at M <= 16");
    Epi e;
    std::memset(&e, 0, sizeof(e));
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    switch (mode) {
        case MNMT_EPI_Q8:
        case MNMT_EPI_RELU_Q8:
            if (!out_q || !inv_out) return fail(MNMT_EINVAL, "linear: int8 output needs out_q and inv_out");
            e.mode = mode == MNMT_EPI_Q8 ? EPI_Q8 : EPI_RELU_Q8;
            e.out = out_q;
            e.ldo = N;
            e.inv_out = inv_out;
            break;
        case MNMT_EPI_RESID:
        case MNMT_EPI_F32:
            if (!out_f) return fail(MNMT_EINVAL, "linear: fp32 output needs out_f");
            e.mode = mode == MNMT_EPI_RESID ? EPI_RESID : EPI_F32;
            e.f32 = out_f;
            e.ldf = N;
            e.gamma = gamma;
            break;
        default:
            return fail(MNMT_EINVAL, "linear: unknown mode %d", mode);
    }
    cudaError_t err = launch_linear(A, K, W, M, N, K, e, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "linear launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_linear_w4(const int8_t *A, const uint8_t *Wp, const float *s_w, const float *m_w,
                              const float *bias, float s_x, const float *inv_out, float gamma, int32_t M, int32_t N,
                              int32_t K, int32_t mode, int8_t *out_q, float *out_f, uint64_t *keys,
                              void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!A || !Wp || !s_w || !bias || M < 1 || N < 1 || K < 32 || K % 32 || K > 3072)
        return fail(MNMT_EINVAL, "linear_w4: bad shape M=%d N=%d K=%d", M, N, K);
    if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(Wp)) & 15)
        return fail(MNMT_EINVAL, "linear_w4: A and Wp must be 16-byte aligned");
    Epi e;
    std::memset(&e, 0, sizeof(e));
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    switch (mode) {
        case MNMT_EPI_Q8:
        case MNMT_EPI_RELU_Q8:
            if (!out_q || !inv_out) return fail(MNMT_EINVAL, "linear_w4: int8 output needs out_q and inv_out");
            e.mode = mode == MNMT_EPI_Q8 ? EPI_Q8 : EPI_RELU_Q8;
            e.out = out_q;
            e.ldo = N;
            e.inv_out = inv_out;
            break;
        case MNMT_EPI_RESID:
        case MNMT_EPI_F32:
            if (!out_f) return fail(MNMT_EINVAL, "linear_w4: fp32 output needs out_f");
            e.mode = mode == MNMT_EPI_RESID ? EPI_RESID : EPI_F32;
            e.f32 = out_f;
            e.ldf = N;
            e.gamma = gamma;
            break;
        case MNMT_EPI_ARGMAX:
            if (!keys) return fail(MNMT_EINVAL, "linear_w4: argmax needs keys");
            e.mode = EPI_ARGMAX;
            e.keys = reinterpret_cast<unsigned long long *>(keys);
            break;
        default:
            return fail(MNMT_EINVAL, "linear_w4: unknown mode %d", mode);
    }
    cudaError_t err = launch_linear_w4(A, K, Wp, m_w, M, N, K, e, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "linear_w4 launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_fake_quant(const float *x, size_t n, float s, float r_m, int32_t bits, int32_t minmax, float *y,
                               int32_t *codes, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!x || (!y && !codes) || bits < 2 || bits > 8 || !(s > 0.0f) || !std::isfinite(s) || !std::isfinite(r_m))
        return fail(MNMT_EINVAL, "fake_quant: bad argument");
    cudaError_t err = launch_fake_quant(x, n, s, r_m, bits, minmax ? 1 : 0, y, codes,
                                        static_cast<cudaStream_t>(cuda_stream));
    return err == cudaSuccess ? MNMT_OK : fail(MNMT_ECUDA, "fake_quant: %s", cudaGetErrorString(err));
}

extern "C" int mnmt_fake_quant_backward(const float *x, const float *g, size_t n, float s, float r_m, int32_t bits,
                                        int32_t minmax, float *gx, double *gs, double *gr, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!x || !g || !gx || !gs || bits < 2 || bits > 8 || !(s > 0.0f) || !std::isfinite(s) || !std::isfinite(r_m))
        return fail(MNMT_EINVAL, "fake_quant_backward: bad argument");
    cudaError_t err = launch_fake_quant_backward(x, g, n, s, r_m, bits, minmax ? 1 : 0, gx, gs, gr,
                                                 static_cast<cudaStream_t>(cuda_stream));
    return err == cudaSuccess ? MNMT_OK : fail(MNMT_ECUDA, "fake_quant_backward: %s", cudaGetErrorString(err));
}

extern "C" int mnmt_fake_quant_linear(const float *X, const float *W, float s_x, const float *s_w, const float *bias,
                                      int32_t M, int32_t N, int32_t K, int32_t wbits, void *workspace, float *y,
                                      void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!X || !W || !s_w || !bias || !workspace || !y || M < 1 || N < 1 || K < 16 || K % 16 || (M > 16 && K % 64) ||
        (M <= 16 && K > 2048) || wbits < 2 || wbits > 8 || !(s_x > 0.0f) || !std::isfinite(s_x))
        return fail(MNMT_EINVAL, "fake_quant_linear: bad argument or shape (M=%d N=%d K=%d)", M, N, K);
    if (reinterpret_cast<uintptr_t>(workspace) & 15)
        return fail(MNMT_EINVAL, "fake_quant_linear: workspace must be 16-byte aligned");
    int8_t *qx = static_cast<int8_t *>(workspace);
    int8_t *qw = qx + (((size_t)M * K + 15) & ~(size_t)15);
    cudaError_t err = launch_fake_quant_linear(X, W, s_x, s_w, bias, M, N, K, wbits, qx, qw, y,
                                               static_cast<cudaStream_t>(cuda_stream));
    return err == cudaSuccess ? MNMT_OK : fail(MNMT_ECUDA, "fake_quant_linear: %s", cudaGetErrorString(err));
}

extern "C" int mnmt_linear_tc(const uint16_t *A16, const uint16_t *W16, const float *s_w, const float *bias,
                              float s_x, const float *inv_out, float gamma, int32_t M, int32_t N, int32_t K,
                              int32_t mode, int8_t *out_q, float *out_f, uint64_t *keys, int32_t *status,
                              void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!A16 || !W16 || !s_w || !bias || M < 1 || N < 1 || !linear_tc_shape_ok(M, N, K, K, K, A16, W16))
        return fail(MNMT_EINVAL, "linear_tc: bad shape or alignment M=%d N=%d K=%d", M, N, K);
    Epi e;
    std::memset(&e, 0, sizeof(e));
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    switch (mode) {
        case MNMT_EPI_Q8:
        case MNMT_EPI_RELU_Q8:
            if (!out_q || !inv_out) return fail(MNMT_EINVAL, "linear_tc: int8 output needs out_q and inv_out");
            e.mode = mode == MNMT_EPI_Q8 ? EPI_Q8 : EPI_RELU_Q8;
            e.out = out_q;
            e.ldo = N;
            e.inv_out = inv_out;
            break;
        case MNMT_EPI_RESID:
        case MNMT_EPI_F32:
            if (!out_f) return fail(MNMT_EINVAL, "linear_tc: fp32 output needs out_f");
            e.mode = mode == MNMT_EPI_RESID ? EPI_RESID : EPI_F32;
            e.f32 = out_f;
            e.ldf = N;
            e.gamma = gamma;
            break;
        case MNMT_EPI_ARGMAX:
            if (!keys) return fail(MNMT_EINVAL, "linear_tc: argmax needs keys");
            e.mode = EPI_ARGMAX;
            e.keys = reinterpret_cast<unsigned long long *>(keys);
            break;
        default:
            return fail(MNMT_EINVAL, "linear_tc: unknown mode %d", mode);
    }
    cudaError_t err = launch_linear_tc(reinterpret_cast<const __half *>(A16), K, reinterpret_cast<const __half *>(W16),
                                       K, M, N, K, e, status, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "linear_tc launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_codes_to_f16(const int8_t *src, uint16_t *dst, size_t n, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!src || !dst || ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15))
        return fail(MNMT_EINVAL, "codes_to_f16: null or unaligned pointer");
    cudaError_t err = launch_codes_to_f16_flat(src, reinterpret_cast<__half *>(dst), n,
                                               static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "codes_to_f16 launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_wait_timeout_selftest(int32_t *status, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!status) return fail(MNMT_EINVAL, "wait_timeout_selftest: status is required");
    cudaError_t err = launch_wait_timeout_selftest(status, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "wait_timeout_selftest launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_linear_argmax(const int8_t *A, const int8_t *W, const float *s_w, const float *bias,
                                  float s_x, int32_t M, int32_t N, int32_t K, uint64_t *keys, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!A || !W || !s_w || !bias || !keys || M < 1 || N < 1 || K < 16 || K % 16 || (M > 16 && K % 64) ||
        (M <= 16 && K > 2048))
        return fail(MNMT_EINVAL, "linear_argmax: bad shape M=%d N=%d K=%d", M, N, K);
    if ((reinterpret_cast<uintptr_t>(A) | reinterpret_cast<uintptr_t>(W)) & 15)
        return fail(MNMT_EINVAL, "linear_argmax: A and W must be 16-byte aligned");
    Epi e;
    std::memset(&e, 0, sizeof(e));
    e.mode = EPI_ARGMAX;
    e.s_x = s_x;
    e.s_w = s_w;
    e.bias = bias;
    e.keys = reinterpret_cast<unsigned long long *>(keys);
    cudaError_t err = launch_linear(A, K, W, M, N, K, e, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "linear_argmax launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_attention_decode(const int8_t *q, const int8_t *Kc, const int8_t *Vc, const int32_t *n_keys,
                                     int32_t R, int32_t H, int32_t dh, int32_t T, float sigma, float rho,
                                     int8_t *ctx, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!q || !Kc || !Vc || !n_keys || !ctx || R < 1 || H < 1 || H > 16 || T < 1 || T > 1024 ||
        (dh != 32 && dh != 64 && dh != 128))
        return fail(MNMT_EINVAL, "attention: bad shape R=%d H=%d dh=%d T=%d", R, H, dh, T);
    AttnDecArgs a;
    std::memset(&a, 0, sizeof(a));
    a.q = q;
    a.kc = Kc;
    a.vc = Vc;
    a.ctx = ctx;
    a.R = R;
    a.H = H;
    a.dh = dh;
    a.T = T;
    a.beam = 1;
    a.n_keys = n_keys;
    a.sigma = sigma;
    a.rho = rho;
    cudaError_t err = launch_attention_decode(a, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "attention launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}

extern "C" int mnmt_layernorm(const float *r, const float *g, const float *b, int32_t M, int32_t d, float inv,
                              float *out_f, int8_t *out_q, int32_t *status, void *cuda_stream) {
    int rc = lib_init();
    if (rc) return rc;
    if (!r || !g || !b || M < 1 || d < 1 || d > 2048)
        return fail(MNMT_EINVAL, "layernorm: d must be in [1, 2048]");
    LnArgs a;
    std::memset(&a, 0, sizeof(a));
    a.r = r;
    a.g = g;
    a.b = b;
    a.M = M;
    a.d = d;
    a.inv = inv;
    a.out_f = out_f;
    a.out_q = out_q;
    a.status = status;
    cudaError_t err = launch_layernorm(a, static_cast<cudaStream_t>(cuda_stream));
    if (err != cudaSuccess) return fail(MNMT_ECUDA, "layernorm launch: %s", cudaGetErrorString(err));
    return MNMT_OK;
}
