"""Parameter and multiply-accumulate accounting of the encoder-decoder model.

TEST INFRASTRUCTURE (part of the oracle's definition of the model's shape).
Counts follow the model as the oracle computes it: one embedding table shared
by source and target and tied to the output projection unless the embedding
is factorised (Sec. 2.1 "Scaling E", App. D shared vocabularies); an encoder
layer holds self-attention (W_q, W_k, W_v, W_o) and an FFN (W_1, W_2); a
decoder layer adds cross-attention (App. A).  Parameters count weight
matrices only; "FLOPs" in the paper's tables are multiply-accumulates.
"""
from __future__ import annotations


def params(V, d, F, n_enc, n_dec, E=None, tied=True):
    """(total, without embedding) weight-matrix parameter counts."""
    E = d if E is None else E
    emb = V * E + (E * d if E != d else 0)
    if not tied or E != d:
        emb_out = V * d
    else:
        emb_out = 0
    enc_layer = 4 * d * d + 2 * d * F
    dec_layer = 8 * d * d + 2 * d * F
    body = n_enc * enc_layer + n_dec * dec_layer
    return emb + emb_out + body, body


def macs(V, d, F, n_enc, n_dec, src_len, tgt_len):
    """Multiply-accumulates to translate one sentence of src_len tokens into
    tgt_len tokens with incremental decoding: every encoder and decoder linear
    once per token, attention score and context products, and the output
    projection once per target token."""
    enc_lin = src_len * n_enc * (4 * d * d + 2 * d * F)
    enc_att = n_enc * 2 * src_len * src_len * d
    dec_lin = tgt_len * n_dec * (4 * d * d + 2 * d * F)   # self qkv+o, ffn
    dec_cross_q_o = tgt_len * n_dec * 2 * d * d
    dec_cross_kv = n_dec * src_len * 2 * d * d               # once per source
    dec_self_att = n_dec * 2 * d * sum(t + 1 for t in range(tgt_len))
    dec_cross_att = n_dec * 2 * tgt_len * src_len * d
    out = tgt_len * d * V
    return (enc_lin + enc_att + dec_lin + dec_cross_q_o + dec_cross_kv + dec_self_att
            + dec_cross_att + out)
