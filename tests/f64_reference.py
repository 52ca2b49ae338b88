"""Independent float64 brute-force forward of the same decoder, written with
whole-matrix numpy operations (full score matrix with a causal mask, rotary
embedding as a complex multiplication, grouped-query attention by repeating
KV heads) so that it shares no structure with the row-by-row fp32 oracle.
Used only to pin the oracle on tiny shapes."""
from __future__ import annotations

import numpy as np


def bf16_to_f64(bits):
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def rmsnorm(x, g, eps):
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope(x, pos, theta):
    """x[n, heads, hd]; pairs (i, i + hd/2) rotated by pos * theta^(-2i/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    inv = theta ** (-2.0 * np.arange(half) / hd)
    ang = pos[:, None].astype(np.float64) * inv[None, :]
    z = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * ang)[:, None, :]
    return np.concatenate([z.real, z.imag], axis=-1)


def forward(shape, weights, tokens, kv_round=None):
    """Full prefill of `tokens` from position 0. Returns (logits of the last
    row, K per layer [n, hkv, hd], V per layer). kv_round(x) optionally maps
    the stored K/V values (after rotary) to the storage precision."""
    d, hq, hkv, hd = shape["d_model"], shape["n_q_heads"], shape["n_kv_heads"], shape["head_dim"]
    eps, theta = shape["rms_eps"], shape["rope_theta"]
    n = len(tokens)
    pos = np.arange(n)
    x = bf16_to_f64(weights["embed"])[np.asarray(tokens)]
    mask = pos[None, :] <= pos[:, None]  # [query, key]
    Ks, Vs = [], []
    for lw in weights["layers"]:
        W = {k: bf16_to_f64(lw[k]) for k in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")}
        h = rmsnorm(x, lw["attn_norm"].astype(np.float64), eps)
        q = (h @ W["wq"].T).reshape(n, hq, hd)
        k = (h @ W["wk"].T).reshape(n, hkv, hd)
        v = (h @ W["wv"].T).reshape(n, hkv, hd)
        q, k = rope(q, pos, theta), rope(k, pos, theta)
        if kv_round is not None:
            k, v = kv_round(k), kv_round(v)
        Ks.append(k); Vs.append(v)
        kr = np.repeat(k, hq // hkv, axis=1)  # query head a -> KV head a // group
        vr = np.repeat(v, hq // hkv, axis=1)
        s = np.einsum("qhc,khc->hqk", q, kr) / np.sqrt(hd)
        s = np.where(mask[None], s, -np.inf)
        s = s - s.max(axis=-1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=-1, keepdims=True)
        a = np.einsum("hqk,khc->qhc", p, vr).reshape(n, hq * hd)
        x = x + a @ W["wo"].T
        h = rmsnorm(x, lw["ffn_norm"].astype(np.float64), eps)
        gt = h @ W["w_gate"].T
        up = h @ W["w_up"].T
        x = x + (gt / (1.0 + np.exp(-gt)) * up) @ W["w_down"].T
    hf = rmsnorm(x[-1], weights["final_norm"].astype(np.float64), eps)
    logits = bf16_to_f64(weights["lm_head"]) @ hf
    return logits, Ks, Vs
