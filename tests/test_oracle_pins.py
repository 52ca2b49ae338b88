"""Pins of the CPU oracle to things other than itself: an independent float64
brute force, closed forms, exact invariants and library conversions."""
import math

import numpy as np
import pytest

import oracle
import synth
from synth import workloads as W
from tests import f64_reference as ref

F32_TINY = W.scaled(W.TINY, n_layers=2, d_model=64, n_q_heads=4, n_kv_heads=2, head_dim=16,
                    ffn_dim=96, vocab=97, kv_dtype=oracle.KV_F32)


def _weights(shape, seed=0):
    w = synth.model_weights(shape, seed=seed)
    # non-trivial norm gains so a dropped gain is caught
    rng = np.random.default_rng(seed + 11)
    for lw in w["layers"]:
        lw["attn_norm"] = rng.uniform(0.5, 1.5, shape["d_model"]).astype(np.float32)
        lw["ffn_norm"] = rng.uniform(0.5, 1.5, shape["d_model"]).astype(np.float32)
    w["final_norm"] = rng.uniform(0.5, 1.5, shape["d_model"]).astype(np.float32)
    return w


def _rel(a, b):
    return float(np.max(np.abs(np.asarray(a, np.float64) - b)) / np.max(np.abs(b)))


# ---- P-1: float64 brute force --------------------------------------------------

@pytest.mark.parametrize("hq,hkv", [(4, 2), (4, 4), (4, 1)])
def test_oracle_matches_float64_bruteforce(hq, hkv):
    sh = W.scaled(F32_TINY, n_q_heads=hq, n_kv_heads=hkv)
    w = _weights(sh)
    toks = synth.tokens(synth.SEED_CONTEXT, 0, 37, sh["vocab"])
    kv = oracle.KVState(sh, 64)
    lg = oracle.prefill(sh, w, kv, toks, 0)
    rlg, Ks, Vs = ref.forward(sh, w, toks)
    assert _rel(lg, rlg) < 2e-5
    for l in range(sh["n_layers"]):
        assert _rel(kv.k[l, :37], Ks[l]) < 2e-5
        assert _rel(kv.v[l, :37], Vs[l]) < 2e-5
    # the weights are large enough that a wrong head mapping changes the answer
    assert np.max(np.abs(rlg)) > 1e-2


def test_bruteforce_detects_planted_rope_mistake():
    """A plausible mistake (interleaved instead of half-split rotary pairs)
    planted in a copy of the oracle's inputs path is caught by the pin."""
    sh = F32_TINY
    w = _weights(sh)
    toks = synth.tokens(synth.SEED_CONTEXT, 1, 20, sh["vocab"])
    rlg, _, _ = ref.forward(sh, w, toks)
    # emulate interleaved pairing by permuting q/k output features: the oracle
    # then computes the interleaved convention relative to the original weights
    hd = sh["head_dim"]
    perm = np.concatenate([np.arange(0, hd, 2), np.arange(1, hd, 2)])
    w2 = synth.model_weights(sh)
    for a, b in zip(w2["layers"], w["layers"]):
        a.update({k: b[k] for k in b})
        for k, nh in (("wq", sh["n_q_heads"]), ("wk", sh["n_kv_heads"])):
            m = b[k].reshape(nh, hd, -1)[:, perm, :]
            a[k] = np.ascontiguousarray(m.reshape(nh * hd, -1))
    w2["final_norm"] = w["final_norm"]
    kv = oracle.KVState(sh, 32)
    lg = oracle.prefill(sh, w2, kv, toks, 0)
    assert _rel(lg, rlg) > 1e-3


def test_kv_is_rounded_after_rotary():
    """Stored layer-0 K/V in bf16 (fp16) mode equal the rounding of the exact
    fp32-mode values: the rounding point is after RoPE (Sec. 4.3 footnote:
    chunks hold FP16 K/V)."""
    for kvd, conv in ((oracle.KV_BF16, "bf16"), (oracle.KV_FP16, "f16")):
        sh32 = F32_TINY
        sh = W.scaled(F32_TINY, kv_dtype=kvd)
        w = _weights(sh)
        toks = synth.tokens(synth.SEED_CONTEXT, 2, 25, sh["vocab"])
        kv32 = oracle.KVState(sh32, 32)
        oracle.prefill(sh32, w, kv32, toks, 0, logits=False)
        kvr = oracle.KVState(sh, 32)
        oracle.prefill(sh, w, kvr, toks, 0, logits=False)
        exact = kv32.k[0, :25]
        if conv == "f16":
            want = exact.astype(np.float16).astype(np.float32)
        else:
            import torch
            want = torch.from_numpy(exact).to(torch.bfloat16).float().numpy()
        assert np.array_equal(kvr.k[0, :25], want)
        assert not np.array_equal(kvr.k[0, :25], exact)


# ---- P-2: closed forms ----------------------------------------------------------

def test_single_key_attention_returns_value():
    rng = np.random.default_rng(0)
    q = rng.standard_normal((1, 4, 8)).astype(np.float32)
    k = rng.standard_normal((1, 2, 8)).astype(np.float32)
    v = rng.standard_normal((1, 2, 8)).astype(np.float32)
    out = oracle.attention(q, [0], k, v)
    assert np.array_equal(out[0, 0], v[0, 0]) and np.array_equal(out[0, 3], v[0, 1])


def test_identical_keys_average_causal_values():
    rng = np.random.default_rng(1)
    ctx = 9
    k = np.repeat(rng.standard_normal((1, 1, 16)).astype(np.float32), ctx, axis=0)
    v = rng.standard_normal((ctx, 1, 16)).astype(np.float32)
    q = rng.standard_normal((3, 2, 16)).astype(np.float32)
    pos = [0, 4, 8]
    out = oracle.attention(q, pos, k, v)
    for i, p in enumerate(pos):
        np.testing.assert_allclose(out[i, 1], v[: p + 1, 0].mean(0), rtol=1e-5, atol=1e-6)


def test_attention_scale_and_causality():
    """Two keys: weights follow softmax(q.k/sqrt(hd)); a later key is ignored."""
    hd = 4
    q = np.array([[[1.0, 0, 0, 0]]], np.float32)
    k = np.array([[[2.0, 0, 0, 0]], [[0.0, 0, 0, 0]], [[50.0, 0, 0, 0]]], np.float32)
    v = np.array([[[1.0, 0, 0, 0]], [[0.0, 1, 0, 0]], [[0.0, 0, 1, 0]]], np.float32)
    out = oracle.attention(q, [1], k, v)
    w0 = math.exp(2.0 / math.sqrt(hd))
    w1 = 1.0
    np.testing.assert_allclose(out[0, 0], [w0 / (w0 + w1), w1 / (w0 + w1), 0, 0], rtol=1e-6)


def test_rope_identity_at_zero_and_norm_preserving():
    rng = np.random.default_rng(2)
    x = rng.standard_normal((5, 3, 32)).astype(np.float32)
    y = oracle.rope(x, [0, 1, 7, 1000, 32000], 500000.0)
    assert np.array_equal(y[0], x[0])
    half = 16
    n0 = x[..., :half] ** 2 + x[..., half:] ** 2
    n1 = y[..., :half] ** 2 + y[..., half:] ** 2
    np.testing.assert_allclose(n1, n0, rtol=1e-5)


def test_rope_relative_position_property():
    """<R(m) q, R(n) k> depends on m - n only (RoFormer Sec. 3.4)."""
    rng = np.random.default_rng(3)
    q = rng.standard_normal((1, 1, 64)).astype(np.float32)
    k = rng.standard_normal((1, 1, 64)).astype(np.float32)
    th = 10000.0
    a = float(np.dot(oracle.rope(q, [10], th).ravel(), oracle.rope(k, [3], th).ravel()))
    b = float(np.dot(oracle.rope(q, [107], th).ravel(), oracle.rope(k, [100], th).ravel()))
    assert abs(a - b) < 1e-4


def test_rope_table_angles():
    c, s = oracle.rope_table(40000, 128, 500000.0)
    for p, i in ((1, 0), (1, 1), (33, 17), (32767, 63), (39999, 5)):
        ang = p * 500000.0 ** (-2.0 * i / 128)
        assert c[p, i] == np.float32(math.cos(ang)) and s[p, i] == np.float32(math.sin(ang))


def test_rmsnorm_constant_vector():
    d, c, eps = 64, -0.75, 1e-5
    g = np.linspace(0.5, 2.0, d).astype(np.float32)
    y = oracle.rmsnorm(np.full((1, d), c, np.float32), g, eps)
    np.testing.assert_allclose(y[0], c * g / math.sqrt(c * c + eps), rtol=1e-6)


def test_linear_identity_and_swiglu():
    d = 32
    one = np.uint16(0x3F80)  # bf16 1.0
    w = np.zeros((d, d), np.uint16)
    w[np.arange(d), np.arange(d)] = one
    x = np.random.default_rng(4).standard_normal((3, d)).astype(np.float32)
    assert np.array_equal(oracle.linear(x, w), x)
    g = np.array([0.0, 1.0, -1.0, 20.0], np.float32)
    u = np.array([5.0, 2.0, 2.0, 1.0], np.float32)
    np.testing.assert_allclose(oracle.swiglu(g, u),
                               [0.0, 2 / (1 + math.exp(-1)), -2 / (1 + math.exp(1)), 20.0],
                               rtol=1e-6)


def test_kv_rounding_matches_libraries():
    import torch
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(10000) * s for s in (1e-6, 1e-3, 1.0, 100.0, 7e4)])
    x = np.concatenate([x, [0.0, -0.0, 65504.0, 65519.0, 65520.0, 1e5, 2.0 ** -25, 2.0 ** -24 * 1.5,
                            5.96e-8, 6.1e-5]]).astype(np.float32)
    with np.errstate(over="ignore"):
        want16 = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(oracle.to_f16_bits(x), want16)
    tb = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.to_bf16_bits(x), tb)


# ---- P-3: exact invariants ------------------------------------------------------

def test_chunked_prefill_equals_full_prefill_bitwise():
    sh = W.scaled(F32_TINY, kv_dtype=oracle.KV_BF16)
    w = _weights(sh)
    toks = synth.tokens(synth.SEED_CONTEXT, 3, 50, sh["vocab"])
    kv_full = oracle.KVState(sh, 64)
    lg_full = oracle.prefill(sh, w, kv_full, toks, 0)
    kv_ch = oracle.KVState(sh, 64)
    for a, b in ((0, 16), (16, 17), (17, 40), (40, 50)):
        lg = oracle.prefill(sh, w, kv_ch, toks[a:b], a)
    assert np.array_equal(lg, lg_full)
    assert np.array_equal(kv_ch.k[:, :50], kv_full.k[:, :50])
    assert np.array_equal(kv_ch.v[:, :50], kv_full.v[:, :50])


def test_recompute_tail_plus_prompt_equals_full_prefill_bitwise():
    """Drop the KV tail [p, N), re-run its rows fused with the prompt: the
    logits and KV equal those of one prefill of context || prompt."""
    sh = W.scaled(F32_TINY, kv_dtype=oracle.KV_BF16)
    w = _weights(sh)
    ctx = synth.tokens(synth.SEED_CONTEXT, 4, 48, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 4, 7, sh["vocab"])
    kv_ref = oracle.KVState(sh, 64)
    lg_ref = oracle.prefill(sh, w, kv_ref, np.concatenate([ctx, prm]), 0)
    kv = oracle.KVState(sh, 64)
    oracle.prefill(sh, w, kv, ctx, 0, logits=False)
    p = 32
    kv.k[:, p:] = np.nan
    kv.v[:, p:] = np.nan
    rows = np.concatenate([ctx[p:], prm])
    lg = oracle.forward(sh, w, kv, rows, np.arange(p, 55))
    assert np.array_equal(lg, lg_ref)
    assert np.array_equal(kv.k[:, :55], kv_ref.k[:, :55])


def test_row_order_does_not_matter():
    sh = W.scaled(F32_TINY, kv_dtype=oracle.KV_FP16)
    w = _weights(sh)
    toks = synth.tokens(synth.SEED_CONTEXT, 5, 30, sh["vocab"])
    kv_a = oracle.KVState(sh, 32)
    oracle.prefill(sh, w, kv_a, toks, 0, logits=False)
    perm = synth.permutation(synth.SEED_EVICT, 9, 30)
    kv_b = oracle.KVState(sh, 32)
    oracle.forward(sh, w, kv_b, toks[perm], perm, logits=False)
    assert np.array_equal(kv_a.k[:, :30], kv_b.k[:, :30])


# ---- P-6: a library routine for the same operation ---------------------------

@pytest.mark.parametrize("hq,hkv,hd", [(4, 2, 64), (24, 8, 128), (8, 8, 32)])
def test_attention_matches_torch_sdpa(hq, hkv, hd):
    """The oracle's causal GQA attention over positions equals torch's
    scaled_dot_product_attention (CPU, float64) with each KV head repeated
    over its query group and a key mask of key position <= query position."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(hq + hkv + hd)
    ctx, n = 37, 6
    q = rng.standard_normal((n, hq, hd)).astype(np.float32)
    k = rng.standard_normal((ctx, hkv, hd)).astype(np.float32)
    v = rng.standard_normal((ctx, hkv, hd)).astype(np.float32)
    pos = np.array([0, 3, 17, 18, 30, 36])
    got = oracle.attention(q, pos, k, v)
    g = hq // hkv
    qt = torch.from_numpy(q.astype(np.float64)).permute(1, 0, 2)                 # [hq][n][hd]
    kt = torch.from_numpy(k.astype(np.float64)).permute(1, 0, 2).repeat_interleave(g, 0)
    vt = torch.from_numpy(v.astype(np.float64)).permute(1, 0, 2).repeat_interleave(g, 0)
    mask = torch.from_numpy(np.arange(ctx)[None, :] <= pos[:, None])              # [n][ctx]
    want = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
    np.testing.assert_allclose(got, want.permute(1, 0, 2).numpy(), rtol=2e-5, atol=2e-6)


def test_linear_matches_a_float64_matmul_on_a_non_square_weight():
    """x W^T with W [n_out][n_in] in bf16 bits, against numpy's float64 matmul
    of the decoded weights (a transposed operand or a swapped dimension
    fails on the 48 x 80 weight; the identity pin above cannot tell)."""
    rng = np.random.default_rng(9)
    x = rng.standard_normal((5, 80)).astype(np.float32)
    w_bits = synth.normal_bf16(3, 77, (48, 80), sigma=0.05)
    w = synth.bf16_bits_to_f32(w_bits).astype(np.float64)
    want = x.astype(np.float64) @ w.T
    np.testing.assert_allclose(oracle.linear(x, w_bits), want, rtol=1e-5, atol=1e-6)


def test_rmsnorm_matches_torch_rms_norm():
    """RMSNorm with gains against torch.nn.functional.rms_norm in float64 on
    random rows of varied scale."""
    torch = pytest.importorskip("torch")
    if not hasattr(torch.nn.functional, "rms_norm"):
        pytest.skip("torch without rms_norm")
    rng = np.random.default_rng(12)
    x = (rng.standard_normal((7, 96)) * rng.uniform(0.01, 30.0, (7, 1))).astype(np.float32)
    g = (1.0 + 0.3 * rng.standard_normal(96)).astype(np.float32)
    want = torch.nn.functional.rms_norm(torch.from_numpy(x.astype(np.float64)), (96,),
                                        torch.from_numpy(g.astype(np.float64)), eps=1e-5).numpy()
    np.testing.assert_allclose(oracle.rmsnorm(x, g, 1e-5), want, rtol=2e-6, atol=1e-7)
