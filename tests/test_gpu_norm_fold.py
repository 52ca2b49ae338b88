"""RMSNorm folded into the projections of short row sets (5-256 rows), on the
GPU through the C ABI, against the oracle's pre-norm decoder layer.

The fold rests on RMSNorm(x) W^T = diag(1 / RMS(x)) ((x * g) W^T): the
residual-add GEMM that finishes x also writes h = fp16(x * g) and each row's
sum of x^2 per 128-column tile, and the next projection scales its rows by
rstd.  What is fixed exactly is checked exactly (h is the fp16 rounding of the
returned x times g); the projection is checked against the oracle's
RMSNorm + linear (+ SwiGLU) with the bound that the fp16 rounding of h and of
the output gives, element by element.  End to end, prefills of 200 and 37 rows
and two one-token steps (the GEMV kernels' one-row fold, also taken by the
last layer's logits row of every prefill) match the oracle's prefill of the
same tokens as the separate-norm path does, and run the RMSNorm kernel only
for the first layer's attention norm."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
from tests.gpu_util import bf16_dev, f32_dev, to_np_u16, f16_to_f32, f16_bits, rel_err, \
    bf16_weights_exact_in_f16

pytestmark = pytest.mark.gpu

U16 = 2.0 ** -11  # fp16 unit roundoff (round to nearest)
EPS = 1e-5


def _torch():
    import torch
    return torch


def _rand_bf16(tid, shape, sigma=1.0):
    return synth.normal_bf16(13, tid, shape, sigma=sigma)


# (rows, d = the producer's N and the consumer's K, the producer's K, the
# consumer's N, consumer epilogue: 0 fp16 store, 2 SwiGLU)
FOLD_SHAPES = [
    (128, 3072, 3072, 5120, 0),    # 3B: O -> QKV (split-K consumer)
    (128, 3072, 8192, 16384, 2),   # 3B: down -> gate/up (row-scaled persistent kernel, 128-wide tiles)
    (256, 3072, 3072, 16384, 2),   # two row tiles: 256-wide persistent tiles
    (200, 2048, 2048, 3072, 0),    # 1B widths, ragged rows (split-K over two row tiles)
    (5, 2048, 8192, 16384, 2),     # the fewest rows the fold takes
    (37, 256, 688, 1408, 2),       # tiny widths (split-K SwiGLU consumer; FFN padded to 704)
    (64, 1024, 1024, 1040, 0),     # consumer N not a multiple of 128: persistent 64-wide tiles
    (130, 1024, 1024, 10240, 0),   # 80 column tiles: no split, persistent store
]


@pytest.mark.parametrize("mm,d,kp,nn,epi", FOLD_SHAPES)
def test_folded_norm_pair_matches_the_oracle(mm, d, kp, nn, epi):
    torch = _torch()
    rng = np.random.default_rng(mm * 7 + d)
    a = f16_bits(synth.bf16_bits_to_f32(_rand_bf16(1, (mm, kp))))
    wpb, wph = bf16_weights_exact_in_f16(_rand_bf16(2, (d, kp), sigma=0.05))
    x0 = rng.standard_normal((mm, d)).astype(np.float32)
    g = (1.0 + 0.1 * rng.standard_normal(d)).astype(np.float32)
    wb, wh = bf16_weights_exact_in_f16(_rand_bf16(3, (nn, d), sigma=0.05))
    ncol = nn // 2 if epi == 2 else nn
    w_dev = bf16_dev(m.mzc_k_swiglu_pack(wh[: nn // 2], wh[nn // 2:]) if epi == 2 else wh)
    nt = d // 128
    runs = []
    for _ in range(2):  # the same bits on a second run
        x = f32_dev(x0)
        h = torch.zeros((mm, d), dtype=torch.int16, device="cuda")
        ss = torch.zeros((mm, nt), dtype=torch.float32, device="cuda")
        out = torch.zeros((mm, ncol), dtype=torch.int16, device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        m.mzc_k_gemm_norm_out(bf16_dev(a), bf16_dev(wph), x, mm, d, kp, f32_dev(g), h, ss, st)
        m.mzc_k_gemm_norm_in(h, w_dev, out, mm, nn, d, epi, ss, EPS, st)
        torch.cuda.synchronize()
        runs.append((x.cpu().numpy(), to_np_u16(h), ss.cpu().numpy(), to_np_u16(out), int(st.item())))
    for r0, r1 in zip(runs[0], runs[1]):
        assert np.array_equal(np.asarray(r0), np.asarray(r1))
    xg, hg, ssg, outg, status = runs[0]
    assert status == 0
    # the residual add, as the plain mzc_k_gemm residual-add test bounds it
    x_ref = x0 + oracle.linear(f16_to_f32(a), wpb)
    assert np.max(np.abs(xg - x_ref)) <= 1e-4 * np.max(np.abs(x_ref))
    # h is the fp16 rounding of (returned x) * g, bit for bit
    assert np.array_equal(hg, f16_bits(xg * g))
    # per-tile sums of squares of the returned x
    ss_ref = (xg.astype(np.float64) ** 2).reshape(mm, nt, 128).sum(axis=2)
    assert rel_err(ssg, ss_ref) < 1e-5
    # the projection of RMSNorm(x): the oracle's norm and linear layer on the
    # returned x; the GPU multiplies h, not the normalised row, so each output
    # may differ by the fp16 rounding of its inputs (u * sum |y_k w_k|) and of
    # itself (u * |ref|), plus fp32 accumulation noise
    y = oracle.rmsnorm(xg, g, EPS).astype(np.float64)
    got = f16_to_f32(outg).astype(np.float64)
    wf = synth.bf16_bits_to_f32(wb).astype(np.float64)
    mag = np.abs(y) @ np.abs(wf).T
    if epi == 0:
        ref = oracle.linear(y.astype(np.float32), wb).astype(np.float64)
        bound = U16 * mag + U16 * np.abs(ref) + 1e-5 * np.max(np.abs(ref))
    else:
        f = nn // 2
        gate = oracle.linear(y.astype(np.float32), wb[:f]).astype(np.float64)
        up = oracle.linear(y.astype(np.float32), wb[f:]).astype(np.float64)
        ref = oracle.swiglu(gate, up).astype(np.float64)
        sig = 1.0 / (1.0 + np.exp(-gate))
        dsilu = np.abs(sig * (1.0 + gate * (1.0 - sig)))  # |d silu / d gate|
        e_gate, e_up = U16 * mag[:, :f] * 1.01, U16 * mag[:, f:] * 1.01
        bound = (dsilu * np.abs(up) * e_gate + np.abs(gate * sig) * e_up + e_gate * e_up
                 + U16 * np.abs(ref) + 2e-5 * np.max(np.abs(ref)))
    assert np.all(np.abs(got - ref) <= bound)


def test_folded_norm_rejects_what_it_cannot_fold():
    """Rows outside 5..256, a producer N that is not a multiple of 128, or a
    residual-add consumer are refused before anything is launched."""
    def st(fn, *args):
        return m.status_of(fn, *args)
    p = 16  # any nonzero address: the checks come first
    assert st("mzc_k_gemm_norm_out", p, p, p, 4, 256, 256, p, p, p, None, None) == m.MZC_ERR_INVALID
    assert st("mzc_k_gemm_norm_out", p, p, p, 257, 256, 256, p, p, p, None, None) == m.MZC_ERR_INVALID
    assert st("mzc_k_gemm_norm_out", p, p, p, 64, 200, 256, p, p, p, None, None) == m.MZC_ERR_INVALID
    assert st("mzc_k_gemm_norm_in", p, p, p, 64, 256, 256, 1, p, 1e-5, None, None) == m.MZC_ERR_INVALID
    assert st("mzc_k_gemm_norm_in", p, p, p, 64, 256, 200, 0, p, 1e-5, None, None) == m.MZC_ERR_INVALID


CASES = {
    "tiny": W.TINY,
    "1b_widths": W.scaled(W.ONE_B, n_layers=3, vocab=1024, max_ctx=1024),
    "3b_widths": W.scaled(W.THREE_B, n_layers=3, vocab=1024, max_ctx=1024),
}


@pytest.mark.parametrize("name", list(CASES))
def test_folded_norm_prefill_matches_the_oracle(name):
    """A 200-row context prefill, a 37-row prompt prefill and two one-token
    steps (all folded) against the oracle's prefill of the same tokens: logits
    max-abs <= 2e-2, K/V max|d| / max|ref| <= 1e-2 per layer, as for the
    separate norm launches, which run beside it; the fold leaves one RMSNorm
    launch a prefill.  The same with the rotary write inside the QKV
    projection (option fused_rope): no rotary launch for the 5-256-row sets,
    and every position it wrote matches."""
    sh = CASES[name]
    L = sh["n_layers"]
    w = synth.model_weights(sh)
    # distinct norm gains per layer and norm, so that a gain applied to the
    # wrong norm shows (the synthetic model's gains are all ones)
    rng = np.random.default_rng(5)
    for lw in w["layers"]:
        for key in ("attn_norm", "ffn_norm"):
            lw[key] = (1.0 + 0.25 * rng.standard_normal(sh["d_model"])).astype(np.float32)
    ctx = synth.tokens(synth.SEED_CONTEXT, 21, 200, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 21, 37, sh["vocab"])
    kv_ref = oracle.KVState(sh, sh["max_ctx"])
    lg_ctx = oracle.prefill(sh, w, kv_ref, ctx, 0)
    lg_prm = oracle.prefill(sh, w, kv_ref, prm, 200)
    steps = synth.tokens(synth.SEED_PROMPT, 22, 2, sh["vocab"])
    lg_steps = [oracle.prefill(sh, w, kv_ref, steps[i:i + 1], 237 + i) for i in range(2)]
    n_tok = 239
    for sep, fused_rope in ((0, 0), (0, 1), (1, 0)):
        c = m.mzc_create(sh, w, separate_norm=sep, fused_rope=fused_rope)
        try:
            norms, ropes = [], []
            lgs = []
            for toks in (ctx, prm, steps[:1], steps[1:]):
                m.mzc_set_kernel_timing(c, 0)  # resets the launch counters
                out = np.empty(sh["vocab"], np.float32)
                m.mzc_prefill(c, toks, out)
                lgs.append(out)
                norms.append(m.mzc_kernel_stats(c, m.MZC_K_RMSNORM).launches)
                ropes.append(m.mzc_kernel_stats(c, m.MZC_K_ROPE_KV).launches)
            assert np.max(np.abs(lgs[0] - lg_ctx)) < 2e-2
            assert np.max(np.abs(lgs[1] - lg_prm)) < 2e-2
            for i in range(2):
                assert np.max(np.abs(lgs[2 + i] - lg_steps[i])) < 2e-2
            k, v = m.mzc_read_kv_all(c, n_tok, sh)
            for l in range(L):
                assert rel_err(k[l], kv_ref.k[l, :n_tok]) < 1e-2
                assert rel_err(v[l], kv_ref.v[l, :n_tok]) < 1e-2
            # separate: every layer's attention norm, the MLP norms of the first
            # L - 1 layers over all rows, the last layer's over the logits row
            assert norms == ([1] * 4 if sep == 0 else [2 * L] * 4)
            # fused_rope: the rotary write runs inside the QKV projection for the
            # 200- and 37-row prefills; one-row steps keep their rotary launch
            assert ropes == ([0, 0, L, L] if fused_rope else [L] * 4)
        finally:
            m.mzc_destroy(c)
