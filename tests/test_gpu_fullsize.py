"""Parity at the full sizes of the benchmarked workloads, in the launch
configuration bench.py uses (same ctx options), on outputs the CPU oracle can
compute one at a time.

The oracle cannot prefill a 32k-token context on the CPU, so these checks are
KV-conditioned: after the GPU's restore + prefill, the GPU's KV of every
position except one row is read back and the oracle recomputes that one row
through every layer over it -- giving that row's K/V at every layer and, for
the last prompt row, the first-token logits.  Copy restores are checked bit
for bit against the pre-eviction state and a no-eviction run."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
from tests.gpu_util import rel_err

pytestmark = pytest.mark.gpu

LOGIT_TOL = 2e-2
KV_TOL = 1e-2


def _ctx(sc):
    sh = sc["model"]
    w = synth.model_weights(sh)
    c = m.mzc_create(sh, w, max_rows=min(sh["max_ctx"], 16384 + 1024))  # as bench.py
    ctx_tok = synth.tokens(synth.SEED_CONTEXT, 0, sc["context"], sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 0, sc["prompt"], sh["vocab"])
    m.mzc_prefill(c, ctx_tok)
    return sh, w, c, ctx_tok, prm


def _kv_state(k, v):
    kv = oracle.KVState.__new__(oracle.KVState)
    kv.k, kv.v, kv.max_ctx = k, v, k.shape[1]
    return kv


def _row_check(sh, w, k, v, row_pos, token, gpu_logits=None):
    """Oracle forward of one row at row_pos over the GPU's K/V of every other
    position (k, v: [n_layers][n][n_kv_heads][head_dim], as read back, left
    unchanged); compares that row's K/V per layer and (optionally) the
    first-token logits."""
    kv = _kv_state(k, v)
    gpu_k_row, gpu_v_row = k[:, row_pos].copy(), v[:, row_pos].copy()
    kv.k[:, row_pos] = np.nan
    kv.v[:, row_pos] = np.nan
    try:
        lg = oracle.forward(sh, w, kv, [token], [row_pos], logits=gpu_logits is not None)
        for l in range(sh["n_layers"]):
            assert rel_err(gpu_k_row[l], kv.k[l, row_pos]) < KV_TOL, (row_pos, l)
            assert rel_err(gpu_v_row[l], kv.v[l, row_pos]) < KV_TOL, (row_pos, l)
        if gpu_logits is not None:
            assert np.max(np.abs(gpu_logits - lg)) < LOGIT_TOL
    finally:
        k[:, row_pos], v[:, row_pos] = gpu_k_row, gpu_v_row


def _one_row_check(sh, w, c, n_total, row_pos, token, gpu_logits=None):
    k, v = m.mzc_read_kv_all(c, n_total, sh)
    _row_check(sh, w, k, v, row_pos, token, gpu_logits)
    return k, v


def test_1b_recompute_full_size():
    """The 1B-class workload bench.py times: 8192-token context, tail
    [4096, 8192) dropped and recomputed fused with a 128-token prompt."""
    sc = W.SCENARIOS["1b_recompute"]
    sh, w, c, ctx_tok, prm = _ctx(sc)
    N, P = sc["context"], sc["prompt"]
    k_pre, v_pre = m.mzc_read_kv_all(c, N, sh)
    m.mzc_evict(c, 0, sh["n_layers"], N - sc["evict_tail"], N, m.MZC_DROP)
    m.mzc_restore_async(c)
    m.mzc_recompute_tail(c, N - sc["evict_tail"], sc["evict_tail"])
    logits = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, prm, logits)
    # recomputed K/V equal the pre-eviction K/V (recompute is an exact restore)
    k, v = _one_row_check(sh, w, c, N + P, N + P - 1, prm[-1], logits)
    p = N - sc["evict_tail"]
    for l in range(sh["n_layers"]):
        assert rel_err(k[l, p:N], k_pre[l, p:N]) < KV_TOL
        assert rel_err(v[l, p:N], v_pre[l, p:N]) < KV_TOL
        assert np.array_equal(k[l, :p], k_pre[l, :p])  # resident prefix untouched
    # eight recomputed rows, evenly spaced over [p, N) (first and last
    # included), each checked one by one against the oracle
    for r in np.linspace(p, N - 1, 8).astype(int):
        _row_check(sh, w, k, v, int(r), int(ctx_tok[r]))
    m.mzc_destroy(c)


def test_3b_scattered_copy_full_size():
    """The 3B-class scattered-copy workload: 32768-token context, 30% of the
    (layer, block) pairs swapped to pinned host and copied back while a
    256-token prompt runs."""
    sc = W.SCENARIOS["3b_scattered_copy"]
    sh, w, c, ctx_tok, prm = _ctx(sc)
    N, P, L = sc["context"], sc["prompt"], sh["n_layers"]
    # reference: the prompt on the intact context (then rolled back)
    ref_logits = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, prm, ref_logits)
    m.mzc_truncate(c, N)
    nblk = N // 16
    sel = synth.permutation(synth.SEED_EVICT, 0, L * nblk)[: int(round(0.3 * L * nblk))]
    sample = sel[:: max(1, sel.size // 64)]
    before = {int(x): m.mzc_read_kv(c, int(x) // nblk, int(x) % nblk, sh) for x in sample}
    m.mzc_evict_blocks(c, sel // nblk, sel % nblk)
    assert m.mzc_query(c, int(sel[0]) // nblk, int(sel[0]) % nblk)[0] == m.MZC_SWAPPED
    m.mzc_restore_async(c)
    logits = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, prm, logits)
    for x, (k0, v0) in before.items():
        k1, v1 = m.mzc_read_kv(c, x // nblk, x % nblk, sh)
        assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    assert np.array_equal(logits, ref_logits)  # copy restore is bit-exact
    _one_row_check(sh, w, c, N + P, N + P - 1, prm[-1], logits)
    m.mzc_destroy(c)
