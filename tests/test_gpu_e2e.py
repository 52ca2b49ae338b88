"""End-to-end parity on the GPU through the C ABI (mzc_create / evict /
restore_async / recompute_tail / prefill) against the CPU oracle, plus the
exact invariants of the restore paths (a copy restore is bit-exact)."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
from tests.gpu_util import rel_err

pytestmark = pytest.mark.gpu

LOGIT_TOL = 2e-2   # max-abs on logits
KV_TOL = 1e-2      # max|d| / max|ref| per layer on recomputed K/V


def _oracle_full(shape, weights, toks, max_ctx):
    kv = oracle.KVState(shape, max_ctx)
    lg = oracle.prefill(shape, weights, kv, toks, 0)
    return lg, kv


@pytest.fixture(scope="module")
def tiny():
    sh = W.TINY
    w = synth.model_weights(sh)
    ctx = synth.tokens(synth.SEED_CONTEXT, 0, 512, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 0, 32, sh["vocab"])
    lg_ref, kv_ref = _oracle_full(sh, w, np.concatenate([ctx, prm]), sh["max_ctx"])
    lg_ctx, _ = _oracle_full(sh, w, ctx, sh["max_ctx"])
    return dict(shape=sh, w=w, ctx=ctx, prm=prm, lg_ref=lg_ref, kv_ref=kv_ref, lg_ctx=lg_ctx)


def _new(case, **kw):
    return m.mzc_create(case["shape"], case["w"], **kw)


def _logits(case, c, toks):
    out = np.empty(case["shape"]["vocab"], np.float32)
    m.mzc_prefill(c, toks, out)
    return out


def _check_kv(case, c, n, tol=KV_TOL):
    k, v = m.mzc_read_kv_all(c, n, case["shape"])
    for l in range(case["shape"]["n_layers"]):
        assert rel_err(k[l], case["kv_ref"].k[l, :n]) < tol
        assert rel_err(v[l], case["kv_ref"].v[l, :n]) < tol


def test_context_prefill_matches_oracle(tiny):
    c = _new(tiny)
    lg = _logits(tiny, c, tiny["ctx"])
    assert np.max(np.abs(lg - tiny["lg_ctx"])) < LOGIT_TOL
    _check_kv(tiny, c, 512)
    m.mzc_destroy(c)


def test_recompute_tail_then_prompt(tiny):
    """The tiny scenario: 512-token context, last 256 tokens dropped
    (backward-out), recomputed fused with a 32-token prompt."""
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_DROP)
    assert m.mzc_query(c, 0, 20)[0] == m.MZC_DROPPED
    m.mzc_restore_async(c)
    m.mzc_recompute_tail(c, 256, 256)
    lg = _logits(tiny, c, tiny["prm"])
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    _check_kv(tiny, c, 544)
    st = m.mzc_stats(c)
    assert st.recompute_rows_last == 256 and st.rows_last == 288
    m.mzc_destroy(c)


def _baseline_logits(tiny, **kw):
    c = _new(tiny, **kw)
    m.mzc_prefill(c, tiny["ctx"])
    lg = _logits(tiny, c, tiny["prm"])
    m.mzc_destroy(c)
    return lg


def test_copy_restore_is_bit_exact(tiny):
    base = _baseline_logits(tiny)
    assert np.max(np.abs(base - tiny["lg_ref"])) < LOGIT_TOL
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    before = {(l, b): m.mzc_read_kv(c, l, b, tiny["shape"]) for l in range(2) for b in range(32)}
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_COPY)
    assert m.mzc_query(c, 1, 31)[0] == m.MZC_SWAPPED
    m.mzc_restore_async(c)
    lg = _logits(tiny, c, tiny["prm"])
    assert np.array_equal(lg, base)
    for (l, b), (k0, v0) in before.items():
        k1, v1 = m.mzc_read_kv(c, l, b, tiny["shape"])
        assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    m.mzc_destroy(c)


def test_scattered_copy_restore_bit_exact(tiny):
    base = _baseline_logits(tiny)
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    perm = synth.permutation(synth.SEED_EVICT, 0, 2 * 32)[: int(0.3 * 64)]
    m.mzc_evict_blocks(c, perm // 32, perm % 32)
    m.mzc_restore_async(c)
    lg = _logits(tiny, c, tiny["prm"])
    assert np.array_equal(lg, base)
    m.mzc_destroy(c)


def test_hybrid_copy_plus_recompute(tiny):
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    m.mzc_evict(c, 0, 2, 256, 384, m.MZC_DROP)
    m.mzc_evict(c, 0, 2, 384, 512, m.MZC_COPY)
    m.mzc_restore_async(c)
    m.mzc_recompute_tail(c, 256, 128)
    lg = _logits(tiny, c, tiny["prm"])
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    _check_kv(tiny, c, 544)
    m.mzc_destroy(c)


def test_weight_eviction_and_no_overlap_are_bit_exact(tiny):
    base = _baseline_logits(tiny)
    for overlap in (1, 0):
        c = _new(tiny, overlap=overlap)
        m.mzc_prefill(c, tiny["ctx"])
        m.mzc_evict_weights(c, 1, 2)
        m.mzc_evict(c, 0, 2, 100, 512, m.MZC_COPY)
        m.mzc_restore_async(c)
        lg = _logits(tiny, c, tiny["prm"])
        assert np.array_equal(lg, base)
        assert m.mzc_stats(c).weights_evicted_layers == 0
        m.mzc_destroy(c)


def test_repeat_with_truncate_is_deterministic(tiny):
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    outs = []
    for _ in range(3):
        m.mzc_evict(c, 0, 2, 256, 512, m.MZC_DROP)
        m.mzc_recompute_tail(c, 256, 256)
        outs.append(_logits(tiny, c, tiny["prm"]))
        m.mzc_truncate(c, 512)
    assert all(np.array_equal(outs[0], o) for o in outs[1:])
    m.mzc_destroy(c)


def test_auto_policies_match(tiny):
    prof = m.mzc_profile(200.0, 110.0, 260.0, 700.0, 800.0, 2000.0, 600.0, 150.0, 15.0)
    res = {}
    for pol in (m.MZC_POLICY_COPY, m.MZC_POLICY_RECOMPUTE, m.MZC_POLICY_HYBRID):
        c = _new(tiny)
        m.mzc_set_policy(c, pol, prof)
        m.mzc_prefill(c, tiny["ctx"])
        m.mzc_evict(c, 0, 2, 256, 512, m.MZC_AUTO)
        st = m.mzc_stats(c)
        m.mzc_restore_async(c)
        if st.blocks_dropped:
            n_drop = st.blocks_dropped // 2 * 16
            m.mzc_recompute_tail(c, 256, n_drop)
        res[pol] = _logits(tiny, c, tiny["prm"])
        m.mzc_destroy(c)
        assert np.max(np.abs(res[pol] - tiny["lg_ref"])) < LOGIT_TOL


def test_error_paths(tiny):
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    S = m.mzc.status_of
    assert S("mzc_evict", c, 0, 2, 256, 600, m.MZC_COPY) == m.MZC_ERR_RANGE
    assert S("mzc_evict", c, 0, 1, 256, 512, m.MZC_DROP) == m.MZC_ERR_INVALID
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_DROP)
    assert S("mzc_evict", c, 0, 2, 256, 512, m.MZC_DROP) == m.MZC_ERR_STATE
    toks = np.array(tiny["prm"], np.int32)
    assert S("mzc_prefill", c, toks.ctypes.data, toks.size, None) == m.MZC_ERR_STATE
    assert S("mzc_recompute_tail", c, 256, 100) == m.MZC_ERR_RANGE
    bad = np.array([5, 2000], np.int32)
    m.mzc_recompute_tail(c, 256, 256)
    assert S("mzc_prefill", c, bad.ctypes.data, 2, None) == m.MZC_ERR_INVALID
    m.mzc_sync(c)  # runs the pending recompute alone
    assert m.mzc_stats(c).blocks_dropped == 0
    lg = _logits(tiny, c, tiny["prm"])
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    m.mzc_destroy(c)


# ---- a wider case: several GEMM tiles, GQA 4, ragged tail ------------------

MID = W.scaled(W.ONE_B, n_layers=2, vocab=4096, max_ctx=1024)


@pytest.fixture(scope="module")
def mid():
    sh = MID
    w = synth.model_weights(sh)
    ctx = synth.tokens(synth.SEED_CONTEXT, 1, 600, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 1, 37, sh["vocab"])
    lg_ref, kv_ref = _oracle_full(sh, w, np.concatenate([ctx, prm]), sh["max_ctx"])
    return dict(shape=sh, w=w, ctx=ctx, prm=prm, lg_ref=lg_ref, kv_ref=kv_ref)


def test_mid_hybrid_restore(mid):
    c = _new(mid)
    m.mzc_prefill(c, mid["ctx"])
    m.mzc_evict(c, 0, 2, 200, 424, m.MZC_DROP)      # rounds out to [192, 432)
    m.mzc_evict(c, 0, 2, 432, 600, m.MZC_COPY)
    perm = synth.permutation(synth.SEED_EVICT, 1, 2 * 12)[:7]
    m.mzc_evict_blocks(c, perm // 12, perm % 12)
    m.mzc_restore_async(c)
    m.mzc_recompute_tail(c, 192, 240)
    lg = _logits(mid, c, mid["prm"])
    assert np.max(np.abs(lg - mid["lg_ref"])) < LOGIT_TOL
    _check_kv(mid, c, 637)
    m.mzc_destroy(c)


def test_row_sets_beyond_max_rows_run_in_causal_chunks(tiny):
    """max_rows=100: the 512-token context and the 288-row recompute + prompt
    set both run in chunks of 100 rows; logits and KV still match the oracle."""
    c = _new(tiny, max_rows=100)
    m.mzc_prefill(c, tiny["ctx"])
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_DROP)
    m.mzc_recompute_tail(c, 256, 256)
    lg = _logits(tiny, c, tiny["prm"])
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    _check_kv(tiny, c, 544)
    assert m.mzc_stats(c).rows_last == 288
    m.mzc_destroy(c)


def test_q8_swap_restore_decodes_the_oracle_codes(tiny):
    """Compressed swap (MZC_CODEC_Q8): the restored blocks hold exactly the
    oracle's decode of its encoding of the pre-eviction blocks; a second swap
    cycle restores the same values (idempotence, Sec. 6.5); the prompt's
    logits match the oracle's forward over the restored KV; the link moves
    about 0.56 of the raw bytes."""
    sh = tiny["shape"]
    L = sh["n_layers"]
    e = 2 * sh["n_kv_heads"] * 16 * sh["head_dim"]
    c = _new(tiny, swap_codec=m.MZC_CODEC_Q8)
    m.mzc_prefill(c, tiny["ctx"])
    blocks = [(l, b) for l in range(L) for b in range(16, 32)]  # positions [256, 512)

    def read():
        return np.stack([np.concatenate(m.mzc_read_kv(c, l, b, sh)) for l, b in blocks])

    want = oracle.q8_decode_blocks(oracle.q8_encode_blocks(read()), e, sh["kv_dtype"])
    for cycle in range(2):
        m.mzc_evict(c, 0, L, 256, 512, m.MZC_COPY)
        assert m.mzc_query(c, 1, 20)[0] == m.MZC_SWAPPED
        m.mzc_restore_async(c)
        m.mzc_sync(c)
        assert np.array_equal(read(), want), cycle
        if cycle == 0:
            assert m.mzc_stats(c).bytes_h2d_last == len(blocks) * m.mzc_q8_block_bytes(
                sh["n_kv_heads"], sh["head_dim"])
    k, v = m.mzc_read_kv_all(c, 512, sh)
    kv = oracle.KVState(sh, sh["max_ctx"])
    kv.k[:, :512], kv.v[:, :512] = k, v
    ref = oracle.forward(sh, tiny["w"], kv, tiny["prm"], np.arange(512, 544))
    lg = _logits(tiny, c, tiny["prm"])
    assert np.max(np.abs(lg - ref)) < LOGIT_TOL
    m.mzc_destroy(c)


def test_q8_swap_overlapped_with_prompt_matches_sync_restore(tiny):
    """The decode stream feeds the zero-wait prefill: restoring while the
    prompt runs gives the same logits as restoring first (bit-exact)."""
    outs = []
    for overlap in (1, 0):
        c = _new(tiny, swap_codec=m.MZC_CODEC_Q8, overlap=overlap)
        m.mzc_prefill(c, tiny["ctx"])
        m.mzc_evict(c, 0, tiny["shape"]["n_layers"], 100, 512, m.MZC_COPY)
        m.mzc_restore_async(c)
        outs.append(_logits(tiny, c, tiny["prm"]))
        m.mzc_destroy(c)
    assert np.array_equal(outs[0], outs[1])


def test_q8_copies_with_recomputed_tail(tiny):
    """8-bit copies of [256, 384) restored while the dropped tail [384, 512)
    is recomputed and the prompt runs: the copies hold the oracle's decode of
    its encoding, the logits equal the restore-first run bit for bit and the
    oracle's forward of the tail and the prompt over the decoded copies; a
    sync with copies pending and nothing to recompute decodes them too."""
    sh, w, L = tiny["shape"], tiny["w"], tiny["shape"]["n_layers"]
    e = 2 * sh["n_kv_heads"] * 16 * sh["head_dim"]
    blocks = [(l, b) for l in range(L) for b in range(16, 24)]  # positions [256, 384)

    def read(c):
        return np.stack([np.concatenate(m.mzc_read_kv(c, l, b, sh)) for l, b in blocks])

    outs = []
    for overlap in (1, 0):
        c = _new(tiny, swap_codec=m.MZC_CODEC_Q8, overlap=overlap)
        m.mzc_prefill(c, tiny["ctx"])
        want = oracle.q8_decode_blocks(oracle.q8_encode_blocks(read(c)), e, sh["kv_dtype"])
        m.mzc_evict(c, 0, L, 384, 512, m.MZC_DROP)
        m.mzc_evict(c, 0, L, 256, 384, m.MZC_COPY)
        m.mzc_restore_async(c)
        m.mzc_recompute_tail(c, 384, 128)
        outs.append(_logits(tiny, c, tiny["prm"]))
        assert np.array_equal(read(c), want)
        if overlap:
            k, v = m.mzc_read_kv_all(c, 384, sh)
            kv = oracle.KVState(sh, sh["max_ctx"])
            kv.k[:, :384], kv.v[:, :384] = k, v
            toks = np.concatenate([tiny["ctx"][384:512], tiny["prm"]])
            ref = oracle.forward(sh, w, kv, toks, np.arange(384, 544))
        m.mzc_destroy(c)
    assert np.array_equal(outs[0], outs[1])
    assert np.max(np.abs(outs[0] - ref)) < LOGIT_TOL
    # copies pending at a sync with nothing to recompute: decoded by the sync
    c = _new(tiny, swap_codec=m.MZC_CODEC_Q8)
    m.mzc_prefill(c, tiny["ctx"])
    want = oracle.q8_decode_blocks(oracle.q8_encode_blocks(read(c)), e, sh["kv_dtype"])
    m.mzc_evict(c, 0, L, 0, 512, m.MZC_COPY)
    m.mzc_restore_async(c)
    m.mzc_sync(c)
    assert np.array_equal(read(c), want)
    m.mzc_destroy(c)


def test_decode_steps_match_oracle(tiny):
    """Decode after the first token: single-token steps (the few-row GEMV
    projections, one-row attention) match the oracle's forward of the same
    row step after step, across a newly allocated KV block."""
    sh, w = tiny["shape"], tiny["w"]
    c = _new(tiny)
    m.mzc_prefill(c, tiny["ctx"])
    kv = oracle.KVState(sh, sh["max_ctx"])
    lg_ref = oracle.prefill(sh, w, kv, tiny["ctx"], 0)
    tok = int(np.argmax(lg_ref))
    for step in range(20):
        pos = len(tiny["ctx"]) + step
        lg = _logits(tiny, c, np.array([tok], np.int32))
        lg_ref = oracle.forward(sh, w, kv, [tok], [pos])
        assert np.max(np.abs(lg - lg_ref)) < LOGIT_TOL, step
        tok = int(np.argmax(lg_ref))
    assert m.mzc_stats(c).context_tokens == len(tiny["ctx"]) + 20
    m.mzc_destroy(c)


_PDL_SCRIPT = r"""
import sys
import numpy as np
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
sh = W.TINY
w = synth.model_weights(sh)
ctx = synth.tokens(synth.SEED_CONTEXT, 0, 512, sh["vocab"])
prm = synth.tokens(synth.SEED_PROMPT, 0, 32, sh["vocab"])
c = m.mzc_create(sh, w)
outs = []
for toks in (ctx, prm, prm[:1], prm[1:2], prm[2:4]):  # 512, 32, then 1, 1 and 2 rows
    lg = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, toks, lg)
    outs.append(lg)
m.mzc_destroy(c)
np.save(sys.argv[1], np.stack(outs))
"""


def test_programmatic_dependent_launch_changes_no_bit(tmp_path):
    """The same prefill and decode steps with programmatic dependent launch
    off and on (a fresh process each: the switch is read at load) give
    bit-identical logits, so no kernel touches memory before its wait."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    got = []
    for v in ("0", "1"):
        out = tmp_path / f"pdl{v}.npy"
        env = dict(os.environ, MZC_PDL=v, PYTHONPATH=root + os.pathsep + os.environ.get("PYTHONPATH", ""))
        subprocess.run([sys.executable, "-c", _PDL_SCRIPT, str(out)], cwd=root, env=env, check=True,
                       timeout=600)
        got.append(np.load(out))
    assert got[0].shape == (5, W.TINY["vocab"])
    assert np.array_equal(got[0], got[1])
