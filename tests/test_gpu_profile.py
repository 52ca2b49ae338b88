"""The per-unit profile (the paper's one-time offline profiling, Sec. 4.3)
measured on a ctx that holds a live context must leave that context as it
was: the resident K/V bytes, the residency and the next prompt's logits are
bit-identical to a ctx that was never profiled."""
import numpy as np
import pytest

import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W

pytestmark = pytest.mark.gpu

# 2048-token context: long enough that the attention part of the profile runs
# too (it times recompute-like and prompt-like rows over the resident blocks)
SH = W.scaled(W.TINY, max_ctx=4096)
N_CTX, N_PROMPT = 2048, 24


def _ctx_and_prompt():
    w = synth.model_weights(SH)
    ctx = synth.tokens(synth.SEED_CONTEXT, 5, N_CTX, SH["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 5, N_PROMPT, SH["vocab"])
    return w, ctx, prm


def test_profile_measure_leaves_the_live_state_unchanged():
    w, ctx_tok, prm = _ctx_and_prompt()
    # reference: the same context and prompt on a ctx that is never profiled
    ref = m.mzc_create(SH, w)
    m.mzc_prefill(ref, ctx_tok)
    lg_ref = np.empty(SH["vocab"], np.float32)
    m.mzc_prefill(ref, prm, lg_ref)
    m.mzc_destroy(ref)

    c = m.mzc_create(SH, w)
    m.mzc_prefill(c, ctx_tok)
    k0, v0 = m.mzc_read_kv_all(c, N_CTX, SH)
    st0 = [[m.mzc_query(c, l, b) for b in range(N_CTX // 16)] for l in range(SH["n_layers"])]
    free0 = m.mzc_stats(c).pool_free_blocks
    prof = m.mzc_profile_measure(c)
    assert prof.h2d_gbs > 1.0
    assert prof.gemm_us_128 > 0 and prof.gemm_us_2048 > 0
    assert prof.attn_tflops > 0 and prof.attn_prompt_tflops > 0
    k1, v1 = m.mzc_read_kv_all(c, N_CTX, SH)
    assert np.array_equal(k0.view(np.uint32), k1.view(np.uint32))
    assert np.array_equal(v0.view(np.uint32), v1.view(np.uint32))
    st1 = [[m.mzc_query(c, l, b) for b in range(N_CTX // 16)] for l in range(SH["n_layers"])]
    assert st0 == st1
    assert m.mzc_stats(c).pool_free_blocks == free0
    lg = np.empty(SH["vocab"], np.float32)
    m.mzc_prefill(c, prm, lg)
    assert np.array_equal(lg, lg_ref)
    m.mzc_destroy(c)


def test_profile_measure_refuses_while_work_is_pending():
    w, ctx_tok, prm = _ctx_and_prompt()
    c = m.mzc_create(SH, w)
    m.mzc_prefill(c, ctx_tok)
    m.mzc_evict(c, 0, SH["n_layers"], 1024, N_CTX, m.MZC_DROP)
    m.mzc_recompute_tail(c, 1024, N_CTX - 1024)
    S = m.mzc.status_of
    out = m.mzc_profile()
    import ctypes
    assert S("mzc_profile_measure", c, ctypes.byref(out)) == m.MZC_ERR_STATE
    m.mzc_sync(c)                                  # runs the recompute
    m.mzc_evict(c, 0, SH["n_layers"], 0, 512, m.MZC_COPY)
    m.mzc_restore_async(c)
    assert S("mzc_profile_measure", c, ctypes.byref(out)) == m.MZC_ERR_STATE
    m.mzc_sync(c)
    assert S("mzc_profile_measure", c, ctypes.byref(out)) == m.MZC_OK
    m.mzc_destroy(c)
