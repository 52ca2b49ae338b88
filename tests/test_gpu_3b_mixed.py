"""The 3B-class mixed restore against the full CPU oracle, at 3B widths
(d 3072, 24 query / 8 KV heads of 128, FFN 8192, bf16 KV, vocab 128256) with 4
layers and a 4096-token context, in the proportions of the 3B mixed workload
(32768-token context: last 8 of 28 layers' weights streamed, tail from 16384
dropped and recomputed, 20% of the rest copied, 512-token prompt):

  - the last layer's weights evicted and streamed back per layer;
  - the tail [2048, 4096) dropped and recomputed, fused with the prompt;
  - 20% of the (layer, block) pairs below position 2048 swapped to pinned host
    and copied back while the prefill runs;
  - a 64-token prompt.

This covers, in one pass against the oracle's full prefill of context and
prompt, the bf16-KV rotary write, the head-dim-128 tensor-core attention over
many row tiles whose keys partly arrive by copy, the weight stream and the
LM head at the full vocabulary.  Bars: logits max-abs <= 2e-2, recomputed and
prompt K/V max|d|/max|ref| <= 1e-2 per layer, copied blocks bit-exact."""
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

N_CTX, N_PROMPT, DROP_FROM, COPY_FRAC = 4096, 64, 2048, 0.20
SH = W.scaled(W.THREE_B, n_layers=4, max_ctx=N_CTX + 128)


def test_3b_widths_mixed_restore_matches_the_oracle():
    sh, L = SH, SH["n_layers"]
    w = synth.model_weights(sh)
    ctx_tok = synth.tokens(synth.SEED_CONTEXT, 7, N_CTX, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 7, N_PROMPT, sh["vocab"])

    c = m.mzc_create(sh, w)
    m.mzc_prefill(c, ctx_tok)
    eligible = DROP_FROM // 16
    sel = synth.permutation(synth.SEED_EVICT, 7, L * eligible)[: int(round(COPY_FRAC * L * eligible))]
    before = {int(x): m.mzc_read_kv(c, int(x) // eligible, int(x) % eligible, sh) for x in sel}
    k_pre, v_pre = m.mzc_read_kv_all(c, DROP_FROM, sh)

    m.mzc_evict_weights(c, L - 1, L)
    m.mzc_evict_blocks(c, sel // eligible, sel % eligible)
    m.mzc_evict(c, 0, L, DROP_FROM, N_CTX, m.MZC_DROP)
    x = int(sel[0])
    assert m.mzc_query(c, x // eligible, x % eligible)[0] == m.MZC_SWAPPED
    assert m.mzc_query(c, 0, DROP_FROM // 16)[0] == m.MZC_DROPPED
    assert m.mzc_stats(c).weights_evicted_layers == 1

    m.mzc_restore_async(c)
    m.mzc_recompute_tail(c, DROP_FROM, N_CTX - DROP_FROM)
    logits = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, prm, logits)
    st = m.mzc_stats(c)
    assert st.recompute_rows_last == N_CTX - DROP_FROM and st.rows_last == N_CTX - DROP_FROM + N_PROMPT
    assert st.weights_evicted_layers == 0 and st.blocks_swapped == 0 and st.blocks_dropped == 0

    # copy restores are bit-exact, and the whole resident prefix is untouched
    for x, (k0, v0) in before.items():
        k1, v1 = m.mzc_read_kv(c, x // eligible, x % eligible, sh)
        assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
    k, v = m.mzc_read_kv_all(c, N_CTX + N_PROMPT, sh)
    assert np.array_equal(k[:, :DROP_FROM], k_pre) and np.array_equal(v[:, :DROP_FROM], v_pre)
    m.mzc_destroy(c)

    # the oracle: one full prefill of context || prompt from scratch
    kv_ref = oracle.KVState(sh, N_CTX + N_PROMPT)
    lg_ref = oracle.prefill(sh, w, kv_ref, np.concatenate([ctx_tok, prm]), 0)
    assert np.max(np.abs(logits - lg_ref)) < LOGIT_TOL
    for l in range(L):
        for a, b in ((0, DROP_FROM), (DROP_FROM, N_CTX), (N_CTX, N_CTX + N_PROMPT)):
            assert rel_err(k[l, a:b], kv_ref.k[l, a:b]) < KV_TOL, (l, a)
            assert rel_err(v[l, a:b], kv_ref.v[l, a:b]) < KV_TOL, (l, a)
