"""evict(size) on the GPU (the paper's Sec. 5 interface driving Algorithm 1,
Sec. 4.3): each call's plan, stage and placement against the oracle's
policy, then the restore (copies, weight stream, recompute of the dropped
tail, fused with the prompt) against the oracle's full prefill."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from oracle import evict_policy as P
from synth import workloads as W
from tests.gpu_util import rel_err

pytestmark = pytest.mark.gpu

LOGIT_TOL, KV_TOL = 2e-2, 1e-2

# per-unit times chosen so that the policy goes through KVonly with both
# paths, then KVandW: at 16.384 GB/s a tiny-model KV unit (16 KiB) takes
# 1 us and a weight layer ~90 us; recomputing a unit (16 rows x 2 layers at
# 0.5 us a row, attention at 100 TFLOP/s) ~16 us: q = 5, T = 10
PROFILE = (16.384, 100.0, 300.0, 1024.0, 100.0, 0.0, 100.0, 0.0, 10.0)


@pytest.fixture(scope="module")
def tiny():
    sh = W.TINY
    w = synth.model_weights(sh)
    ctx = synth.tokens(synth.SEED_CONTEXT, 0, 512, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 0, 32, sh["vocab"])
    kv = oracle.KVState(sh, sh["max_ctx"])
    lg = oracle.prefill(sh, w, kv, np.concatenate([ctx, prm]), 0)
    return dict(shape=sh, w=w, ctx=ctx, prm=prm, lg_ref=lg, kv_ref=kv)


def _new(tiny):
    c = m.mzc_create(tiny["shape"], tiny["w"])
    m.mzc_set_policy(c, m.MZC_POLICY_COPY, m.mzc_profile(*PROFILE))
    m.mzc_prefill(c, tiny["ctx"])
    return c


def _oracle_step(plan, request):
    return P.plan(plan.t_copy_w, plan.t_copy_kv, plan.t_rec_kv, plan.kv_total, plan.w_total,
                  plan.kv_copy, plan.kv_rec, plan.w_evicted, plan.kv_bytes, plan.w_bytes, request)


def _check_placement(c, sh, n_ctx, counts):
    (cb0, cb1), drop, (w0, _) = P.layout(n_ctx, sh["n_layers"], *counts)
    nb = -(-n_ctx // 16)
    for l in range(sh["n_layers"]):
        for b in range(nb):
            st = m.mzc_query(c, l, b)[0]
            want = (m.MZC_DROPPED if drop and b >= drop[0] // 16 else
                    m.MZC_SWAPPED if cb0 <= b < cb1 else m.MZC_RESIDENT)
            assert st == want, (l, b, st, want)
    assert m.mzc_stats(c).weights_evicted_layers == sh["n_layers"] - w0
    return drop


def _restore_and_check(tiny, c, drop):
    sh = tiny["shape"]
    m.mzc_restore_async(c)
    if drop:
        m.mzc_recompute_tail(c, drop[0], drop[1] - drop[0])
    lg = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, tiny["prm"], lg)
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    k, v = m.mzc_read_kv_all(c, 544, sh)
    for l in range(sh["n_layers"]):
        assert rel_err(k[l], tiny["kv_ref"].k[l, :544]) < KV_TOL
        assert rel_err(v[l], tiny["kv_ref"].v[l, :544]) < KV_TOL
    st = m.mzc_stats(c)
    assert st.blocks_swapped == 0 and st.blocks_dropped == 0 and st.weights_evicted_layers == 0


def test_evict_size_calls_follow_the_policy_and_restore_exactly(tiny):
    sh = tiny["shape"]
    c = _new(tiny)
    before = m.mzc_read_kv_all(c, 512, sh)
    plan = m.mzc_evict_size_plan(c)
    assert (plan.kv_copy, plan.kv_rec, plan.w_evicted, plan.kv_total, plan.w_total) == (0, 0, 0, 32, 2)
    # q = floor(t_W / t_rec) >= 1 so that KVandW is reached
    assert plan.t_copy_w >= plan.t_rec_kv > plan.t_copy_kv > 0
    stages = []
    for request in (10 * plan.kv_bytes, 9 * plan.kv_bytes + 1, plan.w_bytes):
        want = _oracle_step(plan, request)
        freed, stage = m.mzc_evict_size(c, request)
        assert (freed, stage) == want[3:]
        plan = m.mzc_evict_size_plan(c)
        assert (plan.kv_copy, plan.kv_rec, plan.w_evicted) == want[:3]
        drop = _check_placement(c, sh, 512, want[:3])
        stages.append(stage)
    assert P.KV_ONLY in stages and P.KV_AND_W in stages
    assert plan.kv_copy > 0 and plan.kv_rec > 0 and plan.w_evicted > 0
    # copied blocks come back bit for bit
    (cb0, cb1), _, _ = P.layout(512, sh["n_layers"], plan.kv_copy, plan.kv_rec, plan.w_evicted)
    _restore_and_check(tiny, c, drop)
    after = m.mzc_read_kv_all(c, 512, sh)
    for kv0, kv1 in zip(before, after):
        assert np.array_equal(kv0[:, :cb1 * 16], kv1[:, :cb1 * 16])  # resident + copied
    m.mzc_destroy(c)


def test_evict_size_to_the_last_stage(tiny):
    sh = tiny["shape"]
    c = _new(tiny)
    plan = m.mzc_evict_size_plan(c)
    want = _oracle_step(plan, 1 << 40)
    freed, stage = m.mzc_evict_size(c, 1 << 40)
    assert (freed, stage) == want[3:] and stage == P.COMP_KV
    assert want[0] + want[1] == 32 and want[2] == 2   # every unit evicted
    drop = _check_placement(c, sh, 512, want[:3])
    # nothing more to free
    assert m.mzc_evict_size(c, 1) == (0, P.COMP_KV)
    _restore_and_check(tiny, c, drop)
    m.mzc_destroy(c)
