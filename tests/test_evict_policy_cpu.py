"""The library's eviction policy (mzc_plan_evict_size, mzc_state_evict_size:
Algorithm 1 of Sec. 4.3 behind the paper's evict(size), Sec. 5) against the
oracle's statement of it (oracle/evict_policy.py, pinned by hand-derived
plans), on the CPU: the planned counts for random per-unit times, totals and
requests; and the residency the state-level evict(size) leaves, against the
oracle's placement applied to the oracle's state model."""
import numpy as np
import pytest

import paper_2609_01338_gb300 as m
from oracle import evict_policy as P
from oracle.state_model import StateModel
from synth import workloads as W


def _lib_plan(t, counts, totals, sizes, request):
    p = m.mzc_evict_plan(t[0], t[1], t[2], totals[0], totals[1], counts[2], counts[0], counts[1],
                         sizes[0], sizes[1])
    freed, stage = m.mzc_plan_evict_size(p, request)
    return p.kv_copy, p.kv_rec, p.w_evicted, freed, stage


@pytest.mark.parametrize("seed", range(8))
def test_planner_matches_the_oracle(seed):
    rng = np.random.default_rng(seed)
    for _ in range(200):
        t = (float(rng.uniform(0.1, 20)), float(rng.uniform(0.01, 5)), float(rng.uniform(0.05, 10)))
        kv_total, w_total = int(rng.integers(0, 300)), int(rng.integers(0, 30))
        kv_copy = int(rng.integers(0, kv_total + 1))
        kv_rec = int(rng.integers(0, kv_total - kv_copy + 1))
        w_ev = int(rng.integers(0, w_total + 1))
        sizes = (int(rng.integers(1, 5000)), int(rng.integers(1, 80000)))
        req = int(rng.integers(0, 400000))
        want = P.plan(*t, kv_total, w_total, kv_copy, kv_rec, w_ev, *sizes, req)
        got = _lib_plan(t, (kv_copy, kv_rec, w_ev), (kv_total, w_total), sizes, req)
        assert got == want, (t, kv_total, w_total, kv_copy, kv_rec, w_ev, sizes, req)


def test_planner_rejects_bad_counts():
    S = m.mzc.status_of
    import ctypes
    f, st = ctypes.c_int64(), ctypes.c_int32()
    bad = m.mzc_evict_plan(1.0, 1.0, 1.0, 10, 2, 0, 8, 5, 100, 1000)  # 8 + 5 > 10 units
    assert S("mzc_plan_evict_size", ctypes.byref(bad), 100, ctypes.byref(f), ctypes.byref(st)) == m.MZC_ERR_INVALID
    neg = m.mzc_evict_plan(-1.0, 1.0, 1.0, 10, 2, 0, 0, 0, 100, 1000)
    assert S("mzc_plan_evict_size", ctypes.byref(neg), 100, ctypes.byref(f), ctypes.byref(st)) == m.MZC_ERR_INVALID


SMALL = W.scaled(W.TINY, n_layers=3, max_ctx=640)


def _model_apply(model, n_ctx, L, before, after):
    """The oracle's placement for `after`, reached from `before` with the
    state model's own evictions (COPY of the new front, DROP of the new
    rear range, which may take swapped blocks)."""
    c0, r0, w0 = before
    c1, r1, w1 = after
    nb = -(-n_ctx // 16)
    e0, e1, d0, d1 = nb - r0 - c0, nb - r1 - c1, nb - r0, nb - r1
    cb1 = min(e0, d1)
    if cb1 > e1:
        assert model.evict(0, L, e1 * 16, min(cb1 * 16, n_ctx), 0) == 0
    if d0 > d1:
        assert model.evict(0, L, d1 * 16, min(d0 * 16, n_ctx), 1) == 0


@pytest.mark.parametrize("seed", range(4))
def test_state_evict_size_places_units_backward_out(seed):
    rng = np.random.default_rng(100 + seed)
    L, n_ctx = SMALL["n_layers"], int(rng.integers(200, 641))
    st = m.mzc_state_create(SMALL, pool_blocks=4 * L * 40)
    m.mzc._call("mzc_state_append", st, n_ctx)
    model = StateModel(L, 640)
    assert model.append(n_ctx) == 0
    t = (float(rng.uniform(1, 10)), float(rng.uniform(0.1, 2)), float(rng.uniform(0.2, 5)))
    sizes = (L * 8192, 1_000_000)
    times = m.mzc_evict_plan(*t, 0, 0, 0, 0, 0, *sizes)
    counts = (0, 0, 0)
    kv_total = -(-n_ctx // 16)
    for _ in range(int(rng.integers(1, 6))):
        req = int(rng.integers(1, 30)) * sizes[0]
        want = P.plan(*t, kv_total, L, *counts, *sizes, req)
        freed, stage = m.mzc_state_evict_size(st, times, req)
        assert (freed, stage) == want[3:]
        _model_apply(model, n_ctx, L, counts, want[:3])
        counts = want[:3]
        nb = model.nblk
        got = [[m.mzc_state_query(st, l, b)[0] for b in range(nb)] for l in range(L)]
        assert got == model.st
        # the placement: dropped tail, swapped blocks before it, resident front
        (cb0, cb1), drop, _ = P.layout(n_ctx, L, *counts)
        for l in range(L):
            assert all(x == m.MZC_SWAPPED for x in got[l][cb0:cb1])
            if drop:
                assert all(x == m.MZC_DROPPED for x in got[l][drop[0] // 16: kv_total])
            assert all(x == m.MZC_RESIDENT for x in got[l][:cb0])
        if stage == P.COMP_KV:
            break
    m.mzc._call("mzc_state_destroy", st)


def test_state_evict_size_refuses_other_placements():
    st = m.mzc_state_create(SMALL, pool_blocks=400)
    m.mzc._call("mzc_state_append", st, 320)
    ls = np.array([0], np.int32)
    bs = np.array([3], np.int64)
    m.mzc._call("mzc_state_evict_blocks", st, ls.ctypes.data, bs.ctypes.data, 1, 0)
    times = m.mzc_evict_plan(10.0, 1.0, 3.0, 0, 0, 0, 0, 0, 3 * 8192, 10 ** 6)
    import ctypes
    f, s = ctypes.c_int64(), ctypes.c_int32()
    assert m.mzc.status_of("mzc_state_evict_size", st, ctypes.byref(times), 100, ctypes.byref(f),
                           ctypes.byref(s)) == m.MZC_ERR_STATE
    m.mzc._call("mzc_state_destroy", st)
