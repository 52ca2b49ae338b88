"""Pins of the oracle's eviction policy (oracle/evict_policy.py, Algorithm 1 of
Sec. 4.3 with the GB300 reading stated there).  Every expected plan below is
worked out by hand from the algorithm's steps, not produced by the code:

Case A: t_W = 10, t_copy = 1, t_rec = 3, 40 KV units, 4 weight layers,
100 bytes per KV unit, 1000 per layer.  q = floor(10 / 3) = 3, T = 4 * 3 = 12.
  KVonly unit by unit (recompute time with the unit vs link time with it):
    1: 3 vs 1 link   2: 3 vs 2 link   3: 3 vs 3 link (tie)   4: 3 vs 4 recompute
    5: 6 vs 4 link   6: 6 vs 5 link   7: 6 vs 6 link (tie)   8: 6 vs 7 recompute
  so every 4 units: 3 to the link, 1 to recompute (the inverse of 1 : 3).
  28 units bring N_KV to T = 12: 21 copied, 7 recomputed.  Each KVandW step
  then drops a layer and recomputes 3 units (1300 bytes); after 4 steps
  N_KV = 40 - 21 - 19 = 0 and no layer is left: both run out together.
Case B: the same times, 5 KV units (N_KV <= T from the start): KVandW takes
  3 units, then the last 2, then Wonly takes the other 2 layers.
Case C: t_W = 2 < t_rec = 3: q = 0, T = 0, all KV in KVonly, then Wonly.
Case D: two layers already on the link (20 s of link time): KV units go to
  recompute while the recompute path stays below it.
A plausible mistake fails one of these: ties to recompute (A), ceil for q
(A's transition), the link time without the weights (D), KVandW taking KV
from the link (A), no stop when nothing is left (B, C)."""
from oracle.evict_policy import COMP_KV, KV_AND_W, KV_ONLY, W_ONLY, layout, plan

A = dict(t_copy_w=10.0, t_copy_kv=1.0, t_rec_kv=3.0, kv_total=40, w_total=4, kv_bytes=100,
         w_bytes=1000)


def _plan(case, counts, request):
    c = dict(case)
    return plan(c["t_copy_w"], c["t_copy_kv"], c["t_rec_kv"], c["kv_total"], c["w_total"],
                *counts, c["kv_bytes"], c["w_bytes"], request)


def test_kvonly_splits_in_inverse_proportion_with_ties_to_the_link():
    assert _plan(A, (0, 0, 0), 300) == (3, 0, 0, 300, KV_ONLY)
    assert _plan(A, (0, 0, 0), 400) == (3, 1, 0, 400, KV_ONLY)
    assert _plan(A, (0, 0, 0), 800) == (6, 2, 0, 800, KV_ONLY)
    assert _plan(A, (0, 0, 0), 2800) == (21, 7, 0, 2800, KV_ONLY)
    # a request smaller than one unit still evicts one whole unit
    assert _plan(A, (0, 0, 0), 1) == (1, 0, 0, 100, KV_ONLY)
    # calls add up: 800 then 2000 more is the same as 2800 at once
    c, r, w, f, _ = _plan(A, (0, 0, 0), 800)
    assert _plan(A, (c, r, w), 2000) == (21, 7, 0, 2000, KV_ONLY)


def test_kvandw_drops_a_layer_and_recomputes_q_units_per_step():
    assert _plan(A, (21, 7, 0), 1300) == (21, 10, 1, 1300, KV_AND_W)
    assert _plan(A, (21, 7, 0), 1301) == (21, 13, 2, 2600, KV_AND_W)
    assert _plan(A, (21, 7, 0), 5200) == (21, 19, 4, 5200, KV_AND_W)
    # everything evicted: CompKV frees nothing more on the device
    assert _plan(A, (21, 19, 4), 1) == (21, 19, 4, 0, COMP_KV)


def test_whole_run_from_resident_to_empty():
    assert _plan(A, (0, 0, 0), 10 ** 9) == (21, 19, 4, 2800 + 4 * 1300, COMP_KV)


def test_few_kv_units_go_kvandw_then_wonly():
    B = dict(A, kv_total=5)
    assert _plan(B, (0, 0, 0), 1300) == (0, 3, 1, 1300, KV_AND_W)
    assert _plan(B, (0, 3, 1), 1) == (0, 5, 2, 1200, KV_AND_W)
    assert _plan(B, (0, 5, 2), 1) == (0, 5, 3, 1000, W_ONLY)
    assert _plan(B, (0, 0, 0), 10 ** 9) == (0, 5, 4, 4500, COMP_KV)


def test_recompute_slower_than_a_weight_layer_has_no_threshold():
    C = dict(A, t_copy_w=2.0, kv_total=6, w_total=2)
    assert _plan(C, (0, 0, 0), 600) == (5, 1, 0, 600, KV_ONLY)
    assert _plan(C, (0, 0, 0), 10 ** 9) == (5, 1, 2, 2600, COMP_KV)


def test_weights_already_on_the_link_push_kv_to_recompute():
    assert _plan(A, (0, 0, 2), 200) == (0, 2, 2, 200, KV_ONLY)
    # units 1-6 recompute (3 .. 18 < 21), the 7th ties (21 = 21) and goes to the
    # link, the 8th recomputes (21 < 22)
    assert _plan(A, (0, 0, 2), 800) == (1, 7, 2, 800, KV_ONLY)


def test_layout_backward_out():
    # 600 positions = 38 blocks; recompute the last 2, copy the 6 before, weights of layer 3
    copy_blocks, drop, weights = layout(600, 4, 6, 2, 1)
    assert copy_blocks == (30, 36)
    assert drop == (576, 600)
    assert weights == (3, 4)
    assert layout(600, 4, 3, 0, 0)[1] is None
