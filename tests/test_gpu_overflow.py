"""fp16 range checks on the GPU.  The projections read fp16 activations and
K/V are held fp16-encoded, so a value of magnitude 65520 or more would be
stored as infinity; the kernels that store such values record
MZC_ERR_OVERFLOW in the status word, the call fails with that status, and the
context stays usable.  In-range inputs (every other parity test) record
nothing."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
from tests.gpu_util import bf16_dev, f16_bits, f32_dev, i32_dev

pytestmark = pytest.mark.gpu


def _planted_weights(sh):
    """Layer 0's query weights set to +-60000 with seeded random signs (inside
    fp16's range, so the weights are accepted): each q output is 60000 times a
    signed sum of 256 normalised inputs, about N(0, 16) * 60000, so nearly
    every one of the 256 outputs of a row is far beyond 65504."""
    w = synth.model_weights(sh)
    signs = np.where(np.random.default_rng(11).random(w["layers"][0]["wq"].shape) < 0.5, -1.0, 1.0)
    w["layers"][0]["wq"] = oracle.to_bf16_bits((signs * 60000.0).astype(np.float32))
    return w


@pytest.mark.parametrize("rows", [512, 32, 1])  # persistent GEMM, split-K GEMM, GEMV
def test_projection_overflow_is_reported(rows):
    sh = W.TINY
    c = m.mzc_create(sh, _planted_weights(sh))
    toks = synth.tokens(synth.SEED_CONTEXT, 3, rows, sh["vocab"])
    st = m.mzc.status_of("mzc_prefill", c, toks.ctypes.data, rows, None)
    assert st == m.MZC_ERR_OVERFLOW
    assert "overflow" in m.mzc_last_error(c)
    m.mzc_destroy(c)
    # the context (and a ctx with ordinary weights) still works
    c = m.mzc_create(sh, synth.model_weights(sh))
    lg = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, toks, lg)
    assert np.all(np.isfinite(lg))
    m.mzc_destroy(c)


def test_rotary_overflow_of_in_range_inputs_is_reported():
    """Two fp16 inputs of 60000 rotated at angle 1 rad give
    60000 * (cos 1 + sin 1) = 82903 > 65504 in the second half of the pair."""
    import torch
    hq, hkv, hd, n = 4, 2, 64, 3
    qkv = np.zeros((n, (hq + 2 * hkv) * hd), np.float32)
    qkv[1, hq * hd + 0] = 60000.0             # k head 0, pair (0, 32), position 1
    qkv[1, hq * hd + hd // 2] = 60000.0
    pos = np.array([0, 1, 2], np.int32)
    n_logical, pool_blocks = 1, 2
    cos_t, sin_t = oracle.rope_table(16, hd, 500000.0)
    pool = torch.zeros(pool_blocks * 2 * hkv * 16 * hd, dtype=torch.int16, device="cuda")
    q_out = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for kvd in (m.MZC_KV_BF16, m.MZC_KV_FP16):
        status.zero_()
        m.mzc_k_rope_kv_write(bf16_dev(f16_bits(qkv)), i32_dev(pos), n, hq, hkv, hd, f32_dev(cos_t),
                              f32_dev(sin_t), i32_dev(np.array([1], np.int32)), n_logical, pool,
                              pool_blocks, kvd, q_out, status)
        torch.cuda.synchronize()
        assert int(status.item()) == m.MZC_ERR_OVERFLOW, kvd
    # the same inputs at half the size stay in range: nothing recorded
    status.zero_()
    m.mzc_k_rope_kv_write(bf16_dev(f16_bits(qkv / 2)), i32_dev(pos), n, hq, hkv, hd, f32_dev(cos_t),
                          f32_dev(sin_t), i32_dev(np.array([1], np.int32)), n_logical, pool,
                          pool_blocks, m.MZC_KV_FP16, q_out, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
