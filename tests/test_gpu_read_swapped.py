"""Reading swapped blocks in place (option read_swapped; the paper's shared
buffers, Sec. 4.2, where the GPU computes on restored units without a copy):
a prefill issued without mzc_restore_async fetches the SWAPPED blocks from
the pinned store over the host link with plain loads, inside the attention
kernels.  The bytes are the evicted bytes, so the logits equal a run that
never evicted, bit for bit: the tensor-core prompt path and the decode path,
at head dims 64 and 128, with scattered and tail evictions; the blocks stay
swapped until a restore brings them back."""
import numpy as np
import pytest

import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W

pytestmark = pytest.mark.gpu

SHAPES = {
    "hd64": W.TINY,
    # head dim 128, bf16 KV, GQA 4
    "hd128": W.shape(2, 512, 8, 2, 128, 1024, 2048, W.KV_BF16, max_ctx=1024),
}


def _run(sh, w, ctx_tok, steps, evict=None, read_swapped=0, restore_after=None):
    c = m.mzc_create(sh, w, read_swapped=read_swapped)
    m.mzc_prefill(c, ctx_tok)
    if evict:
        evict(c)
    outs, swapped = [], []
    for i, toks in enumerate(steps):
        if restore_after is not None and i == restore_after:
            m.mzc_restore_async(c)
        lg = np.empty(sh["vocab"], np.float32)
        m.mzc_prefill(c, toks, lg)
        outs.append(lg)
        swapped.append(m.mzc_stats(c).blocks_swapped)
    m.mzc_destroy(c)
    return outs, swapped


@pytest.mark.parametrize("name", ["hd64", "hd128"])
def test_in_place_reads_equal_the_unevicted_run(name):
    sh = SHAPES[name]
    w = synth.model_weights(sh)
    ctx_tok = synth.tokens(synth.SEED_CONTEXT, 11, 512, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 11, 40, sh["vocab"])
    L, nblk = sh["n_layers"], 32
    # a 40-token prompt (tensor-core attention), then three one-token steps
    # (decode attention), a restore before the last one
    steps = [prm, prm[:1], prm[1:2], prm[2:3]]
    base, _ = _run(sh, w, ctx_tok, steps)
    perm = synth.permutation(synth.SEED_EVICT, 12, L * 16)[:11]  # blocks of positions < 256

    def evict(c):
        m.mzc_evict(c, 0, L, 256, 512, m.MZC_COPY)
        m.mzc_evict_blocks(c, perm // 16, perm % 16)

    got, swapped = _run(sh, w, ctx_tok, steps, evict, read_swapped=1, restore_after=3)
    n_sw = L * 16 + 11
    assert swapped == [n_sw, n_sw, n_sw, 0]       # in place until the restore
    for a, b in zip(base, got):
        assert np.array_equal(a, b)


def test_in_place_reads_need_the_written_block_resident():
    sh = W.TINY
    w = synth.model_weights(sh)
    c = m.mzc_create(sh, w, read_swapped=1)
    m.mzc_prefill(c, synth.tokens(synth.SEED_CONTEXT, 13, 500, sh["vocab"]))  # block 31 partial
    m.mzc_evict(c, 0, 2, 480, 500, m.MZC_COPY)
    toks = np.array([1, 2], np.int32)
    assert m.mzc.status_of("mzc_prefill", c, toks.ctypes.data, 2, None) == m.MZC_ERR_STATE
    m.mzc_restore_async(c)
    m.mzc_prefill(c, toks)          # restored: fine
    m.mzc_destroy(c)


def test_in_place_reads_refuse_the_8bit_store():
    import ctypes
    sh = W.TINY
    opt = m.mzc_options(0, 0, 0, 1, 0, m.MZC_CODEC_Q8, 0, 0, 1, None, None)
    w, keep = m.make_weights(synth.model_weights(sh))
    out = ctypes.c_void_p()
    shs = m.make_shape(sh)
    st = m.mzc.status_of("mzc_create", ctypes.byref(shs), ctypes.byref(opt), ctypes.byref(w),
                         ctypes.byref(out))
    assert st == m.MZC_ERR_INVALID and not out.value
    del keep
