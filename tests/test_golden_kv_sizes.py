"""The KV bytes of a context, pinned to the sizes the paper prints for its
evaluation models (tests/golden/paper_kv_sizes.txt, Sec. 6.1).

Two sides are checked against the same printed numbers: the oracle's KV
state (K and V for every layer, KV head and head-dim entry of a position,
held in fp16 by the method), and the library's swap-store accounting (a
pinned store of exactly the context's KV bytes takes a COPY eviction of the
whole context; one byte less is refused).  A dropped term on either side (V
forgotten, the KV heads or the layers missed) fails here."""
import math
import os


import oracle
import paper_2609_01338_gb300 as m
from paper_2609_01338_gb300 import mzc as M
from synth import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
CONTEXTS = (8192, 16384, 32768)


def _rows():
    for line in open(os.path.join(HERE, "golden", "paper_kv_sizes.txt")):
        if line.startswith("#") or not line.strip():
            continue
        f = line.split()
        yield f[0], int(f[1]), int(f[2]), int(f[3]), [float(x) for x in f[4:7]]


def _shape(layers, kv_heads, head_dim, max_ctx):
    # only the KV dimensions matter here; the rest is any valid decoder
    return W.shape(layers, kv_heads * head_dim, kv_heads, kv_heads, head_dim, 256, 1024,
                   W.KV_FP16, max_ctx=max_ctx)


def test_golden_file_has_both_models():
    assert [r[0] for r in _rows()] == ["Qwen3-0.6B", "EXAONE-4.0-1.2B"]


def test_oracle_kv_state_matches_the_printed_sizes():
    for name, layers, kvh, hd, printed in _rows():
        kv = oracle.KVState(_shape(layers, kvh, hd, 16), 16)
        per_token_fp16 = (kv.k.size + kv.v.size) * 2 / 16
        for ctx, want in zip(CONTEXTS, printed):
            gib = per_token_fp16 * ctx / 2 ** 30
            assert math.ceil(gib * 10 - 1e-9) / 10 == want, (name, ctx, gib)


def test_library_swap_store_holds_exactly_the_context_kv():
    for name, layers, kvh, hd, printed in _rows():
        for ctx, want in zip(CONTEXTS, printed):
            need = layers * ctx * 2 * kvh * hd * 2  # fp16 K and V of every layer
            assert math.ceil(need / 2 ** 30 * 10 - 1e-9) / 10 == want, (name, ctx)
            for store, ok in ((need, True), (need - 1, False)):
                st = m.mzc_state_create(_shape(layers, kvh, hd, ctx), host_store_bytes=store)
                try:
                    assert M.status_of("mzc_state_append", st, ctx) == m.MZC_OK
                    s = M.status_of("mzc_state_evict", st, 0, layers, 0, ctx, m.MZC_COPY)
                    assert s == (m.MZC_OK if ok else m.MZC_ERR_OOM), (name, ctx, store)
                finally:
                    M.status_of("mzc_state_destroy", st)
