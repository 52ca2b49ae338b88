"""The ctx options around the zero-wait overlap (Sec. 4.4: prefill consumes
each restored unit as soon as it lands), on the GPU through the C ABI:

  - MZC_WAIT_BLOCK_FLAG (per-block residency flags written by the copy engine,
    waited on by the attention kernels) gives the same logits as the
    per-layer events for copy restores, bit for bit, and matches the oracle
    for hybrid copy + recompute restores;
  - a flag that nothing sets makes the attention's bounded wait run out with
    MZC_ERR_TIMEOUT, and the CUDA context stays usable (tensor-core and
    decode kernels);
  - caller-owned compute and copy streams: the same logits, and the prefill
    runs behind work the caller queued on its compute stream;
  - debug_checks: the same logits."""
import time

import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from synth import workloads as W
from tests.gpu_util import f16_bits, f16_to_f32, f32_to_kv_bits, i32_dev, kv_bits_to_f32, rel_err, to_np_u16

pytestmark = pytest.mark.gpu

LOGIT_TOL = 2e-2


@pytest.fixture(scope="module")
def tiny():
    sh = W.TINY
    w = synth.model_weights(sh)
    ctx = synth.tokens(synth.SEED_CONTEXT, 0, 512, sh["vocab"])
    prm = synth.tokens(synth.SEED_PROMPT, 0, 32, sh["vocab"])
    kv = oracle.KVState(sh, sh["max_ctx"])
    lg_ref = oracle.prefill(sh, w, kv, np.concatenate([ctx, prm]), 0)
    return dict(shape=sh, w=w, ctx=ctx, prm=prm, lg_ref=lg_ref)


def _run(case, scenario, **opt):
    sh = case["shape"]
    c = m.mzc_create(sh, case["w"], **opt)
    m.mzc_prefill(c, case["ctx"])
    rec = scenario(c)
    m.mzc_restore_async(c)
    if rec:
        m.mzc_recompute_tail(c, *rec)
    lg = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, case["prm"], lg)
    k, v = m.mzc_read_kv_all(c, 544, sh)
    m.mzc_destroy(c)
    return lg, k, v


def _copy_tail(c):
    m.mzc_evict(c, 0, 2, 100, 512, m.MZC_COPY)


def _scattered(c):
    perm = synth.permutation(synth.SEED_EVICT, 0, 64)[:19]
    m.mzc_evict_blocks(c, perm // 32, perm % 32)


def _weights_and_copy(c):
    m.mzc_evict_weights(c, 1, 2)
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_COPY)


def _hybrid(c):
    m.mzc_evict(c, 0, 2, 256, 384, m.MZC_DROP)
    m.mzc_evict(c, 0, 2, 384, 512, m.MZC_COPY)
    return (256, 128)


def _hybrid_scattered(c):
    perm = synth.permutation(synth.SEED_EVICT, 4, 32)[:9]   # blocks of positions < 256
    m.mzc_evict_blocks(c, perm // 16, perm % 16)
    m.mzc_evict(c, 0, 2, 256, 512, m.MZC_DROP)
    return (256, 256)


@pytest.mark.parametrize("scenario", [_copy_tail, _scattered, _weights_and_copy])
def test_block_flags_copy_restores_are_bit_exact(tiny, scenario):
    ev = _run(tiny, scenario, wait_mode=m.MZC_WAIT_LAYER_EVENT)
    fl = _run(tiny, scenario, wait_mode=m.MZC_WAIT_BLOCK_FLAG)
    assert np.array_equal(ev[0], fl[0])
    assert np.array_equal(ev[1], fl[1]) and np.array_equal(ev[2], fl[2])
    assert np.max(np.abs(fl[0] - tiny["lg_ref"])) < LOGIT_TOL


@pytest.mark.parametrize("scenario", [_hybrid, _hybrid_scattered])
def test_block_flags_hybrid_restores_match_the_oracle(tiny, scenario):
    lg, _, _ = _run(tiny, scenario, wait_mode=m.MZC_WAIT_BLOCK_FLAG)
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    lg0, _, _ = _run(tiny, scenario, wait_mode=m.MZC_WAIT_BLOCK_FLAG, overlap=0)
    assert np.max(np.abs(lg0 - tiny["lg_ref"])) < LOGIT_TOL


def test_block_flags_refuse_the_8bit_store(tiny):
    import ctypes
    sh = m.make_shape(tiny["shape"])
    opt = m.mzc_options(0, 0, 0, 1, 0, m.MZC_CODEC_Q8, m.MZC_WAIT_BLOCK_FLAG, 0, 0, None, None)
    w, keep = m.make_weights(tiny["w"])
    out = ctypes.c_void_p()
    st = m.mzc.status_of("mzc_create", ctypes.byref(sh), ctypes.byref(opt), ctypes.byref(w),
                         ctypes.byref(out))
    assert st == m.MZC_ERR_INVALID and not out.value
    del keep


def test_debug_checks_change_no_result(tiny):
    for scenario in (_hybrid_scattered, _weights_and_copy):
        a = _run(tiny, scenario)
        b = _run(tiny, scenario, debug_checks=1)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_caller_streams(tiny):
    """The ctx runs on the caller's streams: the same logits as with its own
    streams, and a prefill queued behind a ~0.2 s sleep kernel on the caller's
    compute stream returns only after it."""
    import torch
    cs, xs = torch.cuda.Stream(), torch.cuda.Stream()
    base = _run(tiny, _hybrid_scattered)
    got = _run(tiny, _hybrid_scattered, compute_stream=cs.cuda_stream, copy_stream=xs.cuda_stream)
    assert np.array_equal(base[0], got[0]) and np.array_equal(base[1], got[1])
    sh = tiny["shape"]
    c = m.mzc_create(sh, tiny["w"], compute_stream=cs.cuda_stream, copy_stream=xs.cuda_stream)
    m.mzc_prefill(c, tiny["ctx"])
    _copy_tail(c)
    m.mzc_restore_async(c)
    with torch.cuda.stream(cs):
        torch.cuda._sleep(int(0.2 * 2.07e9))  # ~0.2 s at the top SM clock, longer below it
    t0 = time.perf_counter()
    lg = np.empty(sh["vocab"], np.float32)
    m.mzc_prefill(c, tiny["prm"], lg)
    dt = time.perf_counter() - t0
    assert dt > 0.05  # the prefill waited for the caller's queued work
    assert np.max(np.abs(lg - tiny["lg_ref"])) < LOGIT_TOL
    m.mzc_destroy(c)
    cs.synchronize()
    # the caller's streams outlive the ctx
    with torch.cuda.stream(cs):
        x = torch.ones(16, device="cuda") * 2
    cs.synchronize()
    assert float(x.sum()) == 32.0


# ---- kernel level: the bounded flag wait -------------------------------------

def _flag_case(hq, hkv, hd, kvd, ctx, pos, seed):
    import torch
    n = pos.size
    n_logical = -(-ctx // 16)
    pool_blocks = n_logical + 5
    table = synth.permutation(synth.SEED_EVICT, 200 + seed, pool_blocks)[:n_logical].astype(np.int32)
    rng = np.random.default_rng(seed)
    kf = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    vf = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    qf = f16_bits((rng.standard_normal((n, hq, hd)) * 2.0).astype(np.float32))
    pool_np = np.zeros((pool_blocks, 2, hkv, 16, hd), np.uint16)
    for p in range(ctx):
        pool_np[table[p // 16], 0, :, p % 16] = kf[p]
        pool_np[table[p // 16], 1, :, p % 16] = vf[p]
    dev = dict(q=torch.from_numpy(qf.view(np.int16)).cuda(), pos=i32_dev(pos), table=i32_dev(table),
               pool=torch.from_numpy(pool_np.view(np.int16)).cuda())
    ref = oracle.attention(f16_to_f32(qf), pos, kv_bits_to_f32(kf), kv_bits_to_f32(vf))
    return dev, n_logical, pool_blocks, table, ref


@pytest.mark.parametrize("hq,hkv,hd,kvd,ctx,n", [
    (32, 8, 64, 1, 700, 40),     # tensor-core kernel: 160 rows per KV head
    (24, 8, 128, 0, 3000, 60),   # tensor-core kernel, head dim 128
    (32, 8, 64, 1, 8197, 1),     # decode kernel: 4 rows per KV head, split-KV
])
def test_flag_wait_runs_out_and_the_context_stays_usable(hq, hkv, hd, kvd, ctx, n):
    import torch
    pos = np.arange(ctx - n, ctx).astype(np.int32)
    dev, n_logical, pool_blocks, table, ref = _flag_case(hq, hkv, hd, kvd, ctx, pos, seed=hd + n)
    flags = torch.ones(pool_blocks, dtype=torch.int32, device="cuda")
    flags[int(table[5])] = 0                       # a block whose restore never lands
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    sb = m.mzc_k_attention_scratch_bytes(n, hq, hkv, hd, ctx)
    scratch = torch.empty(max(sb, 16), dtype=torch.uint8, device="cuda")
    limit = 100_000_000                            # ~50 ms of SM clocks
    t0 = time.perf_counter()
    m.mzc_k_attention_wait(dev["q"], dev["pos"], n, hq, hkv, hd, dev["table"], n_logical, dev["pool"],
                           pool_blocks, kvd, out, ctx, scratch, sb, flags, limit, status)
    torch.cuda.synchronize()
    assert int(status.item()) == m.MZC_ERR_TIMEOUT
    assert time.perf_counter() - t0 < 30.0
    # the same call with every flag set completes and matches the oracle
    flags.fill_(1)
    status.zero_()
    m.mzc_k_attention_wait(dev["q"], dev["pos"], n, hq, hkv, hd, dev["table"], n_logical, dev["pool"],
                           pool_blocks, kvd, out, ctx, scratch, sb, flags, limit, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got = f16_to_f32(to_np_u16(out))
    assert rel_err(got, ref) < 1e-2
    # and the ordinary entry point still runs
    out2 = torch.zeros_like(out)
    m.mzc_k_attention(dev["q"], dev["pos"], n, hq, hkv, hd, dev["table"], n_logical, dev["pool"],
                      pool_blocks, kvd, out2, ctx, scratch, sb, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    assert np.array_equal(to_np_u16(out2), to_np_u16(out))
