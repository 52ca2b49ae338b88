"""The allocation-free attention entry point against the CPU oracle and the
ordinary entry point.

Some callers cannot allocate device memory when they call: a process whose
device memory is being reclaimed cannot count on an allocation succeeding at
request time, a host framework may own all device memory through its own
allocator, and cudaFree synchronizes the device.  mzc_k_attention_noalloc
serves them by keeping its split-KV partials in a fixed device array inside
the library.  This file checks, through the C ABI, on two calls in a row with
different shapes and inputs (so the second call cannot lean on the first
call's partials left in the array):
  - the output against the CPU oracle's attention over the same K/V, q and
    positions, at the tolerance of the other attention parity tests;
  - the output against mzc_k_attention with caller-allocated scratch, at the
    same tolerance;
and that a call whose partials would not fit in the array is refused without
a launch.  It is named to be collected last."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from tests.gpu_util import f16_to_f32, f32_to_kv_bits, i32_dev, kv_bits_to_f32, rel_err, to_np_u16

pytestmark = pytest.mark.gpu

ATTN_TOL = 1e-2  # max|d| / max|ref|, as in the attention parity tests


def _inputs(seed, hq, hkv, hd, kvd, ctx, n):
    import torch
    n_logical = -(-ctx // 16)
    pool_blocks = n_logical + 7
    table = synth.permutation(synth.SEED_EVICT, 100 + seed, pool_blocks)[:n_logical].astype(np.int32)
    rng = np.random.default_rng(seed)
    k = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    v = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    q = (rng.standard_normal((n, hq, hd)) * 2.0).astype(np.float16).view(np.uint16)
    pool = np.zeros((pool_blocks, 2, hkv, 16, hd), np.uint16)
    for p in range(ctx):
        pool[table[p // 16], 0, :, p % 16] = k[p]
        pool[table[p // 16], 1, :, p % 16] = v[p]
    pos = np.arange(ctx - n, ctx).astype(np.int32)
    dev = dict(q=torch.from_numpy(q.view(np.int16)).cuda(), pos=i32_dev(pos),
               table=i32_dev(table), pool=torch.from_numpy(pool.view(np.int16)).cuda())
    # the oracle's attention over the same stored values (fp16-encoded pool)
    ref = oracle.attention(f16_to_f32(q), pos, kv_bits_to_f32(k), kv_bits_to_f32(v))
    return dev, n_logical, pool_blocks, ref


def _one_call(seed, hq, hkv, hd, kvd, ctx, n):
    import torch
    dev, n_logical, pool_blocks, oracle_ref = _inputs(seed, hq, hkv, hd, kvd, ctx, n)
    need = m.mzc_k_attention_scratch_bytes(n, hq, hkv, hd, ctx)
    assert 0 < need <= m.MZC_ATTENTION_NOALLOC_SCRATCH_BYTES  # the split path is exercised
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    scratch = torch.empty(need, dtype=torch.uint8, device="cuda")
    m.mzc_k_attention(dev["q"], dev["pos"], n, hq, hkv, hd, dev["table"], n_logical, dev["pool"],
                      pool_blocks, kvd, ref, ctx, scratch, need, status)
    out = torch.full((n, hq, hd), -1, dtype=torch.int16, device="cuda")
    m.mzc_k_attention_noalloc(dev["q"], dev["pos"], n, hq, hkv, hd, dev["table"], n_logical,
                              dev["pool"], pool_blocks, kvd, out, ctx, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got, want = f16_to_f32(to_np_u16(out)), f16_to_f32(to_np_u16(ref))
    assert np.all(np.isfinite(got))
    assert rel_err(got, oracle_ref) < ATTN_TOL
    assert np.mean(np.abs(got - oracle_ref)) < 2e-3 * np.max(np.abs(oracle_ref))
    assert rel_err(got, want) < ATTN_TOL


def test_noalloc_matches_scratch_entry_on_consecutive_calls():
    _one_call(1, 24, 8, 128, 0, 5000, 9)   # first call on this device sets the array up
    _one_call(2, 32, 8, 64, 1, 3000, 5)    # second call, different shape and KV type


def test_noalloc_rejects_calls_beyond_the_array():
    import torch
    hq, hkv, hd, n, ctx = 24, 8, 128, 200, 32768
    assert m.mzc_k_attention_scratch_bytes(n, hq, hkv, hd, ctx) > m.MZC_ATTENTION_NOALLOC_SCRATCH_BYTES
    small = torch.zeros(16, dtype=torch.int32, device="cuda")
    out = torch.zeros(16, dtype=torch.int16, device="cuda")
    st = m.mzc.status_of("mzc_k_attention_noalloc", small.data_ptr(), small.data_ptr(), n, hq, hkv,
                         hd, small.data_ptr(), 1, small.data_ptr(), 1, 0, out.data_ptr(), ctx,
                         None, None)
    assert st == m.MZC_ERR_RANGE
    assert "fixed" in m.mzc_last_error(None)
    torch.cuda.synchronize()
