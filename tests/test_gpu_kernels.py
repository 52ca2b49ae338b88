"""Kernel parity on the GPU: each sm_103a kernel, called through the C ABI,
against the CPU oracle's definition of the same operation on the same seeded
inputs.  Tolerances follow from the arithmetic: fp16 outputs are within one
fp16 rounding (2^-11 relative) of an fp32 reference plus fp32 accumulation-
order noise; the attention's P operand is rounded to the KV type."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from tests.gpu_util import (bf16_dev, f32_dev, i32_dev, to_np_u16, kv_bits_to_f32,
                            f32_to_kv_bits, rel_err, f16_bits, f16_to_f32,
                            bf16_weights_exact_in_f16)

pytestmark = pytest.mark.gpu


def _torch():
    import torch
    return torch


def _rand_bf16(tid, shape, sigma=1.0):
    return synth.normal_bf16(7, tid, shape, sigma=sigma)


# ---- GEMM (tcgen05 / TMEM / TMA) -------------------------------------------

# m <= 4: the few-row GEMV path; larger m: the tcgen05 GEMM
# m > 512: the paired-SM kernel (256 x 256 tiles over a CTA pair), with an odd
# M-tile count (4224 rows: 33 tiles) and N not a multiple of 256 (384)
GEMM_SHAPES = [(1, 64, 64), (2, 1024, 2048), (4, 3072, 3072), (7, 80, 72), (128, 256, 512),
               (130, 384, 320), (300, 1024, 2048), (1000, 512, 256), (1000, 384, 320),
               (4224, 3072, 2048)]


def _act16(tid, shape):
    return f16_bits(synth.bf16_bits_to_f32(_rand_bf16(tid, shape)))


@pytest.mark.parametrize("mm,nn,kk", GEMM_SHAPES)
def test_gemm_store_f16(mm, nn, kk):
    torch = _torch()
    a = _act16(1, (mm, kk))
    wb, wh = bf16_weights_exact_in_f16(_rand_bf16(2, (nn, kk), sigma=0.05))
    out = torch.zeros((mm, nn), dtype=torch.int16, device="cuda")
    m.mzc_k_gemm(bf16_dev(a), bf16_dev(wh), out, mm, nn, kk, 0)
    torch.cuda.synchronize()
    got = f16_to_f32(to_np_u16(out))
    rows = np.unique(np.linspace(0, mm - 1, min(mm, 256)).astype(int))
    ref = oracle.linear(f16_to_f32(a[rows]), wb)
    err = np.abs(got[rows] - ref)
    assert np.all(err <= 2.0 ** -10 * np.abs(ref) + 1e-5 * np.max(np.abs(ref)))


@pytest.mark.parametrize("mm,nn,kk", [(1, 2048, 8192), (3, 3072, 1024), (5, 64, 128), (200, 256, 768),
                                     (1300, 640, 200), (4224, 2048, 2048)])
def test_gemm_residual_add(mm, nn, kk):
    torch = _torch()
    a = _act16(3, (mm, kk))
    wb, wh = bf16_weights_exact_in_f16(_rand_bf16(4, (nn, kk), sigma=0.05))
    x0 = np.random.default_rng(0).standard_normal((mm, nn)).astype(np.float32)
    out = f32_dev(x0)
    m.mzc_k_gemm(bf16_dev(a), bf16_dev(wh), out, mm, nn, kk, 1)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    rows = np.unique(np.linspace(0, mm - 1, min(mm, 256)).astype(int))
    ref = x0[rows] + oracle.linear(f16_to_f32(a[rows]), wb)
    assert np.max(np.abs(got[rows] - ref)) <= 1e-4 * np.max(np.abs(ref))


@pytest.mark.parametrize("mm,f,kk", [(1, 1024, 2048), (3, 128, 256), (4, 256, 512), (260, 384, 512),
                                     (70, 704, 256), (900, 384, 512),
                                     (4224, 1024, 2048)])
def test_gemm_swiglu(mm, f, kk):
    torch = _torch()
    a = _act16(5, (mm, kk))
    wg, wgh = bf16_weights_exact_in_f16(_rand_bf16(6, (f, kk), sigma=0.05))
    wu, wuh = bf16_weights_exact_in_f16(_rand_bf16(8, (f, kk), sigma=0.05))
    packed = m.mzc_k_swiglu_pack(wgh, wuh)
    out = torch.zeros((mm, f), dtype=torch.int16, device="cuda")
    m.mzc_k_gemm(bf16_dev(a), bf16_dev(packed), out, mm, 2 * f, kk, 2)
    torch.cuda.synchronize()
    got = f16_to_f32(to_np_u16(out))
    rows = np.unique(np.linspace(0, mm - 1, min(mm, 128)).astype(int))
    af = f16_to_f32(a[rows])
    ref = oracle.swiglu(oracle.linear(af, wg), oracle.linear(af, wu))
    err = np.abs(got[rows] - ref)
    assert np.all(err <= 2.0 ** -9 * np.abs(ref) + 2e-5 * np.max(np.abs(ref)))


@pytest.mark.parametrize("mm,nn,kk,epi", [(128, 3072, 8192, 1), (128, 5120, 3072, 0), (256, 3072, 3072, 1),
                                         (200, 2048, 4096, 2), (37, 1024, 1000, 0), (9, 128, 64, 1)])
def test_gemm_split_k_over_a_cluster(mm, nn, kk, epi):
    """m <= 256 with few 128-column tiles: the K range is split over the CTAs
    of a cluster and the partials summed in split order through distributed
    shared memory; the result matches the oracle and repeats bit for bit."""
    torch = _torch()
    a = _act16(11, (mm, kk))
    wb, wh = bf16_weights_exact_in_f16(_rand_bf16(12, (nn, kk), sigma=0.05))
    ncol = nn // 2 if epi == 2 else nn
    x0 = np.random.default_rng(1).standard_normal((mm, ncol)).astype(np.float32)
    if epi == 2:
        w = m.mzc_k_swiglu_pack(wh[: nn // 2], wh[nn // 2:])
        wg, wu = wb[: nn // 2], wb[nn // 2:]
    else:
        w = wh
    outs = []
    for _ in range(2):
        out = f32_dev(x0) if epi == 1 else torch.zeros((mm, ncol), dtype=torch.int16, device="cuda")
        m.mzc_k_gemm(bf16_dev(a), bf16_dev(w), out, mm, nn, kk, epi)
        torch.cuda.synchronize()
        outs.append(out.cpu().numpy() if epi == 1 else f16_to_f32(to_np_u16(out)))
    assert np.array_equal(outs[0], outs[1])
    got = outs[0]
    af = f16_to_f32(a)
    if epi == 0:
        ref = oracle.linear(af, wb)
        assert np.all(np.abs(got - ref) <= 2.0 ** -10 * np.abs(ref) + 1e-5 * np.max(np.abs(ref)))
    elif epi == 1:
        ref = x0 + oracle.linear(af, wb)
        assert np.max(np.abs(got - ref)) <= 1e-4 * np.max(np.abs(ref))
    else:
        ref = oracle.swiglu(oracle.linear(af, wg), oracle.linear(af, wu))
        assert np.all(np.abs(got - ref) <= 2.0 ** -9 * np.abs(ref) + 2e-5 * np.max(np.abs(ref)))


@pytest.mark.parametrize("epi", [0, 1, 2])
@pytest.mark.parametrize("mm,nn", [(5, 128), (300, 384), (1000, 2048)])
def test_gemm_writes_only_its_rows(epi, mm, nn):
    """The epilogue's TMA stores are clipped at m rows: guard rows after the
    output keep their sentinel, every row before it is written."""
    torch = _torch()
    kk = 128
    a = _act16(9, (mm, kk))
    _, wh = bf16_weights_exact_in_f16(_rand_bf16(10, (nn, kk), sigma=0.05))
    ncol = nn // 2 if epi == 2 else nn
    guard = 40
    if epi == 1:
        buf = torch.full((mm + guard, ncol), 7.0, dtype=torch.float32, device="cuda")
    else:
        buf = torch.full((mm + guard, ncol), 0x1234, dtype=torch.int16, device="cuda")
    w = m.mzc_k_swiglu_pack(wh[: nn // 2], wh[nn // 2:]) if epi == 2 else wh
    m.mzc_k_gemm(bf16_dev(a), bf16_dev(w), buf[:mm], mm, nn, kk, epi)
    torch.cuda.synchronize()
    host = buf.cpu().numpy()
    sentinel = 7.0 if epi == 1 else 0x1234
    assert np.all(host[mm:] == sentinel)
    assert not np.any(np.all(host[:mm] == sentinel, axis=1))


# ---- 8-bit swap codec ------------------------------------------------------------

@pytest.mark.parametrize("hkv,hd,kvd", [(2, 64, 1), (8, 128, 0), (8, 64, 1)])
def test_q8_codec_matches_oracle(hkv, hd, kvd):
    """Encoded bytes (codes and fp32 min/step) and decoded fp16 bits equal the
    oracle's, through a block list and into a contiguous run."""
    torch = _torch()
    e = 2 * hkv * 16 * hd
    nb = 12
    rng = np.random.default_rng(hd + hkv)
    vals = (rng.standard_normal((nb, e)) * np.exp(rng.uniform(-3, 2, (nb, 1)))).astype(np.float32)
    bits = oracle.to_f16_bits(oracle.round_kv(vals, kvd))  # as the pool stores values
    bits[3, :64] = bits[3, 0]                                 # a constant group
    pool = torch.from_numpy(bits.view(np.int16)).cuda()
    phys = np.array([7, 2, 11, 3, 0], np.int32)
    cb = m.mzc_q8_block_bytes(hkv, hd)
    assert cb == oracle.q8_block_bytes(hkv, hd)
    comp = torch.zeros((len(phys), cb), dtype=torch.uint8, device="cuda")
    m.mzc_k_q8_encode(pool, i32_dev(phys), len(phys), hkv, hd, comp)
    torch.cuda.synchronize()
    ref = oracle.q8_encode_blocks(bits[phys])
    assert np.array_equal(comp.cpu().numpy(), ref)
    dec = oracle.q8_decode_blocks(ref, e, kvd)
    out = torch.zeros((nb, e), dtype=torch.int16, device="cuda")
    dst = np.array([1, 9, 4, 10, 6], np.int32)
    m.mzc_k_q8_decode(comp, len(phys), hkv, hd, i32_dev(dst), 0, kvd, out)
    run = torch.zeros((nb, e), dtype=torch.int16, device="cuda")
    m.mzc_k_q8_decode(comp, 3, hkv, hd, None, 5, kvd, run)
    torch.cuda.synchronize()
    got, got_run = to_np_u16(out), to_np_u16(run)
    assert np.array_equal(got[dst], dec)
    assert np.array_equal(got_run[5:8], dec[:3])
    untouched = np.setdiff1d(np.arange(nb), dst)
    assert not got[untouched].any() and not got_run[:5].any() and not got_run[8:].any()


# ---- RMSNorm, embedding, LM head --------------------------------------------

# n <= 512 takes one CTA per row, more rows one warp per row (d a multiple of
# 256), other widths the generic kernel
@pytest.mark.parametrize("n,d", [(1, 256), (37, 2048), (300, 3072), (5, 320), (3, 4608), (9, 4096),
                                 (512, 3072), (513, 3072), (1100, 2048), (700, 4096), (600, 320)])
def test_rmsnorm(n, d):
    torch = _torch()
    rng = np.random.default_rng(n)
    x = (rng.standard_normal((n, d)) * rng.uniform(0.01, 3.0, (n, 1))).astype(np.float32)
    g = rng.uniform(0.5, 1.5, d).astype(np.float32)
    y = torch.zeros((n, d), dtype=torch.int16, device="cuda")
    m.mzc_k_rmsnorm(f32_dev(x), f32_dev(g), n, d, 1e-5, y)
    torch.cuda.synchronize()
    got = f16_to_f32(to_np_u16(y))
    ref = oracle.rmsnorm(x, g, 1e-5)
    assert np.all(np.abs(got - ref) <= 2.0 ** -10 * np.abs(ref) + 1e-6)


def test_embed_exact_and_bad_token_flagged():
    torch = _torch()
    V, d = 1000, 512
    E = _rand_bf16(9, (V, d), sigma=0.02)
    toks = synth.tokens(1, 9, 77, V)
    x = torch.zeros((77, d), dtype=torch.float32, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    m.mzc_k_embed(i32_dev(toks), 77, bf16_dev(E), d, V, x, status)
    torch.cuda.synchronize()
    assert np.array_equal(x.cpu().numpy(), synth.bf16_bits_to_f32(E[toks]))
    assert int(status.item()) == 0
    bad = toks.copy()
    bad[3] = V + 5
    m.mzc_k_embed(i32_dev(bad), 77, bf16_dev(E), d, V, x, status)
    torch.cuda.synchronize()
    assert int(status.item()) == m.MZC_ERR_DEVICE


@pytest.mark.parametrize("V,d", [(1024, 256), (128256, 2048), (50000, 3072)])
def test_lm_head(V, d):
    torch = _torch()
    rng = np.random.default_rng(V)
    x = rng.standard_normal(d).astype(np.float32)
    g = rng.uniform(0.5, 1.5, d).astype(np.float32)
    W = _rand_bf16(10, (V, d), sigma=0.02)
    logits = torch.zeros(V, dtype=torch.float32, device="cuda")
    m.mzc_k_lm_head(f32_dev(x), f32_dev(g), d, 1e-5, bf16_dev(W), V, logits)
    torch.cuda.synchronize()
    h = oracle.rmsnorm(x[None], g, 1e-5)
    ref = oracle.linear(h, W)[0]
    assert np.max(np.abs(logits.cpu().numpy() - ref)) <= 1e-5 * np.max(np.abs(ref)) * np.sqrt(d)


# ---- rotary + KV-block write -------------------------------------------------

def _pool_layout(n_blocks_logical, pool_blocks, seed):
    perm = synth.permutation(synth.SEED_EVICT, seed, pool_blocks)[:n_blocks_logical]
    return perm.astype(np.int32)


@pytest.mark.parametrize("hq,hkv,hd,kvd", [(4, 2, 64, 0), (32, 8, 64, 1), (24, 8, 128, 0)])
def test_rope_kv_write(hq, hkv, hd, kvd):
    torch = _torch()
    n_logical, pool_blocks = 40, 64
    # ragged positions: a recompute range and a prompt range
    pos = np.concatenate([np.arange(100, 180), np.arange(600, 637)]).astype(np.int32)
    n = pos.size
    qkv = _act16(11, (n, (hq + 2 * hkv) * hd))
    table = _pool_layout(n_logical, pool_blocks, hd + kvd)
    cos_t, sin_t = oracle.rope_table(n_logical * 16, hd, 500000.0)
    blk_elems = 2 * hkv * 16 * hd
    pool = torch.zeros(pool_blocks * blk_elems, dtype=torch.int16, device="cuda")
    q_out = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    m.mzc_k_rope_kv_write(bf16_dev(qkv), i32_dev(pos), n, hq, hkv, hd, f32_dev(cos_t),
                          f32_dev(sin_t), i32_dev(table), n_logical, pool, pool_blocks, kvd,
                          q_out, status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    x = f16_to_f32(qkv).reshape(n, hq + 2 * hkv, hd)
    k_ref = oracle.round_kv(oracle.rope(x[:, hq:hq + hkv], pos, 500000.0), kvd)
    v_ref = oracle.round_kv(x[:, hq + hkv:], kvd)
    ulp = 2.0 ** (-10 if kvd == 1 else -7)
    q_got = f16_to_f32(to_np_u16(q_out))  # q is fp16 for both KV types
    q_ref = oracle.rope(x[:, :hq], pos, 500000.0)
    assert np.all(np.abs(q_got - q_ref) <= 2.0 ** -10 * np.abs(q_ref) + 1e-6)
    pool_np = to_np_u16(pool).reshape(pool_blocks, 2, hkv, 16, hd)
    k_got = np.stack([pool_np[table[p // 16], 0, :, p % 16] for p in pos])
    v_got = np.stack([pool_np[table[p // 16], 1, :, p % 16] for p in pos])
    assert np.all(np.abs(kv_bits_to_f32(k_got, kvd) - k_ref) <= ulp * np.abs(k_ref) + 1e-7)
    assert np.array_equal(kv_bits_to_f32(v_got, kvd), v_ref)
    # nothing else in the pool was written
    written = np.zeros((pool_blocks, 16), bool)
    for p in pos:
        written[table[p // 16], p % 16] = True
    untouched = pool_np.transpose(0, 3, 1, 2, 4)[~written]
    assert not untouched.any()


# ---- block-table attention ----------------------------------------------------

def _attention_case(hq, hkv, hd, kvd, ctx, pos, seed, use_scratch=True):
    torch = _torch()
    n = pos.size
    n_logical = -(-ctx // 16)
    pool_blocks = n_logical + 13
    table = _pool_layout(n_logical, pool_blocks, seed)
    rng = np.random.default_rng(seed)
    kf = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    vf = f32_to_kv_bits(rng.standard_normal((ctx, hkv, hd)).astype(np.float32), kvd)
    qf = f16_bits((rng.standard_normal((n, hq, hd)) * 2.0).astype(np.float32))
    pool_np = np.zeros((pool_blocks, 2, hkv, 16, hd), np.uint16)
    for p in range(ctx):
        pool_np[table[p // 16], 0, :, p % 16] = kf[p]
        pool_np[table[p // 16], 1, :, p % 16] = vf[p]
    pool = torch.from_numpy(pool_np.view(np.int16)).cuda()
    out = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    sb = m.mzc_k_attention_scratch_bytes(n, hq, hkv, hd, ctx) if use_scratch else 0
    scratch = torch.empty(max(sb, 4), dtype=torch.uint8, device="cuda") if sb else None
    m.mzc_k_attention(torch.from_numpy(qf.view(np.int16)).cuda(), i32_dev(pos), n, hq, hkv, hd,
                      i32_dev(table), n_logical, pool, pool_blocks, kvd, out, ctx, scratch, sb,
                      status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    got = f16_to_f32(to_np_u16(out))
    ref = oracle.attention(f16_to_f32(qf), pos, kv_bits_to_f32(kf), kv_bits_to_f32(vf))
    return got, ref, sb


@pytest.mark.parametrize("hq,hkv,hd,kvd", [(4, 2, 64, 0), (32, 8, 64, 1), (24, 8, 128, 0),
                                           (8, 8, 128, 1)])
def test_attention_ragged_rows(hq, hkv, hd, kvd):
    ctx = 700
    pos = np.concatenate([np.arange(300, 383), np.arange(680, 700), [0, 17]]).astype(np.int32)
    got, ref, _ = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=hq + hd)
    assert rel_err(got, ref) < 1e-2
    assert np.mean(np.abs(got - ref)) < 2e-3 * np.max(np.abs(ref))


@pytest.mark.parametrize("hq,hkv,hd,kvd", [(32, 8, 64, 1), (24, 8, 128, 0)])
def test_attention_split_kv_long_context(hq, hkv, hd, kvd):
    ctx = 5000
    pos = np.arange(ctx - 9, ctx).astype(np.int32)
    got, ref, sb = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=3)
    assert sb > 0  # the split path ran
    assert rel_err(got, ref) < 1e-2
    got2, ref2, _ = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=3, use_scratch=False)
    assert rel_err(got2, ref2) < 1e-2


@pytest.mark.parametrize("hq,hkv,hd,kvd,n", [(24, 8, 128, 0, 128), (32, 8, 64, 1, 96),
                                             (24, 8, 128, 1, 171)])
def test_attention_split_kv_half_last_row_tile(hq, hkv, hd, kvd, n):
    """A prompt whose rows per KV head (n x hq/hkv) leave the last 256-row
    tile with one Q tile of two (or a single row), split over the keys: the
    padding Q tile gets no work and every real row is merged over all splits."""
    ctx = 4224 + n
    pos = np.arange(ctx - n, ctx).astype(np.int32)  # the prompt's diagonal is in every split's reach
    got, ref, sb = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=n)
    assert sb > 0  # the split path ran
    assert rel_err(got, ref) < 1e-2
    assert np.mean(np.abs(got - ref)) < 2e-3 * np.max(np.abs(ref))


@pytest.mark.parametrize("hq,hkv,hd,kvd,n,ctx", [
    (32, 8, 64, 1, 1, 8197),     # 1B decode token: 4 rows per KV head, split-KV, ragged end
    (32, 8, 64, 1, 1, 70_000),   # more than 32 blocks per warp pair and split
    (24, 8, 128, 0, 1, 32768),   # 3B decode token at the 3B context
    (24, 8, 128, 0, 1, 777),     # ragged last block
    (4, 2, 64, 0, 2, 530),       # tiny config, two tokens: 4 rows per KV head
    (8, 8, 128, 1, 3, 100),      # no GQA; fewer blocks than warp pairs
    (8, 8, 64, 0, 4, 16),        # a single block
])
def test_attention_decode_rows(hq, hkv, hd, kvd, n, ctx):
    """At most 4 query rows per KV head take the decode kernel; with the
    split-KV scratch and without it (one split)."""
    pos = np.arange(ctx - n, ctx).astype(np.int32)
    got, ref, sb = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=n + hd)
    assert rel_err(got, ref) < 1e-2
    assert np.mean(np.abs(got - ref)) < 2e-3 * np.max(np.abs(ref))
    got2, ref2, _ = _attention_case(hq, hkv, hd, kvd, ctx, pos, seed=n + hd, use_scratch=False)
    assert rel_err(got2, ref2) < 1e-2


def test_attention_decode_rows_at_scattered_positions():
    """Rows of one call at far-apart positions each see only their own causal
    prefix (a row at position 0 attends to one key)."""
    pos = np.array([0, 17, 2500, 4098], np.int32)
    got, ref, _ = _attention_case(8, 8, 128, 1, 4099, pos, seed=7)
    assert rel_err(got, ref) < 1e-2
    # the row at position 0 is exactly V of key 0 (one weight of 1)
    assert np.max(np.abs(got[0] - ref[0])) <= 2.0 ** -10 * np.max(np.abs(ref[0])) + 1e-6


def test_bounded_wait_runs_out_and_context_stays_usable():
    """A pipeline wait that nothing completes runs out after its limit (about
    half a second here), records MZC_ERR_TIMEOUT, and the next kernels run."""
    torch = _torch()
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    done = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    m.mzc_k_wait_probe(0, 1_000_000_000, status, done)
    torch.cuda.synchronize()
    assert int(done.item()) == 0 and int(status.item()) == m.MZC_ERR_TIMEOUT
    status.zero_()
    m.mzc_k_wait_probe(1, 1_000_000_000, status, done)
    torch.cuda.synchronize()
    assert int(done.item()) == 1 and int(status.item()) == 0
    # the context is usable: a GEMM right after is still correct
    test_gemm_store_f16(128, 256, 512)


@pytest.mark.parametrize("bad", [-3, 10_000])
@pytest.mark.parametrize("n", [4, 1])  # 16 rows per KV head (tensor-core kernel), 4 (decode kernel)
def test_attention_flags_a_block_table_entry_outside_the_pool(bad, n):
    """A block-table entry outside the pool is a device error: the kernel
    records MZC_ERR_DEVICE and reads an in-pool block instead (no stray
    address)."""
    torch = _torch()
    hq, hkv, hd, ctx = 8, 2, 64, 200
    n_logical = (ctx + 15) // 16
    pool_blocks = n_logical + 3
    table = np.arange(n_logical, dtype=np.int32)
    table[5] = bad
    pool = torch.zeros((pool_blocks, 2, hkv, 16, hd), dtype=torch.int16, device="cuda")
    q = torch.zeros((n, hq, hd), dtype=torch.int16, device="cuda")
    pos = np.array([150, 160, 170, 199], np.int32)[-n:]
    out = torch.zeros_like(q)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    m.mzc_k_attention(q, i32_dev(pos), n, hq, hkv, hd, i32_dev(table), n_logical, pool, pool_blocks,
                      1, out, ctx, None, 0, status)
    torch.cuda.synchronize()
    assert int(status.item()) == m.MZC_ERR_DEVICE
