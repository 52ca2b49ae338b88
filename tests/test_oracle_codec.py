"""Pins of the oracle's 8-bit swap codec (8-bit quantization as the default
swap compression, Sec. 5; idempotent, Sec. 6.5).  Format reading: asymmetric
min/max over groups of 64, fp32 min and step = (max - min) / 255, codes by
round-half-even, value = code * step + min.  Each pin is fixed by that
definition, not by re-running the oracle's own arithmetic."""
import numpy as np

import oracle


def _groups(seed, n, scale_lo=1e-3, scale_hi=30.0):
    rng = np.random.default_rng(seed)
    scales = np.exp(rng.uniform(np.log(scale_lo), np.log(scale_hi), (n, 1)))
    offs = rng.standard_normal((n, 1)) * scales
    return (rng.standard_normal((n, 64)) * scales + offs).astype(np.float32)


def test_code_is_a_nearest_level_and_range_is_full():
    x = _groups(1, 2000)
    codes, mn, st = oracle.q8_encode(x)
    # the exact real ratio (float64) is within half a level of the chosen code
    ratio = (x.astype(np.float64) - mn.astype(np.float64)) / st.astype(np.float64)
    assert np.all(np.abs(codes - ratio) <= 0.5 + 1e-4)
    # min and max of every group are in it; they take the end codes
    assert np.all(mn[:, 0] == x.min(axis=1))
    assert np.all(codes.min(axis=1) == 0) and np.all(codes.max(axis=1) == 255)
    np.testing.assert_allclose(st[:, 0] * 255, x.max(axis=1) - x.min(axis=1), rtol=1e-6)


def test_reconstruction_error_is_at_most_half_a_step():
    x = _groups(2, 2000)
    codes, mn, st = oracle.q8_encode(x)
    y = oracle.q8_decode(codes, mn, st)
    ulp = np.spacing(np.maximum(np.abs(x), np.abs(y)))
    assert np.all(np.abs(x - y) <= st / 2 + 4 * ulp)
    # the minimum of each group decodes exactly
    assert np.all(y[np.arange(len(x)), x.argmin(axis=1)] == x.min(axis=1))


def test_constant_and_two_valued_groups():
    c = np.full((3, 64), 1.25, np.float32)
    codes, mn, st = oracle.q8_encode(c)
    assert np.all(codes == 0) and np.all(st == 0)
    assert np.array_equal(oracle.q8_decode(codes, mn, st), c)
    two = np.where(np.arange(64) % 2 == 0, -3.0, 5.0).astype(np.float32)[None, :]
    codes, mn, st = oracle.q8_encode(two)
    assert set(codes[0].tolist()) == {0, 255}
    assert mn[0, 0] == -3.0 and st[0, 0] == np.float32(8.0) / np.float32(255.0)


def test_idempotent_under_repeated_swap():
    """Sec. 6.5: repeated compression and decompression does not accumulate
    error: the second encoding of the decoded values gives the same codes."""
    x = _groups(3, 5000)
    c1, m1, s1 = oracle.q8_encode(x)
    y1 = oracle.q8_decode(c1, m1, s1)
    c2, m2, s2 = oracle.q8_encode(y1)
    y2 = oracle.q8_decode(c2, m2, s2)
    assert np.array_equal(c1, c2)
    assert np.array_equal(m1, m2)
    assert np.max(np.abs(y2 - y1) / np.maximum(s1, 1e-30)) <= 1e-3


def test_block_format_and_round_trip():
    hkv, hd = 2, 128
    e = 2 * hkv * 16 * hd
    assert oracle.q8_block_bytes(hkv, hd) == e + 8 * (e // 64)
    rng = np.random.default_rng(4)
    vals = (rng.standard_normal((3, e)) * 2).astype(np.float16)
    comp = oracle.q8_encode_blocks(vals.view(np.uint16))
    assert comp.shape == (3, oracle.q8_block_bytes(hkv, hd))
    # group g of block i: codes at [g*64, g*64+64), (min, step) at e + 8g
    g = 5
    grp = vals[1, g * 64:(g + 1) * 64].astype(np.float32)
    mn, st = comp[1, e + 8 * g:e + 8 * g + 8].view(np.float32)
    assert mn == grp.min()
    back = oracle.q8_decode_blocks(comp, e, oracle.KV_FP16).view(np.float16).astype(np.float32)
    ref = vals.astype(np.float32)
    steps = comp[:, e:].view(np.float32).reshape(3, -1, 2)[..., 1]
    # half a step, then the fp16 storage rounding (half an fp16 ulp)
    bound = np.repeat(steps, 64, axis=1) / 2 + (np.abs(ref) + np.repeat(steps, 64, axis=1)) * 2.0 ** -11 + 2.0 ** -24
    assert np.all(np.abs(back - ref) <= bound)
