"""The shared input generator against an independent numpy restatement of
SplitMix64 / Box-Muller, plus determinism and distribution checks."""
import numpy as np

import synth

M64 = (1 << 64) - 1


def _sm64(x):
    z = (x + 0x9E3779B97F4A7C15) & M64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & M64
    return z ^ (z >> 31)


def _key(seed, tid):
    return _sm64(_sm64(seed) ^ ((tid * 0xD1B54A32D192ED03) & M64))


def test_splitmix_stream_matches_python_restatement():
    for seed, tid in ((0, 1), (3, 257), (123456789, 7)):
        k = _key(seed, tid)
        assert synth.lib().synth_key(seed, tid) == k
        for c in (0, 1, 2, 1000, 2 ** 40 + 5):
            assert synth.lib().synth_u64(k, c) == _sm64((k + c) & M64)


def test_splitmix_published_first_outputs():
    # SplitMix64 with state 0: first output is the finaliser of the golden gamma
    assert _sm64(0) == 0xE220A8397B1DCDAF


def test_normals_match_box_muller_restatement():
    import math
    seed, tid = 0, (3 << 8) | 2
    z = synth.normal_f64(seed, tid, 0, 64)
    k = _key(seed, tid)
    for e in range(64):
        j = e >> 1
        r1, r2 = _sm64((k + 2 * j) & M64), _sm64((k + 2 * j + 1) & M64)
        u1 = ((r1 >> 11) + 1) * 2.0 ** -53
        u2 = (r2 >> 11) * 2.0 ** -53
        rad = math.sqrt(-2.0 * math.log(u1))
        want = rad * (math.sin(2 * math.pi * u2) if e & 1 else math.cos(2 * math.pi * u2))
        assert abs(z[e] - want) < 1e-12


def test_bf16_weights_are_rounded_samples_and_slice_independent():
    import torch
    z = synth.normal_f64(0, 5, 0, 4096)
    bits = synth.normal_bf16(0, 5, (4096,))
    want = torch.from_numpy((0.02 * z).astype(np.float32)).to(torch.bfloat16)
    assert np.array_equal(bits, want.view(torch.int16).numpy().view(np.uint16))
    f = synth.bf16_bits_to_f32(synth.normal_bf16(0, 6, (1 << 20,)))
    assert abs(f.mean()) < 1e-4 and abs(f.std() - 0.02) < 1e-4


def test_tokens_uniform_and_permutation_valid():
    t = synth.tokens(1, 0, 200000, 1024)
    assert t.min() >= 0 and t.max() < 1024
    counts = np.bincount(t, minlength=1024)
    assert counts.min() > 120 and counts.max() < 280
    p = synth.permutation(3, 0, 1000)
    assert np.array_equal(np.sort(p), np.arange(1000))
    assert not np.array_equal(p, np.arange(1000))
    assert np.array_equal(p, synth.permutation(3, 0, 1000))
