"""The residual-add GEMM (the O and down projections) with its last, partial
wave split over k (mzc_k_gemm_split; the prefill runs every O and down
projection this way): against the oracle's linear plus the residual, bit for
bit on repeated runs whatever the flag buffer holds, and within rounding of
the unsplit kernel.  The split applies to the single-CTA kernel (at 257-512
rows, 64- or 128-column tiles) when the k-blocks it saves pay for its ordered
adds: long-K shapes split, ragged K included; the value step's O at that size
does not.  Above 512 rows the paired-SM kernel runs whole 256 x 256 tiles and
nothing splits: those shapes must equal mzc_k_gemm bit for bit."""
import numpy as np
import pytest

import oracle
import paper_2609_01338_gb300 as m
import synth
from tests.gpu_util import bf16_dev, f32_dev, f16_bits, f16_to_f32, bf16_weights_exact_in_f16

pytestmark = pytest.mark.gpu


def _torch():
    import torch
    return torch


def _inputs(mm, nn, kk):
    a = f16_bits(synth.bf16_bits_to_f32(synth.normal_bf16(21, 1, (mm, kk))))
    wb, wh = bf16_weights_exact_in_f16(synth.normal_bf16(21, 2, (nn, kk), sigma=0.05))
    x0 = np.random.default_rng(5).standard_normal((mm, nn)).astype(np.float32)
    return a, wb, wh, x0


CASES = [
    # (m, n, k) split by the single-CTA kernel: 64-column tiles (96 of them)
    (384, 1024, 4096),
    (300, 2048, 8192),
    # ragged K (93.75 k-blocks)
    (500, 1536, 6000),
    # the 3B f = 0.5 hybrid step's down projection (448 rows, 128-column tiles)
    (448, 3072, 8192),
    # its O projection: K 3072 saves too little, no split
    (448, 3072, 3072),
    # above 512 rows: the paired-SM kernel, no split (odd M-tile count, ragged K)
    (1000, 2048, 3000),
    (2576, 3072, 8192),
    (4224, 2048, 8192),
    (2000, 3072, 256),
]
SPLIT = {(384, 1024, 4096), (300, 2048, 8192), (500, 1536, 6000), (448, 3072, 8192)}


@pytest.mark.parametrize("mm,nn,kk", CASES)
def test_split_gemm_matches_the_oracle_and_repeats(mm, nn, kk):
    torch = _torch()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    a, wb, wh, x0 = _inputs(mm, nn, kk)
    ad, wd = bf16_dev(a), bf16_dev(wh)
    flags = torch.zeros(max(sms, 256), dtype=torch.int64, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    outs, ctas = [], []
    # epochs 1, 2 and 2^32 - 1 on the same flags; then flags full of unrelated values
    for epoch, junk in ((1, False), (2, False), (0xFFFFFFFF, False), (7, True)):
        if junk:
            flags.copy_(torch.randint(-2 ** 62, 2 ** 62, flags.shape, dtype=torch.int64))
        out = f32_dev(x0)
        ctas.append(m.mzc_k_gemm_split(ad, wd, out, mm, nn, kk, flags, epoch, status))
        torch.cuda.synchronize()
        outs.append(out.cpu().numpy())
    assert int(status.item()) == 0
    assert len(set(ctas)) == 1
    assert (ctas[0] > 0) == ((mm, nn, kk) in SPLIT)
    assert ctas[0] <= sms
    for o in outs[1:]:
        assert np.array_equal(outs[0], o)
    got = outs[0]
    rows = np.unique(np.linspace(0, mm - 1, min(mm, 256)).astype(int))
    ref = x0[rows] + oracle.linear(f16_to_f32(a[rows]), wb)
    assert np.max(np.abs(got[rows] - ref)) <= 1e-4 * np.max(np.abs(ref))
    # the unsplit kernel: the same sums up to the order of the fp32 adds
    plain = f32_dev(x0)
    m.mzc_k_gemm(ad, wd, plain, mm, nn, kk, 1)
    torch.cuda.synchronize()
    plain = plain.cpu().numpy()
    if ctas[0] == 0:
        assert np.array_equal(plain, got)
    else:
        assert np.max(np.abs(plain - got)) <= 2e-6 * np.max(np.abs(plain))


def test_split_gemm_argument_checks():
    torch = _torch()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    a, wb, wh, x0 = _inputs(600, 1024, 512)
    ad, wd, out = bf16_dev(a), bf16_dev(wh), f32_dev(x0)
    S = m.mzc.status_of
    small = torch.zeros(sms - 1, dtype=torch.int64, device="cuda")
    ok = torch.zeros(sms, dtype=torch.int64, device="cuda")
    args = lambda fl, n_fl, ep: (ad.data_ptr(), wd.data_ptr(), out.data_ptr(), 600, 1024, 512,
                                 fl, n_fl, ep, None, None, None)
    assert S("mzc_k_gemm_split", *args(small.data_ptr(), sms - 1, 1)) == m.MZC_ERR_INVALID
    assert S("mzc_k_gemm_split", *args(ok.data_ptr(), sms, 0)) == m.MZC_ERR_INVALID
    assert S("mzc_k_gemm_split", *args(None, sms, 1)) == m.MZC_ERR_INVALID
    assert S("mzc_k_gemm_split", *args(ok.data_ptr(), sms, 1)) == m.MZC_OK
    torch.cuda.synchronize()
