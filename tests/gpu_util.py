"""Helpers for the GPU tests: torch is used for device memory only."""
import numpy as np

import synth


def bf16_dev(bits: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def f32_dev(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).cuda()


def i32_dev(a: np.ndarray):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).cuda()


def to_np_u16(t) -> np.ndarray:
    return t.cpu().numpy().view(np.uint16)


def kv_bits_to_f32(bits: np.ndarray, kv_dtype: int = 1) -> np.ndarray:
    """Decode pool / q bits: the pool holds fp16-encoded values for both KV
    types (bf16-rounded values when kv_dtype is bf16)."""
    return np.asarray(bits).view(np.float16).astype(np.float32)


def f32_to_kv_bits(x: np.ndarray, kv_dtype: int) -> np.ndarray:
    """Round to the KV precision (bf16 or fp16), then fp16-encode."""
    import oracle
    return oracle.round_kv(np.asarray(x, np.float32), kv_dtype).astype(np.float16).view(np.uint16)


def rel_err(got, ref) -> float:
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.max(np.abs(got - ref)) / max(np.max(np.abs(ref)), 1e-30))


def f16_bits(x: np.ndarray) -> np.ndarray:
    return np.asarray(x, np.float32).astype(np.float16).view(np.uint16)


def f16_to_f32(bits: np.ndarray) -> np.ndarray:
    return np.asarray(bits).view(np.float16).astype(np.float32)


def bf16_weights_exact_in_f16(bits: np.ndarray):
    """bf16 weights with magnitudes below 2^-14 flushed to zero, so that every
    value is exactly representable in fp16 too; returns (bf16 bits, fp16 bits)."""
    f = synth.bf16_bits_to_f32(bits)
    f = np.where(np.abs(f) < 2.0 ** -14, 0.0, f).astype(np.float32)
    import oracle
    b = oracle.to_bf16_bits(f)
    assert np.array_equal(synth.bf16_bits_to_f32(b), f)
    h = f16_bits(f)
    assert np.array_equal(f16_to_f32(h), f)
    return b, h
