"""Seeded synthetic inputs: the one module that both the CUDA path's tests and
the CPU oracle draw their inputs from.

It holds no arithmetic of the method. It compiles ``synth.c`` (SplitMix64
counter-based draws, Box-Muller normals, Fisher-Yates choices) with gcc and
exposes numpy-returning wrappers, plus the workload recipes (model shapes,
context/prompt lengths, eviction fractions) in :mod:`synth.workloads`.

Seeds: 0 = weights, 1 = context token ids, 2 = prompt token ids,
3 = choice of scattered evicted blocks.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libsynth.so")
_lock = threading.Lock()
_lib = None

SEED_WEIGHTS = 0
SEED_CONTEXT = 1
SEED_PROMPT = 2
SEED_EVICT = 3
SIGMA = 0.02


def build(force: bool = False) -> str:
    """Compile synth.c into _build/libsynth.so (gcc, OpenMP)."""
    src = os.path.join(_HERE, "synth.c")
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(src)):
        return _LIB_PATH
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared", "-fopenmp",
                    "-o", tmp, src, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            u64, i64, i32, dbl = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            vp = ctypes.c_void_p
            L.synth_key.restype = u64
            L.synth_key.argtypes = [u64, u64]
            L.synth_u64.restype = u64
            L.synth_u64.argtypes = [u64, u64]
            L.synth_normal_bf16.restype = None
            L.synth_normal_bf16.argtypes = [u64, u64, dbl, i64, i64, vp]
            L.synth_normal_f64.restype = None
            L.synth_normal_f64.argtypes = [u64, u64, i64, i64, vp]
            L.synth_tokens.restype = None
            L.synth_tokens.argtypes = [u64, u64, i64, i32, vp]
            L.synth_permutation.restype = None
            L.synth_permutation.argtypes = [u64, u64, i64, vp]
            L.synth_fnv1a.restype = u64
            L.synth_fnv1a.argtypes = [vp, i64]
            _lib = L
    return _lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags.c_contiguous
    return a.ctypes.data


def normal_bf16(seed: int, tensor_id: int, shape, sigma: float = SIGMA, out=None) -> np.ndarray:
    """sigma*N(0,1) samples rounded to bf16, returned as raw uint16 bits."""
    n = int(np.prod(shape))
    if out is None:
        out = np.empty(shape, dtype=np.uint16)
    assert out.dtype == np.uint16 and out.size == n
    lib().synth_normal_bf16(seed, tensor_id, sigma, 0, n, _ptr(out))
    return out


def normal_f64(seed: int, tensor_id: int, begin: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    lib().synth_normal_f64(seed, tensor_id, begin, n, _ptr(out))
    return out


def tokens(seed: int, tensor_id: int, n: int, vocab: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    lib().synth_tokens(seed, tensor_id, n, vocab, _ptr(out))
    return out


def permutation(seed: int, tensor_id: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int64)
    lib().synth_permutation(seed, tensor_id, n, _ptr(out))
    return out


def fnv1a(a: np.ndarray) -> int:
    a = np.ascontiguousarray(a)
    return int(lib().synth_fnv1a(_ptr(a), a.nbytes))


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (no arithmetic: a 16-bit shift)."""
    return (bits.astype(np.uint32) << 16).view(np.float32)


# Tensor ids: embedding 1, LM head 2, per layer (layer+1)<<8 | kind.
KINDS = ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")


def tensor_id(layer: int, kind: str) -> int:
    if layer < 0:
        return {"embed": 1, "lm_head": 2}[kind]
    return ((layer + 1) << 8) | (KINDS.index(kind) + 1)


def layer_shapes(shape) -> dict:
    """Canonical (out_features, in_features) of each per-layer matrix."""
    d, hq, hkv, hd, f = (shape["d_model"], shape["n_q_heads"], shape["n_kv_heads"],
                         shape["head_dim"], shape["ffn_dim"])
    return {"wq": (hq * hd, d), "wk": (hkv * hd, d), "wv": (hkv * hd, d),
            "wo": (d, hq * hd), "w_gate": (f, d), "w_up": (f, d), "w_down": (d, f)}


def model_weights(shape, seed: int = SEED_WEIGHTS) -> dict:
    """All weights of a Llama-style decoder of `shape`, bf16 bits in row-major
    (out_features, in_features) layout; norm gains are ones (fp32)."""
    d, v = shape["d_model"], shape["vocab"]
    w = {"embed": normal_bf16(seed, tensor_id(-1, "embed"), (v, d)),
         "lm_head": normal_bf16(seed, tensor_id(-1, "lm_head"), (v, d)),
         "final_norm": np.ones(d, dtype=np.float32), "layers": []}
    shapes = layer_shapes(shape)
    for l in range(shape["n_layers"]):
        lw = {k: normal_bf16(seed, tensor_id(l, k), shapes[k]) for k in KINDS}
        lw["attn_norm"] = np.ones(d, dtype=np.float32)
        lw["ffn_norm"] = np.ones(d, dtype=np.float32)
        w["layers"].append(lw)
    return w
