"""CPU ORACLE -- test infrastructure, not part of the product.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this package. The product library (``paper_2609_01338_gb300``)
never imports, links or runs it, and the two share no code: the only common
dependency is the input generator in ``synth/``.

``oracle.c`` is a plain fp32 decoder forward over an explicit, contiguous KV
state (see its header for the equations and rounding points); this module
compiles it with gcc/OpenMP and wraps it with ctypes.  ``state_model.py``
is a plain-Python model of the residency state machine (resident / swapped /
dropped blocks) that the library's block bookkeeping is checked against.

Parity status: every function here is pinned by ``tests/test_oracle_pins.py``
(float64 brute force, closed forms, invariants) except where a docstring says
"parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

KV_BF16, KV_FP16, KV_F32 = 0, 1, 2


def build(force: bool = False) -> str:
    src = os.path.join(_HERE, "oracle.c")
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(src)):
        return _LIB_PATH
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    # -ffp-contract=off: no fused multiply-add, so every product and sum is a
    # separately rounded fp32 operation on x86-64 and aarch64 alike.
    subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                    "-fopenmp", "-o", tmp, src, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Shape(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn_dim", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rope_theta", ctypes.c_float),
                ("rms_eps", ctypes.c_float), ("kv_dtype", ctypes.c_int32)]


class _Layer(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down", "attn_norm", "ffn_norm")]


def lib():
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            vp, i64, i32, f32, dbl = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32,
                                      ctypes.c_float, ctypes.c_double)
            L.orc_forward.restype = ctypes.c_int
            L.orc_forward.argtypes = [ctypes.POINTER(_Shape), vp, vp, vp, ctypes.POINTER(_Layer),
                                      vp, vp, i64, vp, vp, i64, vp, vp]
            L.orc_rmsnorm.argtypes = [vp, vp, i64, i32, f32, vp]
            L.orc_linear.argtypes = [vp, vp, i64, i32, i32, vp]
            L.orc_swiglu.argtypes = [vp, vp, i64, vp]
            L.orc_rope.argtypes = [vp, vp, i64, i32, i32, dbl]
            L.orc_rope_table.argtypes = [i64, i32, dbl, vp, vp]
            L.orc_attention.argtypes = [vp, vp, i64, i32, i32, i32, vp, vp, i64, vp]
            L.orc_round_kv_array.argtypes = [vp, i64, i32, vp]
            L.orc_f32_to_f16_array.argtypes = [vp, i64, vp]
            L.orc_f32_to_bf16_array.argtypes = [vp, i64, vp]
            L.orc_q8_encode.argtypes = [vp, i64, vp, vp, vp]
            L.orc_q8_decode.argtypes = [vp, vp, vp, i64, vp]
            L.orc_num_threads.restype = ctypes.c_int
            L.orc_set_num_threads.argtypes = [ctypes.c_int]
            _lib = L
    return _lib


def _p(a: np.ndarray) -> int:
    assert a.flags.c_contiguous, "oracle inputs must be C-contiguous"
    return a.ctypes.data


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def num_threads() -> int:
    return lib().orc_num_threads()


def set_num_threads(n: int) -> None:
    """Thread count of later oracle calls (timing only; results do not depend
    on it: each row is computed by one thread in a fixed order)."""
    lib().orc_set_num_threads(int(n))


def shape_struct(shape: dict) -> _Shape:
    return _Shape(shape["n_layers"], shape["d_model"], shape["n_q_heads"], shape["n_kv_heads"],
                  shape["head_dim"], shape["ffn_dim"], shape["vocab"], shape["rope_theta"],
                  shape["rms_eps"], shape["kv_dtype"])


class KVState:
    """Contiguous fp32 KV state [n_layers][max_ctx][n_kv_heads][head_dim]
    holding stored (already rounded) values; NaN marks never-written slots."""

    def __init__(self, shape: dict, max_ctx: int):
        dims = (shape["n_layers"], max_ctx, shape["n_kv_heads"], shape["head_dim"])
        self.k = np.full(dims, np.nan, dtype=np.float32)
        self.v = np.full(dims, np.nan, dtype=np.float32)
        self.max_ctx = max_ctx

    def copy(self) -> "KVState":
        c = KVState.__new__(KVState)
        c.k, c.v, c.max_ctx = self.k.copy(), self.v.copy(), self.max_ctx
        return c


def forward(shape: dict, weights: dict, kv: KVState, tokens, positions, logits: bool = True,
            return_x: bool = False):
    """Run rows (tokens at positions) through the model over `kv` (updated in
    place). Returns the last row's fp32 logits (or None), and the final
    residual stream if return_x."""
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    positions = np.ascontiguousarray(positions, dtype=np.int64)
    n = tokens.shape[0]
    layers = (_Layer * shape["n_layers"])()
    keep = []
    for l, lw in enumerate(weights["layers"]):
        arrs = [np.ascontiguousarray(lw[k]) for k in
                ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")]
        arrs += [_f32(lw["attn_norm"]), _f32(lw["ffn_norm"])]
        keep += arrs
        layers[l] = _Layer(*[a.ctypes.data for a in arrs])
    emb = np.ascontiguousarray(weights["embed"])
    lm = np.ascontiguousarray(weights["lm_head"])
    fn = _f32(weights["final_norm"])
    out = np.empty(shape["vocab"], dtype=np.float32) if logits and n > 0 else None
    xo = np.empty((n, shape["d_model"]), dtype=np.float32) if return_x else None
    s = shape_struct(shape)
    rc = lib().orc_forward(ctypes.byref(s), _p(emb), _p(lm), _p(fn), layers, _p(kv.k), _p(kv.v),
                           kv.max_ctx, _p(tokens), _p(positions), n,
                           _p(out) if out is not None else None,
                           _p(xo) if xo is not None else None)
    if rc != 0:
        raise ValueError("oracle forward rejected its arguments")
    del keep
    return (out, xo) if return_x else out


def prefill(shape: dict, weights: dict, kv: KVState, tokens, start: int, logits: bool = True):
    """Prefill consecutive tokens at positions start.. (a chunk of a context)."""
    tokens = np.asarray(tokens, dtype=np.int32)
    pos = np.arange(start, start + tokens.shape[0], dtype=np.int64)
    return forward(shape, weights, kv, tokens, pos, logits)


# ---- single operations --------------------------------------------------

def rmsnorm(x, g, eps):
    x = _f32(x); g = _f32(g)
    n, d = x.reshape(-1, x.shape[-1]).shape
    y = np.empty_like(x)
    lib().orc_rmsnorm(_p(x), _p(g), n, d, eps, _p(y))
    return y


def linear(x, w_bits):
    """x[n][n_in] fp32 times bf16 W[n_out][n_in]^T."""
    x = _f32(x); w = np.ascontiguousarray(w_bits, dtype=np.uint16)
    n, k = x.shape
    y = np.empty((n, w.shape[0]), dtype=np.float32)
    lib().orc_linear(_p(x), _p(w), n, k, w.shape[0], _p(y))
    return y


def swiglu(g, u):
    g = _f32(g); u = _f32(u)
    y = np.empty_like(g)
    lib().orc_swiglu(_p(g), _p(u), g.size, _p(y))
    return y


def rope(x, positions, theta):
    """x[n][n_heads][hd] rotated (copy)."""
    x = _f32(x).copy()
    pos = np.ascontiguousarray(positions, dtype=np.int64)
    lib().orc_rope(_p(x), _p(pos), x.shape[0], x.shape[1], x.shape[2], theta)
    return x


def rope_table(n_pos, hd, theta):
    c = np.empty((n_pos, hd // 2), dtype=np.float32)
    s = np.empty((n_pos, hd // 2), dtype=np.float32)
    lib().orc_rope_table(n_pos, hd, theta, _p(c), _p(s))
    return c, s


def attention(q, positions, k, v):
    """q[n][hq][hd] at positions over k/v[ctx][hkv][hd] -> [n][hq][hd]."""
    q = _f32(q); k = _f32(k); v = _f32(v)
    pos = np.ascontiguousarray(positions, dtype=np.int64)
    n, hq, hd = q.shape
    ctx, hkv, _ = k.shape
    out = np.empty_like(q)
    lib().orc_attention(_p(q), _p(pos), n, hq, hkv, hd, _p(k), _p(v), ctx, _p(out))
    return out


def round_kv(x, kv_dtype):
    x = _f32(x)
    y = np.empty_like(x)
    lib().orc_round_kv_array(_p(x), x.size, kv_dtype, _p(y))
    return y


def to_f16_bits(x):
    x = _f32(x); y = np.empty(x.shape, dtype=np.uint16)
    lib().orc_f32_to_f16_array(_p(x), x.size, _p(y))
    return y


def to_bf16_bits(x):
    x = _f32(x); y = np.empty(x.shape, dtype=np.uint16)
    lib().orc_f32_to_bf16_array(_p(x), x.size, _p(y))
    return y


# ---- 8-bit swap codec (oracle.c: orc_q8_encode / orc_q8_decode) -------------

Q8_GROUP = 64


def q8_encode(x):
    """Groups of 64 along the last axis -> (codes uint8, min fp32, step fp32)."""
    x = _f32(x)
    assert x.shape[-1] % Q8_GROUP == 0
    g = x.size // Q8_GROUP
    codes = np.empty(x.shape, np.uint8)
    mn = np.empty(x.shape[:-1] + (x.shape[-1] // Q8_GROUP,), np.float32)
    st = np.empty_like(mn)
    lib().orc_q8_encode(_p(x), g, _p(codes), _p(mn), _p(st))
    return codes, mn, st


def q8_decode(codes, mn, step):
    codes = np.ascontiguousarray(codes, np.uint8)
    mn, step = _f32(mn), _f32(step)
    out = np.empty(codes.shape, np.float32)
    lib().orc_q8_decode(_p(codes), _p(mn), _p(step), codes.size // Q8_GROUP, _p(out))
    return out


def q8_block_bytes(hkv: int, hd: int) -> int:
    """Compressed size of one KV block: the codes, then (min, step) per group."""
    e = 2 * hkv * 16 * hd
    return e + 8 * (e // Q8_GROUP)


def q8_encode_blocks(blocks_f16_bits):
    """KV blocks [n][2*hkv*16*hd] of fp16 bits -> compressed bytes [n][q8_block_bytes]:
    the codes in the block's element order, then fp32 (min, step) pairs in group order."""
    b = np.ascontiguousarray(blocks_f16_bits, np.uint16)
    n, e = b.shape
    x = b.view(np.float16).astype(np.float32).reshape(n, e // Q8_GROUP, Q8_GROUP)
    codes, mn, st = q8_encode(x)
    params = np.stack([mn, st], axis=-1).astype(np.float32).reshape(n, -1)
    return np.concatenate([codes.reshape(n, e), params.view(np.uint8)], axis=1)


def q8_decode_blocks(comp, e: int, kv_dtype: int):
    """Compressed blocks -> fp16 bits [n][e] of the values rounded to the KV type."""
    c = np.ascontiguousarray(comp, np.uint8)
    n = c.shape[0]
    codes = c[:, :e].reshape(n, e // Q8_GROUP, Q8_GROUP)
    params = np.ascontiguousarray(c[:, e:]).view(np.float32).reshape(n, e // Q8_GROUP, 2)
    y = q8_decode(codes, params[..., 0], params[..., 1]).reshape(n, e)
    return to_f16_bits(round_kv(y, kv_dtype))
