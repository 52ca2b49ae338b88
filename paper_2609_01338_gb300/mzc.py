"""ctypes binding of include/mzc.h: the same entry points under the same
names, plus converters from plain dicts / numpy arrays to the C structs.
Argument marshalling only -- no computation happens here."""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = os.path.join(_HERE, "_build", "libmzc.so")
_lock = threading.Lock()
_lib = None

MZC_OK, MZC_ERR_INVALID, MZC_ERR_RANGE, MZC_ERR_STATE = 0, 1, 2, 3
MZC_ERR_OOM, MZC_ERR_CUDA, MZC_ERR_TIMEOUT, MZC_ERR_DEVICE = 4, 5, 6, 7
MZC_ERR_OVERFLOW = 8
MZC_KV_BF16, MZC_KV_FP16 = 0, 1
MZC_CODEC_NONE, MZC_CODEC_Q8 = 0, 1
MZC_COPY, MZC_DROP, MZC_AUTO = 0, 1, 2
MZC_POLICY_COPY, MZC_POLICY_RECOMPUTE, MZC_POLICY_HYBRID = 0, 1, 2
MZC_RESIDENT, MZC_SWAPPED, MZC_DROPPED, MZC_INFLIGHT, MZC_EMPTY = 0, 1, 2, 3, 4
MZC_WAIT_LAYER_EVENT, MZC_WAIT_BLOCK_FLAG = 0, 1
STATUS_NAMES = {0: "OK", 1: "INVALID", 2: "RANGE", 3: "STATE", 4: "OOM", 5: "CUDA",
                6: "TIMEOUT", 7: "DEVICE", 8: "OVERFLOW"}

c_i32, c_i64, c_f32, c_f64, c_vp = (ctypes.c_int32, ctypes.c_int64, ctypes.c_float,
                                    ctypes.c_double, ctypes.c_void_p)


class mzc_model_shape(ctypes.Structure):
    _fields_ = [("n_layers", c_i32), ("d_model", c_i32), ("n_q_heads", c_i32),
                ("n_kv_heads", c_i32), ("head_dim", c_i32), ("ffn_dim", c_i32), ("vocab", c_i32),
                ("rope_theta", c_f32), ("rms_eps", c_f32), ("kv_dtype", c_i32),
                ("block_tokens", c_i32), ("max_ctx", c_i64)]


class mzc_options(ctypes.Structure):
    _fields_ = [("pool_blocks", c_i64), ("max_rows", c_i64), ("host_store_bytes", c_i64),
                ("overlap", c_i32), ("device", c_i32), ("swap_codec", c_i32),
                ("wait_mode", c_i32), ("debug_checks", c_i32), ("read_swapped", c_i32),
                ("compute_stream", c_vp), ("copy_stream", c_vp), ("separate_norm", c_i32),
                ("fused_rope", c_i32)]


class mzc_layer_weights(ctypes.Structure):
    _fields_ = [(n, c_vp) for n in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down",
                                    "attn_norm", "ffn_norm")]


class mzc_weights(ctypes.Structure):
    _fields_ = [("embed", c_vp), ("lm_head", c_vp), ("final_norm", c_vp),
                ("layers", ctypes.POINTER(mzc_layer_weights))]


class mzc_profile(ctypes.Structure):
    _fields_ = [("h2d_gbs", c_f64), ("gemm_us_128", c_f64), ("gemm_us_512", c_f64),
                ("gemm_us_2048", c_f64), ("attn_tflops", c_f64), ("attn_row_ns", c_f64),
                ("attn_prompt_tflops", c_f64),
                ("row_ns", c_f64), ("layer_us", c_f64)]


class mzc_stats_t(ctypes.Structure):
    _fields_ = [("context_tokens", c_i64), ("blocks_resident", c_i64), ("blocks_swapped", c_i64),
                ("blocks_dropped", c_i64), ("pool_free_blocks", c_i64),
                ("bytes_h2d_last", c_i64), ("copies_last", c_i64), ("rows_last", c_i64),
                ("recompute_rows_last", c_i64), ("weights_evicted_layers", c_i32),
                ("reserved", c_i32)]


class mzc_kernel_stat(ctypes.Structure):
    _fields_ = [("launches", c_i64), ("ms", c_f64), ("flops", c_f64), ("bytes", c_f64)]


MZC_K_GEMM, MZC_K_ATTENTION, MZC_K_ROPE_KV, MZC_K_RMSNORM, MZC_K_LM_HEAD, MZC_K_EMBED = range(6)
MZC_K_NCLASS = 6
KERNEL_CLASS_NAMES = ("gemm", "attention", "rope_kv", "rmsnorm", "lm_head", "embed")


class mzc_evict_plan(ctypes.Structure):
    _fields_ = [("t_copy_w", c_f64), ("t_copy_kv", c_f64), ("t_rec_kv", c_f64),
                ("kv_total", c_i64), ("w_total", c_i32), ("w_evicted", c_i32),
                ("kv_copy", c_i64), ("kv_rec", c_i64), ("kv_bytes", c_i64), ("w_bytes", c_i64)]


MZC_STAGE_KV_ONLY, MZC_STAGE_KV_AND_W, MZC_STAGE_W_ONLY, MZC_STAGE_COMP_KV = 1, 2, 3, 4


class mzc_copy_run(ctypes.Structure):
    _fields_ = [("layer", c_i32), ("n_blocks", c_i32), ("host_off", c_i64),
                ("phys_begin", c_i64)]


P = ctypes.POINTER
_SIGS = {
    "mzc_create": [P(mzc_model_shape), P(mzc_options), P(mzc_weights), P(c_vp)],
    "mzc_destroy": [c_vp],
    "mzc_prefill": [c_vp, c_vp, c_i64, c_vp],
    "mzc_evict": [c_vp, c_i32, c_i32, c_i64, c_i64, c_i32],
    "mzc_evict_blocks": [c_vp, c_vp, c_vp, c_i64, c_i32],
    "mzc_evict_weights": [c_vp, c_i32, c_i32],
    "mzc_restore_async": [c_vp],
    "mzc_recompute_tail": [c_vp, c_i64, c_i64],
    "mzc_set_policy": [c_vp, c_i32, P(mzc_profile)],
    "mzc_plan_split": [P(mzc_model_shape), P(mzc_profile), c_i64, c_i64, c_i64, P(c_i64)],
    "mzc_profile_measure": [c_vp, P(mzc_profile)],
    "mzc_truncate": [c_vp, c_i64],
    "mzc_sync": [c_vp],
    "mzc_query": [c_vp, c_i32, c_i64, P(c_i32), P(c_i32)],
    "mzc_read_kv": [c_vp, c_i32, c_i64, c_vp, c_vp],
    "mzc_read_kv_all": [c_vp, c_i64, c_vp, c_vp],
    "mzc_stats": [c_vp, P(mzc_stats_t)],
    "mzc_last_times": [c_vp, c_vp],
    "mzc_set_kernel_timing": [c_vp, c_i32],
    "mzc_kernel_stats": [c_vp, c_i32, P(mzc_kernel_stat)],
    "mzc_state_create": [P(mzc_model_shape), c_i64, c_i64, P(c_vp)],
    "mzc_state_destroy": [c_vp],
    "mzc_state_append": [c_vp, c_i64],
    "mzc_state_evict": [c_vp, c_i32, c_i32, c_i64, c_i64, c_i32],
    "mzc_state_evict_blocks": [c_vp, c_vp, c_vp, c_i64, c_i32],
    "mzc_state_recompute_tail": [c_vp, c_i64, c_i64],
    "mzc_state_plan_restore": [c_vp, P(mzc_copy_run), c_i64, P(c_i64)],
    "mzc_state_complete": [c_vp],
    "mzc_state_truncate": [c_vp, c_i64],
    "mzc_state_query": [c_vp, c_i32, c_i64, P(c_i32), P(c_i32)],
    "mzc_state_counts": [c_vp, P(mzc_stats_t)],
    "mzc_k_rmsnorm": [c_vp, c_vp, c_i64, c_i32, c_f32, c_vp, c_vp],
    "mzc_k_gemm": [c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_i32, c_vp],
    "mzc_k_gemm_split": [c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_vp, c_i64, ctypes.c_uint32, c_vp,
                         c_vp, c_vp],
    "mzc_k_gemm_norm_out": [c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_vp, c_vp, c_vp, c_vp, c_vp],
    "mzc_k_gemm_norm_in": [c_vp, c_vp, c_vp, c_i64, c_i64, c_i64, c_i32, c_vp, c_f32, c_vp, c_vp],
    "mzc_k_swiglu_pack": [c_vp, c_vp, c_i64, c_i64, c_vp],
    "mzc_k_rope_kv_write": [c_vp, c_vp, c_i64, c_i32, c_i32, c_i32, c_vp, c_vp, c_vp, c_i64,
                            c_vp, c_i64, c_i32, c_vp, c_vp, c_vp],
    "mzc_k_attention": [c_vp, c_vp, c_i64, c_i32, c_i32, c_i32, c_vp, c_i64, c_vp, c_i64, c_i32,
                        c_vp, c_i64, c_vp, c_i64, c_vp, c_vp],
    "mzc_k_attention_noalloc": [c_vp, c_vp, c_i64, c_i32, c_i32, c_i32, c_vp, c_i64, c_vp, c_i64,
                                c_i32, c_vp, c_i64, c_vp, c_vp],
    "mzc_k_attention_wait": [c_vp, c_vp, c_i64, c_i32, c_i32, c_i32, c_vp, c_i64, c_vp, c_i64, c_i32,
                             c_vp, c_i64, c_vp, c_i64, c_vp, c_i64, c_vp, c_vp],
    "mzc_k_lm_head": [c_vp, c_vp, c_i32, c_f32, c_vp, c_i64, c_vp, c_vp],
    "mzc_plan_split_ctx": [c_vp, c_i64, c_i64, c_vp],
    "mzc_plan_evict_size": [P(mzc_evict_plan), c_i64, P(c_i64), P(c_i32)],
    "mzc_evict_size": [c_vp, c_i64, P(c_i64), P(c_i32)],
    "mzc_evict_size_plan": [c_vp, P(mzc_evict_plan)],
    "mzc_state_evict_size": [c_vp, P(mzc_evict_plan), c_i64, P(c_i64), P(c_i32)],
    "mzc_k_wait_probe": [c_i32, c_i64, c_vp, c_vp, c_vp],
    "mzc_k_q8_encode": [c_vp, c_vp, c_i64, c_i32, c_i32, c_vp, c_vp],
    "mzc_k_q8_decode": [c_vp, c_i64, c_i32, c_i32, c_vp, c_i64, c_i32, c_vp, c_vp],
    "mzc_k_embed": [c_vp, c_i64, c_vp, c_i32, c_i64, c_vp, c_vp, c_vp],
}
_RESTYPES = {"mzc_last_error": (ctypes.c_char_p, [c_vp]),
             "mzc_k_attention_scratch_bytes": (c_i64, [c_i64, c_i32, c_i32, c_i32, c_i64]),
             "mzc_q8_block_bytes": (c_i64, [c_i32, c_i32])}


def lib_path() -> str:
    return _LIB


def load():
    """Loads libmzc.so; raises if it has not been built (no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB):
                raise RuntimeError(f"libmzc is not built ({_LIB}); run "
                                   "`python -c 'import __graft_entry__ as g; g.build()'`")
            L = ctypes.CDLL(_LIB)
            for name, args in _SIGS.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = ctypes.c_int
            for name, (rt, args) in _RESTYPES.items():
                f = getattr(L, name)
                f.argtypes = args
                f.restype = rt
            _lib = L
    return _lib


class MzcError(RuntimeError):
    def __init__(self, fn, status, msg=""):
        super().__init__(f"{fn} -> {STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


def _call(fn, *args, ctx=None):
    s = getattr(load(), fn)(*args)
    if s != MZC_OK:
        msg = load().mzc_last_error(ctx).decode()
        raise MzcError(fn, s, msg)
    return s


def status_of(fn, *args) -> int:
    """Calls an entry point and returns its status instead of raising."""
    return getattr(load(), fn)(*args)


def _ptr(a):
    if a is None:
        return None
    if isinstance(a, int):
        return a
    if hasattr(a, "data_ptr"):  # torch tensor (host or device)
        return a.data_ptr()
    assert a.flags.c_contiguous
    return a.ctypes.data


def make_shape(shape: dict) -> mzc_model_shape:
    return mzc_model_shape(shape["n_layers"], shape["d_model"], shape["n_q_heads"],
                           shape["n_kv_heads"], shape["head_dim"], shape["ffn_dim"],
                           shape["vocab"], shape["rope_theta"], shape["rms_eps"],
                           shape["kv_dtype"], shape.get("block_tokens", 16), shape["max_ctx"])


def make_weights(weights: dict):
    """C struct over the numpy arrays of `weights` (kept alive by the return)."""
    keep = []

    def arr(a, dt):
        a = np.ascontiguousarray(a, dtype=dt)
        keep.append(a)
        return a.ctypes.data

    n = len(weights["layers"])
    layers = (mzc_layer_weights * n)()
    for i, lw in enumerate(weights["layers"]):
        layers[i] = mzc_layer_weights(
            *[arr(lw[k], np.uint16) for k in ("wq", "wk", "wv", "wo", "w_gate", "w_up", "w_down")],
            arr(lw["attn_norm"], np.float32), arr(lw["ffn_norm"], np.float32))
    keep.append(layers)
    w = mzc_weights(arr(weights["embed"], np.uint16), arr(weights["lm_head"], np.uint16),
                    arr(weights["final_norm"], np.float32), layers)
    return w, keep


# ---- ctx entry points (same names as the C ABI) -------------------------

def mzc_create(shape: dict, weights: dict, pool_blocks=0, max_rows=0, host_store_bytes=0,
               overlap=1, device=0, swap_codec=MZC_CODEC_NONE, wait_mode=MZC_WAIT_LAYER_EVENT,
               debug_checks=0, compute_stream=None, copy_stream=None, read_swapped=0, separate_norm=0,
               fused_rope=0):
    """compute_stream / copy_stream: cudaStream_t handles (ints, e.g. a torch
    stream's cuda_stream) owned by the caller, or None."""
    sh = make_shape(shape)
    opt = mzc_options(pool_blocks, max_rows, host_store_bytes, overlap, device, swap_codec,
                      wait_mode, debug_checks, read_swapped, compute_stream, copy_stream,
                      separate_norm, fused_rope)
    w, keep = make_weights(weights)
    out = c_vp()
    _call("mzc_create", ctypes.byref(sh), ctypes.byref(opt), ctypes.byref(w), ctypes.byref(out))
    del keep
    return out.value


def mzc_destroy(ctx):
    return _call("mzc_destroy", ctx, ctx=ctx)


def mzc_prefill(ctx, tokens, logits_out=None):
    """tokens: int32 host array; logits_out: float32 host array [vocab] or None."""
    tokens = np.ascontiguousarray(tokens, dtype=np.int32)
    return _call("mzc_prefill", ctx, _ptr(tokens) if tokens.size else None, tokens.size,
                 _ptr(logits_out), ctx=ctx)


def mzc_evict(ctx, layer_begin, layer_end, tok_begin, tok_end, mode):
    return _call("mzc_evict", ctx, layer_begin, layer_end, tok_begin, tok_end, mode, ctx=ctx)


def mzc_evict_blocks(ctx, layers, blocks, mode=MZC_COPY):
    layers = np.ascontiguousarray(layers, dtype=np.int32)
    blocks = np.ascontiguousarray(blocks, dtype=np.int64)
    return _call("mzc_evict_blocks", ctx, _ptr(layers), _ptr(blocks), layers.size, mode, ctx=ctx)


def mzc_evict_weights(ctx, layer_begin, layer_end):
    return _call("mzc_evict_weights", ctx, layer_begin, layer_end, ctx=ctx)


def mzc_restore_async(ctx):
    return _call("mzc_restore_async", ctx, ctx=ctx)


def mzc_recompute_tail(ctx, p, n):
    return _call("mzc_recompute_tail", ctx, p, n, ctx=ctx)


def mzc_set_policy(ctx, policy, profile: mzc_profile | None = None):
    return _call("mzc_set_policy", ctx, policy, ctypes.byref(profile) if profile else None, ctx=ctx)


def mzc_plan_split(shape: dict, profile: mzc_profile | None, p, n_ctx, n_prompt) -> int:
    sh = make_shape(shape)
    out = c_i64()
    _call("mzc_plan_split", ctypes.byref(sh), ctypes.byref(profile) if profile else None, p,
          n_ctx, n_prompt, ctypes.byref(out))
    return out.value


def mzc_plan_split_ctx(ctx, p, n_prompt) -> int:
    out = c_i64()
    _call("mzc_plan_split_ctx", ctx, p, n_prompt, ctypes.byref(out), ctx=ctx)
    return out.value


def mzc_profile_measure(ctx) -> mzc_profile:
    p = mzc_profile()
    _call("mzc_profile_measure", ctx, ctypes.byref(p), ctx=ctx)
    return p


def mzc_plan_evict_size(plan: mzc_evict_plan, nbytes):
    """Advances plan's counts (in place) by the eviction policy; returns
    (freed bytes, last stage)."""
    f, st = c_i64(), c_i32()
    _call("mzc_plan_evict_size", ctypes.byref(plan), nbytes, ctypes.byref(f), ctypes.byref(st))
    return f.value, st.value


def mzc_evict_size(ctx, nbytes):
    """evict(size): returns (freed bytes, last stage)."""
    f, st = c_i64(), c_i32()
    _call("mzc_evict_size", ctx, nbytes, ctypes.byref(f), ctypes.byref(st), ctx=ctx)
    return f.value, st.value


def mzc_evict_size_plan(ctx) -> mzc_evict_plan:
    p = mzc_evict_plan()
    _call("mzc_evict_size_plan", ctx, ctypes.byref(p), ctx=ctx)
    return p


def mzc_state_evict_size(state, times: mzc_evict_plan, nbytes):
    f, st = c_i64(), c_i32()
    _call("mzc_state_evict_size", state, ctypes.byref(times), nbytes, ctypes.byref(f), ctypes.byref(st))
    return f.value, st.value


def mzc_truncate(ctx, n_ctx):
    return _call("mzc_truncate", ctx, n_ctx, ctx=ctx)


def mzc_sync(ctx):
    return _call("mzc_sync", ctx, ctx=ctx)


def mzc_query(ctx, layer, block):
    s, p = c_i32(), c_i32()
    _call("mzc_query", ctx, layer, block, ctypes.byref(s), ctypes.byref(p), ctx=ctx)
    return s.value, p.value


def mzc_read_kv(ctx, layer, block, shape: dict):
    n = shape["n_kv_heads"] * 16 * shape["head_dim"]
    k = np.empty(n, np.uint16)
    v = np.empty(n, np.uint16)
    _call("mzc_read_kv", ctx, layer, block, _ptr(k), _ptr(v), ctx=ctx)
    return k, v


def mzc_read_kv_all(ctx, n, shape: dict):
    dims = (shape["n_layers"], n, shape["n_kv_heads"], shape["head_dim"])
    k = np.empty(dims, np.float32)
    v = np.empty(dims, np.float32)
    _call("mzc_read_kv_all", ctx, n, _ptr(k), _ptr(v), ctx=ctx)
    return k, v


def mzc_stats(ctx) -> mzc_stats_t:
    s = mzc_stats_t()
    _call("mzc_stats", ctx, ctypes.byref(s), ctx=ctx)
    return s


def mzc_last_times(ctx):
    """[prefill on the compute stream, restore copies, LM head, device TTFT] in ms."""
    a = np.zeros(4, np.float32)
    _call("mzc_last_times", ctx, _ptr(a), ctx=ctx)
    return a


def mzc_set_kernel_timing(ctx, class_mask: int):
    """Bit c times kernel class c (MZC_K_*); -1 every class; 0 none."""
    return _call("mzc_set_kernel_timing", ctx, int(class_mask), ctx=ctx)


def mzc_kernel_stats(ctx, cls) -> mzc_kernel_stat:
    k = mzc_kernel_stat()
    _call("mzc_kernel_stats", ctx, cls, ctypes.byref(k), ctx=ctx)
    return k


def mzc_last_error(ctx=None) -> str:
    return load().mzc_last_error(ctx).decode()


# ---- host bookkeeping (no device) ----------------------------------------

def mzc_state_create(shape: dict, pool_blocks=0, host_store_bytes=0):
    sh = make_shape(shape)
    out = c_vp()
    _call("mzc_state_create", ctypes.byref(sh), pool_blocks, host_store_bytes, ctypes.byref(out))
    return out.value


def mzc_state_plan_restore(st, cap=1 << 16):
    runs = (mzc_copy_run * cap)()
    n = c_i64()
    _call("mzc_state_plan_restore", st, runs, cap, ctypes.byref(n))
    return [(r.layer, r.n_blocks, r.host_off, r.phys_begin) for r in runs[: n.value]]


def mzc_state_query(st, layer, block):
    s, p = c_i32(), c_i32()
    _call("mzc_state_query", st, layer, block, ctypes.byref(s), ctypes.byref(p))
    return s.value, p.value


def mzc_state_counts(st) -> mzc_stats_t:
    s = mzc_stats_t()
    _call("mzc_state_counts", st, ctypes.byref(s))
    return s


# ---- single kernels (device pointers: ints or torch tensors) -------------

def mzc_k_rmsnorm(x, g, n, d, eps, y, stream=None):
    return _call("mzc_k_rmsnorm", _ptr(x), _ptr(g), n, d, eps, _ptr(y), stream)


def mzc_k_gemm(a, w, out, m, n, k, epilogue, stream=None):
    return _call("mzc_k_gemm", _ptr(a), _ptr(w), _ptr(out), m, n, k, epilogue, stream)


def mzc_k_gemm_split(a, w, out, m, n, k, flags, epoch, status=None, stream=None):
    """Residual-add GEMM with the last wave split over k; returns the number
    of CTAs that shared the split tiles (0 = ran unsplit)."""
    ctas = ctypes.c_int64()
    _call("mzc_k_gemm_split", _ptr(a), _ptr(w), _ptr(out), m, n, k, _ptr(flags), flags.numel(),
          epoch, _ptr(status), ctypes.byref(ctas), stream)
    return ctas.value


def mzc_k_gemm_norm_out(a, w, x, m, n, k, g, h, ss, status=None, stream=None):
    """x += A W^T, also writing h = fp16(x * g) and the per-128-column sums
    of squares ss [m][n / 128] (the producer side of a folded RMSNorm)."""
    return _call("mzc_k_gemm_norm_out", _ptr(a), _ptr(w), _ptr(x), m, n, k, _ptr(g), _ptr(h), _ptr(ss),
                 _ptr(status), stream)


def mzc_k_gemm_norm_in(h, w, out, m, n, k, epilogue, ss, eps, status=None, stream=None):
    """Epilogue 0 / 2 of mzc_k_gemm on diag(rstd) (h W^T), rstd from ss."""
    return _call("mzc_k_gemm_norm_in", _ptr(h), _ptr(w), _ptr(out), m, n, k, epilogue, _ptr(ss), eps,
                 _ptr(status), stream)


def mzc_k_swiglu_pack(gate, up):
    gate = np.ascontiguousarray(gate, np.uint16)
    up = np.ascontiguousarray(up, np.uint16)
    out = np.empty((2 * gate.shape[0], gate.shape[1]), np.uint16)
    _call("mzc_k_swiglu_pack", _ptr(gate), _ptr(up), gate.shape[0], gate.shape[1], _ptr(out))
    return out


def mzc_k_rope_kv_write(qkv, pos, n, hq, hkv, hd, cos_t, sin_t, table, n_logical, pool,
                        pool_blocks, kv_dtype, q_out, status, stream=None):
    return _call("mzc_k_rope_kv_write", _ptr(qkv), _ptr(pos), n, hq, hkv, hd, _ptr(cos_t),
                 _ptr(sin_t), _ptr(table), n_logical, _ptr(pool), pool_blocks, kv_dtype,
                 _ptr(q_out), _ptr(status), stream)


def mzc_k_attention_scratch_bytes(n, hq, hkv, hd, max_keys) -> int:
    return load().mzc_k_attention_scratch_bytes(n, hq, hkv, hd, max_keys)


def mzc_k_attention(q, pos, n, hq, hkv, hd, table, n_logical, pool, pool_blocks, kv_dtype, out,
                    max_keys, scratch, scratch_bytes, status, stream=None):
    return _call("mzc_k_attention", _ptr(q), _ptr(pos), n, hq, hkv, hd, _ptr(table), n_logical,
                 _ptr(pool), pool_blocks, kv_dtype, _ptr(out), max_keys, _ptr(scratch),
                 scratch_bytes, _ptr(status), stream)


def mzc_k_attention_wait(q, pos, n, hq, hkv, hd, table, n_logical, pool, pool_blocks, kv_dtype, out,
                         max_keys, scratch, scratch_bytes, block_flags, flag_wait_cycles, status,
                         stream=None):
    """Attention that waits (bounded) for each block's residency flag."""
    return _call("mzc_k_attention_wait", _ptr(q), _ptr(pos), n, hq, hkv, hd, _ptr(table), n_logical,
                 _ptr(pool), pool_blocks, kv_dtype, _ptr(out), max_keys, _ptr(scratch),
                 scratch_bytes, _ptr(block_flags), flag_wait_cycles, _ptr(status), stream)


MZC_ATTENTION_NOALLOC_SCRATCH_BYTES = 8 << 20


def mzc_k_attention_noalloc(q, pos, n, hq, hkv, hd, table, n_logical, pool, pool_blocks,
                            kv_dtype, out, max_keys, status, stream=None):
    """Attention with the library's fixed split-KV array: allocates nothing."""
    return _call("mzc_k_attention_noalloc", _ptr(q), _ptr(pos), n, hq, hkv, hd, _ptr(table),
                 n_logical, _ptr(pool), pool_blocks, kv_dtype, _ptr(out), max_keys,
                 _ptr(status), stream)


def mzc_k_lm_head(x_row, g, d, eps, w, vocab, logits, stream=None):
    return _call("mzc_k_lm_head", _ptr(x_row), _ptr(g), d, eps, _ptr(w), vocab, _ptr(logits), stream)


def mzc_k_embed(tokens, n, embed, d, vocab, x, status, stream=None):
    return _call("mzc_k_embed", _ptr(tokens), n, _ptr(embed), d, vocab, _ptr(x), _ptr(status), stream)


def mzc_q8_block_bytes(hkv, hd) -> int:
    return load().mzc_q8_block_bytes(hkv, hd)


def mzc_k_q8_encode(pool, phys, n, hkv, hd, out, stream=None):
    return _call("mzc_k_q8_encode", _ptr(pool), _ptr(phys), n, hkv, hd, _ptr(out), stream)


def mzc_k_q8_decode(inp, n, hkv, hd, phys, phys_begin, kv_dtype, pool, stream=None):
    return _call("mzc_k_q8_decode", _ptr(inp), n, hkv, hd, _ptr(phys), phys_begin, kv_dtype,
                 _ptr(pool), stream)


def mzc_k_wait_probe(arrive, limit_cycles, status, completed, stream=None):
    return _call("mzc_k_wait_probe", arrive, limit_cycles, _ptr(status), _ptr(completed), stream)
