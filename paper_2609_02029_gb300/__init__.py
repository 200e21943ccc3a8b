"""Per-head-window KV cache attention for GB300 (HeadWiseKV grouped-cache hot path).

Thin ctypes binding over ``libhwkv.so`` (C ABI in ``include/hwkv.h``). Every
function here has the name of the C entry point it calls and only marshals
arguments: device pointers may be passed as integers or as CUDA tensors
(their ``data_ptr()``), streams as integers or ``torch.cuda.Stream``. All
computation happens in the library's CUDA kernels; if the library is missing
the import fails -- there is no fallback.
"""
import ctypes
import os
import re

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libhwkv.so")
HEADER = os.path.join(os.path.dirname(_HERE), "include", "hwkv.h")

HWKV_OK, HWKV_EINVAL, HWKV_ENOMEM, HWKV_ECAPACITY = 0, 1, 2, 3
HWKV_ECUDA, HWKV_EKERNEL, HWKV_EUNSUPPORTED, HWKV_ETRACE = 4, 5, 6, 7
HWKV_WINDOW_FULL = 0
HWKV_KV_BF16, HWKV_KV_FP8_E4M3 = 0, 1
STATUS_NAMES = {0: "HWKV_OK", 1: "HWKV_EINVAL", 2: "HWKV_ENOMEM", 3: "HWKV_ECAPACITY",
                4: "HWKV_ECUDA", 5: "HWKV_EKERNEL", 6: "HWKV_EUNSUPPORTED", 7: "HWKV_ETRACE"}


class HwkvError(RuntimeError):
    def __init__(self, status, message):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), message))
        self.status = status


class hwkv_policy(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("batch", ctypes.c_int32), ("kv_format", ctypes.c_int32),
                ("max_ctx", ctypes.c_int64), ("windows", ctypes.POINTER(ctypes.c_int64)),
                ("sinks", ctypes.POINTER(ctypes.c_int64))]


def make_policy(n_layers, n_kv_heads, n_q_heads, head_dim, batch, max_ctx, windows,
                kv_format=HWKV_KV_BF16, sinks=None):
    """hwkv_policy with its windows array ([n_layers * n_kv_heads] int64, 0 = full)
    and optional sink counts (same shape) kept alive on the returned object."""
    w = np.ascontiguousarray(np.asarray(windows, dtype=np.int64).ravel())
    sk = None if sinks is None else np.ascontiguousarray(np.asarray(sinks, dtype=np.int64).ravel())
    pol = hwkv_policy(n_layers, n_kv_heads, n_q_heads, head_dim, batch, kv_format, max_ctx,
                      w.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                      None if sk is None else sk.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)))
    pol._windows_keepalive = w
    pol._sinks_keepalive = sk
    return pol


class hwkv_calib_desc(ctypes.Structure):
    _fields_ = [("n_seq", ctypes.c_int32), ("n_pos", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("n_windows", ctypes.c_int32),
                ("T", ctypes.c_int64), ("windows", ctypes.POINTER(ctypes.c_int64)),
                ("positions", ctypes.POINTER(ctypes.c_int64))]


def make_calib_desc(n_seq, n_pos, n_kv_heads, n_q_heads, head_dim, T, windows, positions):
    """hwkv_calib_desc with its windows [K] and positions [n_seq, n_pos] kept alive."""
    w = np.ascontiguousarray(np.asarray(windows, dtype=np.int64).ravel())
    pos = np.ascontiguousarray(np.asarray(positions, dtype=np.int64).ravel())
    d = hwkv_calib_desc(n_seq, n_pos, n_kv_heads, n_q_heads, head_dim, len(w), T,
                        w.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)),
                        pos.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)))
    d._keepalive = (w, pos)
    return d


_lib = None
_vp, _i32, _i64, _u64p = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.POINTER(ctypes.c_uint64)


def lib():
    """The loaded libhwkv.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError("libhwkv.so not built: run `python -c 'import __graft_entry__ as g; "
                              "g.build()'` (needs nvcc for sm_103a)")
        L = ctypes.CDLL(LIB_PATH)
        pp = ctypes.POINTER(hwkv_policy)
        sig = {
            "hwkv_required_bytes": [pp, ctypes.POINTER(ctypes.c_size_t)],
            "hwkv_alloc": [pp, _vp, ctypes.c_size_t, _vp, ctypes.POINTER(_vp)],
            "hwkv_free": [_vp],
            "hwkv_append": [_vp, _i32, _vp, _vp, _i64, _vp],
            "hwkv_prefill": [_vp, _i32, _vp, _vp, _vp, _i64, ctypes.c_float, _vp, _vp],
            "hwkv_decode_attn": [_vp, _i32, _vp, ctypes.c_float, _vp, _vp],
            "hwkv_decode_attn_static": [_vp, _i32, _vp, ctypes.c_float, _vp, _vp],
            "hwkv_decode_static_scratch_bytes": [pp, _i32, ctypes.POINTER(ctypes.c_size_t)],
            "hwkv_decode_step": [_vp, _i32, _vp, _vp, _vp, ctypes.c_float, _vp, _vp],
            "hwkv_decode_step_graph": [_vp, _i32, _vp, _vp, _vp, ctypes.c_float, _vp, _vp],
            "hwkv_append_rows": [_vp, _i32, _i32, _i32, _vp, _vp, _i64, _vp],
            "hwkv_prefill_rows": [_vp, _i32, _i32, _i32, _vp, _vp, _vp, _i64, ctypes.c_float,
                                  _vp, _vp],
            "hwkv_sync_lens": [_vp, _vp],
            "hwkv_reset_rows": [_vp, _i32, _i32, _i32, _vp],
            "hwkv_row_len": [_vp, _i32, _i32, ctypes.POINTER(_i64)],
            "hwkv_residency_bytes": [_vp, _i32, _u64p],
            "hwkv_allocated_ring_bytes": [_vp, _i32, _u64p],
            "hwkv_seq_len": [_vp, _i32, ctypes.POINTER(_i64)],
            "hwkv_ring_capacity": [_vp, _i32, _i32, ctypes.POINTER(_i64)],
            "hwkv_debug_copy_ring": [_vp, _i32, _i32, _i32, _vp, _vp],
            "hwkv_debug_copy_scales": [_vp, _i32, _i32, _i32, _vp, _vp],
            "hwkv_sync_check": [_vp],
            "hwkv_debug_wait_probe": [_vp, _i64, _vp],
            "hwkv_calib_workspace_bytes": [ctypes.POINTER(hwkv_calib_desc),
                                           ctypes.POINTER(ctypes.c_size_t)],
            "hwkv_calib_scores": [ctypes.POINTER(hwkv_calib_desc), _vp, _vp, _vp, ctypes.c_float,
                                  _vp, ctypes.c_size_t, _vp, _vp, _vp],
            "hwkv_calib_select": [_vp, _i32, _vp, _i32, _i64, ctypes.c_double, _vp],
            "hwkv_calib_trace_check": [ctypes.POINTER(hwkv_calib_desc), _vp, _vp, _vp,
                                       ctypes.c_float, _vp, ctypes.c_double, _vp, ctypes.c_size_t,
                                       ctypes.POINTER(ctypes.c_double), _vp, _vp],
            "hwkv_budget_select": [_vp, _vp, _i32, ctypes.c_double, ctypes.POINTER(_i32)],
            "hwkv_policy_save": [ctypes.c_char_p, ctypes.c_char_p, ctypes.c_uint64, _i32, _i32, _vp],
            "hwkv_policy_load": [ctypes.c_char_p, ctypes.c_char_p, ctypes.c_size_t,
                                 ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(_i32),
                                 ctypes.POINTER(_i32), _vp, ctypes.c_size_t],
        }
        for name, args in sig.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        L.hwkv_last_error.argtypes = []
        L.hwkv_last_error.restype = ctypes.c_char_p
        _lib = L
    return _lib


def declared_symbols():
    """Entry points declared in include/hwkv.h."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"HWKV_API\s+[\w\s\*]*?\b(hwkv_\w+)\s*\(", text)))


def hwkv_last_error():
    return lib().hwkv_last_error().decode()


def _check(status):
    if status != HWKV_OK:
        raise HwkvError(status, hwkv_last_error())


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_cuda:
            raise ValueError("expected a CUDA tensor")
        if not x.is_contiguous():
            raise ValueError("expected a contiguous tensor")
        return x.data_ptr()
    raise TypeError("expected a device pointer or CUDA tensor, got %r" % type(x))


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def hwkv_required_bytes(policy):
    n = ctypes.c_size_t(0)
    _check(lib().hwkv_required_bytes(ctypes.byref(policy), ctypes.byref(n)))
    return n.value


def hwkv_alloc(policy, dev_arena=None, arena_bytes=0, stream=None):
    """Returns the opaque cache handle (ctypes.c_void_p)."""
    out = _vp()
    _check(lib().hwkv_alloc(ctypes.byref(policy), _ptr(dev_arena), arena_bytes, _stream(stream),
                            ctypes.byref(out)))
    return out


def hwkv_free(cache):
    _check(lib().hwkv_free(cache))


def hwkv_append(cache, layer, k, v, n, stream=None):
    _check(lib().hwkv_append(cache, layer, _ptr(k), _ptr(v), n, _stream(stream)))


def hwkv_prefill(cache, layer, q, k, v, n, scale, out, stream=None):
    _check(lib().hwkv_prefill(cache, layer, _ptr(q), _ptr(k), _ptr(v), n, scale, _ptr(out),
                              _stream(stream)))


def hwkv_decode_attn(cache, layer, q, scale, out, stream=None):
    _check(lib().hwkv_decode_attn(cache, layer, _ptr(q), scale, _ptr(out), _stream(stream)))


def hwkv_decode_step(cache, layer, q, k_new, v_new, scale, out, stream=None):
    _check(lib().hwkv_decode_step(cache, layer, _ptr(q), _ptr(k_new), _ptr(v_new), scale,
                                  _ptr(out), _stream(stream)))


def hwkv_decode_step_graph(cache, layer, q, k_new, v_new, scale, out, stream=None):
    _check(lib().hwkv_decode_step_graph(cache, layer, _ptr(q), _ptr(k_new), _ptr(v_new), scale,
                                        _ptr(out), _stream(stream)))


def hwkv_append_rows(cache, layer, row0, n_rows, k, v, n, stream=None):
    _check(lib().hwkv_append_rows(cache, layer, row0, n_rows, _ptr(k), _ptr(v), n,
                                  _stream(stream)))


def hwkv_prefill_rows(cache, layer, row0, n_rows, q, k, v, n, scale, out, stream=None):
    _check(lib().hwkv_prefill_rows(cache, layer, row0, n_rows, _ptr(q), _ptr(k), _ptr(v), n,
                                   scale, _ptr(out), _stream(stream)))


def hwkv_sync_lens(cache, stream=None):
    _check(lib().hwkv_sync_lens(cache, _stream(stream)))


def hwkv_reset_rows(cache, row0, n_rows, idle=False, stream=None):
    _check(lib().hwkv_reset_rows(cache, row0, n_rows, 1 if idle else 0, _stream(stream)))


def hwkv_row_len(cache, layer, row):
    v = ctypes.c_int64(0)
    _check(lib().hwkv_row_len(cache, layer, row, ctypes.byref(v)))
    return v.value


def hwkv_decode_attn_static(cache, layer, q, scale, out, stream=None):
    _check(lib().hwkv_decode_attn_static(cache, layer, _ptr(q), scale, _ptr(out),
                                         _stream(stream)))


def hwkv_decode_static_scratch_bytes(policy, num_sms):
    """Static scratch bytes hwkv_decode_attn_static needs (raises HWKV_EINVAL past the array)."""
    n = ctypes.c_size_t(0)
    _check(lib().hwkv_decode_static_scratch_bytes(ctypes.byref(policy), num_sms, ctypes.byref(n)))
    return n.value


def hwkv_residency_bytes(cache, layer=-1):
    v = ctypes.c_uint64(0)
    _check(lib().hwkv_residency_bytes(cache, layer, ctypes.byref(v)))
    return v.value


def hwkv_allocated_ring_bytes(cache, layer=-1):
    v = ctypes.c_uint64(0)
    _check(lib().hwkv_allocated_ring_bytes(cache, layer, ctypes.byref(v)))
    return v.value


def hwkv_seq_len(cache, layer):
    v = ctypes.c_int64(0)
    _check(lib().hwkv_seq_len(cache, layer, ctypes.byref(v)))
    return v.value


def hwkv_ring_capacity(cache, layer, kv_head):
    v = ctypes.c_int64(0)
    _check(lib().hwkv_ring_capacity(cache, layer, kv_head, ctypes.byref(v)))
    return v.value


def hwkv_debug_copy_ring(cache, layer, b, kv_head, head_dim, kv_format=HWKV_KV_BF16):
    """(K, V) of one ring, [cap, head_dim]: uint16 bf16 bits, or uint8 E4M3 codes."""
    cap = hwkv_ring_capacity(cache, layer, kv_head)
    dt = np.uint8 if kv_format == HWKV_KV_FP8_E4M3 else np.uint16
    k = np.zeros((cap, head_dim), dtype=dt)
    v = np.zeros((cap, head_dim), dtype=dt)
    _check(lib().hwkv_debug_copy_ring(cache, layer, b, kv_head,
                                      k.ctypes.data_as(_vp), v.ctypes.data_as(_vp)))
    return k, v


def hwkv_debug_copy_scales(cache, layer, b, kv_head):
    """(K scales, V scales) of one 8-bit ring, float32 [cap]."""
    cap = hwkv_ring_capacity(cache, layer, kv_head)
    k = np.zeros(cap, dtype=np.float32)
    v = np.zeros(cap, dtype=np.float32)
    _check(lib().hwkv_debug_copy_scales(cache, layer, b, kv_head, k.ctypes.data_as(_vp),
                                        v.ctypes.data_as(_vp)))
    return k, v


def hwkv_debug_wait_probe(cache, limit_ns, stream=None):
    _check(lib().hwkv_debug_wait_probe(cache, limit_ns, _stream(stream)))


def hwkv_sync_check(cache):
    _check(lib().hwkv_sync_check(cache))


def hwkv_calib_workspace_bytes(desc):
    n = ctypes.c_size_t(0)
    _check(lib().hwkv_calib_workspace_bytes(ctypes.byref(desc), ctypes.byref(n)))
    return n.value


def hwkv_calib_scores(desc, q, k, v, scale, workspace, ws_bytes, stream=None, with_cos=False):
    """(scores [n_kv_heads, K] float64, cos [N, P, n_q_heads, K] float32 or None)."""
    K = desc.n_windows
    scores = np.zeros((desc.n_kv_heads, K), dtype=np.float64)
    cos = np.zeros((desc.n_seq, desc.n_pos, desc.n_q_heads, K), dtype=np.float32) if with_cos else None
    _check(lib().hwkv_calib_scores(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), scale,
                                   _ptr(workspace), ws_bytes, scores.ctypes.data_as(_vp),
                                   cos.ctypes.data_as(_vp) if cos is not None else None,
                                   _stream(stream)))
    return scores, cos


def hwkv_calib_trace_check(desc, q, k, v, scale, traced, workspace, ws_bytes, threshold=0.99,
                           stream=None):
    """(min cosine, per-row cosines [N, P, n_q_heads]) of the replayed full-window
    outputs against the traced ones; raises HwkvError(HWKV_ETRACE) below threshold."""
    m = ctypes.c_double(0.0)
    per = np.zeros((desc.n_seq, desc.n_pos, desc.n_q_heads), dtype=np.float32)
    _check(lib().hwkv_calib_trace_check(ctypes.byref(desc), _ptr(q), _ptr(k), _ptr(v), scale,
                                        _ptr(traced), threshold, _ptr(workspace), ws_bytes,
                                        ctypes.byref(m), per.ctypes.data_as(_vp), _stream(stream)))
    return m.value, per


def hwkv_calib_select(scores, windows, C, tau):
    s = np.ascontiguousarray(scores, dtype=np.float64)
    w = np.ascontiguousarray(windows, dtype=np.int64)
    H = s.shape[0]
    out = np.zeros(H, dtype=np.int64)
    _check(lib().hwkv_calib_select(s.ctypes.data_as(_vp), H, w.ctypes.data_as(_vp), len(w), C,
                                   tau, out.ctypes.data_as(_vp)))
    return out


def hwkv_budget_select(beta, phi, budget):
    b = np.ascontiguousarray(beta, dtype=np.float64)
    f = np.ascontiguousarray(phi, dtype=np.float64)
    g = ctypes.c_int32(0)
    _check(lib().hwkv_budget_select(b.ctypes.data_as(_vp), f.ctypes.data_as(_vp), len(b), budget,
                                    ctypes.byref(g)))
    return g.value


def hwkv_policy_save(path, artifact, seed, windows):
    """Write a [n_layers, n_kv_heads] window matrix (0 = full) as a policy artifact."""
    w = np.ascontiguousarray(np.asarray(windows, dtype=np.int64))
    L, H = w.shape
    _check(lib().hwkv_policy_save(str(path).encode(), artifact.encode(), seed, L, H,
                                  w.ctypes.data_as(_vp)))


def hwkv_policy_load(path, capacity=1 << 16):
    """(artifact id, seed, windows [n_layers, n_kv_heads] int64)."""
    art = ctypes.create_string_buffer(128)
    seed = ctypes.c_uint64(0)
    L, H = ctypes.c_int32(0), ctypes.c_int32(0)
    out = np.zeros(capacity, dtype=np.int64)
    _check(lib().hwkv_policy_load(str(path).encode(), art, 128, ctypes.byref(seed), ctypes.byref(L),
                                  ctypes.byref(H), out.ctypes.data_as(_vp), capacity))
    return art.value.decode(), seed.value, out[:L.value * H.value].reshape(L.value, H.value).copy()
