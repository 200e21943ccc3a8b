"""CPU fp64 oracle for the per-head-window KV path -- TEST INFRASTRUCTURE.

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg
may import this package. It shares no code with the CUDA library; its only
shared dependency is the seeded input generator (``hwkv_gen``).
Each function states the passage of the HeadWiseKV paper it follows; the C
source ``hwkv_oracle.c`` holds the arithmetic.
"""
import ctypes

import numpy as np

from . import build as _build
from hwkv_gen import GenDesc

FULL = 0
_lib = None

_i64p = ctypes.POINTER(ctypes.c_int64)
_f64p = ctypes.POINTER(ctypes.c_double)


def lib():
    global _lib
    if _lib is None:
        _build.build()
        L = ctypes.CDLL(_build.LIB)
        L.oracle_threads.restype = ctypes.c_int
        L.oracle_set_threads.argtypes = [ctypes.c_int]
        L.oracle_window_lo.argtypes = [ctypes.c_int64, ctypes.c_int64]
        L.oracle_window_lo.restype = ctypes.c_int64
        L.oracle_attend.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_int64, ctypes.c_int64,
                                                            ctypes.c_double, ctypes.c_void_p,
                                                            ctypes.c_void_p]
        L.oracle_attend.restype = ctypes.c_double
        L.oracle_window_attention_bf16.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
            ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_window_attention_bf16.restype = ctypes.c_int
        L.oracle_window_attention_gen.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int64,
            ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_window_attention_gen.restype = ctypes.c_int
        L.oracle_ring_positions.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
        L.oracle_ring_positions.restype = ctypes.c_int
        L.oracle_ring_expected_gen.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_uint32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
        L.oracle_ring_expected_gen.restype = ctypes.c_int
        L.oracle_retained_tokens.argtypes = [ctypes.c_int64, ctypes.c_int64]
        L.oracle_retained_tokens.restype = ctypes.c_int64
        L.oracle_nominal_storage.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                                             ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                             ctypes.c_int64, ctypes.c_int64]
        L.oracle_nominal_storage.restype = ctypes.c_uint64
        L.oracle_normalized_rate.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
                                             ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                             ctypes.c_int64]
        L.oracle_normalized_rate.restype = ctypes.c_double
        L.oracle_cos_eval.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                      ctypes.c_double]
        L.oracle_cos_eval.restype = ctypes.c_double
        L.oracle_conditional_similarity_bf16.argtypes = [
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p,
            ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_double,
            ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_conditional_similarity_bf16.restype = ctypes.c_int
        L.oracle_select_window.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                           ctypes.c_int64, ctypes.c_double]
        L.oracle_select_window.restype = ctypes.c_int64
        L.oracle_budget_select.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                           ctypes.c_double]
        L.oracle_budget_select.restype = ctypes.c_int64
        L.oracle_e4m3_decode.argtypes = [ctypes.c_uint8]
        L.oracle_e4m3_decode.restype = ctypes.c_double
        L.oracle_e4m3_encode.argtypes = [ctypes.c_float]
        L.oracle_e4m3_encode.restype = ctypes.c_uint8
        L.oracle_quantize_row_e4m3.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
                                               ctypes.c_void_p]
        L.oracle_quantize_row_e4m3.restype = ctypes.c_int
        L.oracle_window_attention_fp8.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64,
            ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_window_attention_fp8.restype = ctypes.c_int
        L.oracle_ring_expected_fp8_gen.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_uint32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p,
            ctypes.c_void_p]
        L.oracle_ring_expected_fp8_gen.restype = ctypes.c_int
        L.oracle_sink_visible.argtypes = [ctypes.c_int64] * 4
        L.oracle_sink_visible.restype = ctypes.c_int
        L.oracle_sink_positions.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                            ctypes.c_void_p]
        L.oracle_sink_positions.restype = ctypes.c_int64
        L.oracle_sink_attention_gen.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int64,
            ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_sink_attention_gen.restype = ctypes.c_int
        L.oracle_sink_attention_bf16.argtypes = [
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64, ctypes.c_void_p,
            ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
            ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p]
        L.oracle_sink_attention_bf16.restype = ctypes.c_int
        L.oracle_sink_ring_positions.argtypes = [ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
                                                 ctypes.c_void_p]
        L.oracle_sink_ring_positions.restype = ctypes.c_int
        L.oracle_sink_ring_expected_gen.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_uint32, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, ctypes.c_int64,
            ctypes.c_void_p]
        L.oracle_sink_ring_expected_gen.restype = ctypes.c_int
        L.oracle_sink_retained_tokens.argtypes = [ctypes.c_int64] * 3
        L.oracle_sink_retained_tokens.restype = ctypes.c_int64
        _lib = L
    return _lib


def _p(a):
    return a.ctypes.data_as(ctypes.c_void_p)


def threads():
    return int(lib().oracle_threads())


def set_threads(n):
    lib().oracle_set_threads(int(n))


def window_lo(p, W):
    """Lower end of J_p(W) (Sec. 3.2), 0-based; W = 0 is full history."""
    return int(lib().oracle_window_lo(p, W))


def attend(q, K, V, gamma):
    """Eq. conditional-attention-weight / conditional-attention over an explicit set.

    q [d], K [n, d], V [n, d] float64. Returns (o [d], pi [n])."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    K = np.ascontiguousarray(K, dtype=np.float64)
    V = np.ascontiguousarray(V, dtype=np.float64)
    n, d = K.shape
    o = np.zeros(d)
    pi = np.zeros(max(n, 1))
    lib().oracle_attend(_p(q), _p(K), _p(V), n, d, float(gamma), _p(o), _p(pi))
    return o, pi[:n]


def window_attention_bf16(Q, pos, Kp, Vp, W, gamma):
    """Window-limited attention of rows Q [R, d] (bf16 bits) at positions pos [R]
    over K/V histories Kp, Vp [T, d] (bf16 bits, row = absolute position).
    Returns (O [R, d] float64, sum_pi [R])."""
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    Kp = np.ascontiguousarray(Kp, dtype=np.uint16)
    Vp = np.ascontiguousarray(Vp, dtype=np.uint16)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    R, d = Q.shape
    T = Kp.shape[0]
    O = np.zeros((R, d))
    sp = np.zeros(R)
    rc = lib().oracle_window_attention_bf16(_p(Q), d, _p(pos), R, _p(Kp), _p(Vp), d, T, d,
                                            int(W), float(gamma), _p(O), _p(sp))
    if rc != 0:
        raise ValueError("oracle_window_attention_bf16: bad arguments (rc=%d)" % rc)
    return O, sp


def window_attention_gen(g, layer, b, kvh, qheads, pos, d, W, gamma):
    """Same definition with q/K/V regenerated from the seeded generator.
    Row r: query head qheads[r] of batch row b at position pos[r], reading KV head kvh."""
    qh = np.ascontiguousarray(qheads, dtype=np.int32)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    R = len(pos)
    O = np.zeros((R, d))
    sp = np.zeros(R)
    rc = lib().oracle_window_attention_gen(ctypes.byref(g), layer, b, kvh, _p(qh), _p(pos), R,
                                           d, int(W), float(gamma), _p(O), _p(sp))
    if rc != 0:
        raise ValueError("oracle_window_attention_gen: bad arguments (rc=%d)" % rc)
    return O, sp


def ring_positions(t, cap):
    """Sec. 3.3 residency as a ring: position held by each slot (-1 = empty)."""
    out = np.zeros(cap, dtype=np.int64)
    if lib().oracle_ring_positions(t, cap, _p(out)) != 0:
        raise ValueError("bad ring arguments")
    return out


def ring_expected_gen(g, tensor, layer, b, kvh, d, t, cap):
    out = np.zeros((cap, d), dtype=np.uint16)
    if lib().oracle_ring_expected_gen(ctypes.byref(g), tensor, layer, b, kvh, d, t, cap,
                                      _p(out)) != 0:
        raise ValueError("bad ring arguments")
    return out


def retained_tokens(W, C):
    """r_C(w) (Sec. 3.1)."""
    return int(lib().oracle_retained_tokens(W, C))


def nominal_storage(windows, C, dK, dV, bK=2, bV=2, batch=1):
    """N_C(a), Eq. nominal-storage, in bytes, times `batch` sequences."""
    w = np.ascontiguousarray(windows, dtype=np.int64).ravel()
    return int(lib().oracle_nominal_storage(_p(w), len(w), C, dK, dV, bK, bV, batch))


def normalized_rate(windows, C, dK, dV, bK=2, bV=2):
    """R_C(a), Eq. normalized-rate."""
    w = np.ascontiguousarray(windows, dtype=np.int64).ravel()
    return float(lib().oracle_normalized_rate(_p(w), len(w), C, dK, dV, bK, bV))


EPS_COS = 1e-12  # App. A.2: epsilon of the stabilized cosine


def cos_eval(u, v, eps=EPS_COS):
    """Stabilized cosine (App. A.2, Eq. stabilized-cosine)."""
    u = np.ascontiguousarray(u, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    return float(lib().oracle_cos_eval(_p(u), _p(v), len(u), eps))


def conditional_similarity_bf16(Q, pos, Kp, Vp, windows, gamma, eps=EPS_COS):
    """Eq. conditional-similarity of one KV head: (scores [n_w], cos [R, n_w]).
    Q [R, d] bf16 bits (rows = (position, query head)), pos [R], Kp/Vp [T, d]."""
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    Kp = np.ascontiguousarray(Kp, dtype=np.uint16)
    Vp = np.ascontiguousarray(Vp, dtype=np.uint16)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    W = np.ascontiguousarray(windows, dtype=np.int64)
    R, d = Q.shape
    scores = np.zeros(len(W))
    cos = np.zeros((R, len(W)))
    rc = lib().oracle_conditional_similarity_bf16(_p(Q), _p(pos), R, _p(Kp), _p(Vp), Kp.shape[0],
                                                  d, _p(W), len(W), float(gamma), eps,
                                                  _p(scores), _p(cos))
    if rc != 0:
        raise ValueError("oracle_conditional_similarity_bf16 failed (rc=%d)" % rc)
    return scores, cos


def select_window(scores, windows, C, tau):
    """Eq. threshold-selection for one head; returns the window (0 = full)."""
    s = np.ascontiguousarray(scores, dtype=np.float64)
    W = np.ascontiguousarray(windows, dtype=np.int64)
    return int(lib().oracle_select_window(_p(s), _p(W), len(W), int(C), float(tau)))


def budget_select(beta, phi, budget):
    """Eq. budget-selector: index g* (0-based) of the chosen record, or -1."""
    b = np.ascontiguousarray(beta, dtype=np.float64)
    f = np.ascontiguousarray(phi, dtype=np.float64)
    return int(lib().oracle_budget_select(_p(b), _p(f), len(b), float(budget)))


# ---------------------------------------------------------------- 8-bit format
# The cache format p_KV of Sec. 3.1 with 8-bit keys and values: E4M3 codes and one
# fp32 scale per stored row (a reading; the paper names no 8-bit format).

def e4m3_decode(code):
    """Value of an E4M3 code (exact; NaN for S.1111.111)."""
    return float(lib().oracle_e4m3_decode(int(code)))


def e4m3_encode(x):
    """Nearest E4M3 code of the float32 x (ties to even, |x| > 448 -> 448, NaN -> 0x7F)."""
    return int(lib().oracle_e4m3_encode(float(np.float32(x))))


def quantize_row_e4m3(x_bf16):
    """One stored row: bf16 bits [d] -> (codes uint8 [d], scale float32)."""
    x = np.ascontiguousarray(x_bf16, dtype=np.uint16)
    codes = np.zeros(len(x), dtype=np.uint8)
    scale = np.zeros(1, dtype=np.float32)
    if lib().oracle_quantize_row_e4m3(_p(x), len(x), _p(codes), _p(scale)) != 0:
        raise ValueError("bad row")
    return codes, np.float32(scale[0])


def quantize_rows_e4m3(X_bf16):
    """Rows [n][d] of bf16 bits -> (codes [n][d], scales [n])."""
    X = np.ascontiguousarray(X_bf16, dtype=np.uint16)
    codes = np.zeros(X.shape, dtype=np.uint8)
    scales = np.zeros(X.shape[0], dtype=np.float32)
    for r in range(X.shape[0]):
        codes[r], scales[r] = quantize_row_e4m3(X[r])
    return codes, scales


def dequantize_rows_e4m3(codes, scales):
    """decode(code) * scale, in float64."""
    table = np.array([e4m3_decode(c) for c in range(256)])
    return table[np.asarray(codes)] * np.asarray(scales, dtype=np.float64)[:, None]


def window_attention_fp8(Q, pos, Kc, Ks, Vc, Vs, W, gamma):
    """Window attention (Sec. 3.2) over a history stored in the 8-bit format:
    Q bf16 bits [R][d]; Kc/Vc codes [T][d]; Ks/Vs scales [T]. Returns (O [R][d], sum_pi)."""
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    Kc = np.ascontiguousarray(Kc, dtype=np.uint8)
    Vc = np.ascontiguousarray(Vc, dtype=np.uint8)
    Ks = np.ascontiguousarray(Ks, dtype=np.float32)
    Vs = np.ascontiguousarray(Vs, dtype=np.float32)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    R, d = Q.shape
    O = np.zeros((R, d))
    sp = np.zeros(R)
    rc = lib().oracle_window_attention_fp8(_p(Q), d, _p(pos), R, _p(Kc), _p(Ks), _p(Vc), _p(Vs),
                                           Kc.shape[0], d, int(W), float(gamma), _p(O), _p(sp))
    if rc != 0:
        raise ValueError("oracle_window_attention_fp8 failed (%d)" % rc)
    return O, sp


def ring_expected_fp8_gen(g, tensor, layer, b, kvh, d, t, cap):
    """Expected 8-bit ring after positions 0..t-1: (codes [cap][d], scales [cap])."""
    codes = np.zeros((cap, d), dtype=np.uint8)
    scales = np.zeros(cap, dtype=np.float32)
    if lib().oracle_ring_expected_fp8_gen(ctypes.byref(g), tensor, layer, b, kvh, d, t, cap,
                                          _p(codes), _p(scales)) != 0:
        raise ValueError("bad ring arguments")
    return codes, scales


# ------------------------------------------------------- sink + recent window
# The static sink--recent policy of the StreamingLLM control (App. baseline
# controls): S sink tokens plus a W-token recent window.

def sink_visible(k, p, W, S):
    return bool(lib().oracle_sink_visible(k, p, W, S))


def sink_positions(p, W, S):
    """J of a query at p, increasing."""
    n = int(lib().oracle_sink_positions(p, W, S, None))
    out = np.zeros(max(n, 1), dtype=np.int64)
    lib().oracle_sink_positions(p, W, S, _p(out))
    return out[:n]


def sink_attention_gen(g, layer, b, kvh, qheads, pos, d, W, S, gamma):
    qh = np.ascontiguousarray(qheads, dtype=np.int32)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    R = len(pos)
    O = np.zeros((R, d))
    sp = np.zeros(R)
    rc = lib().oracle_sink_attention_gen(ctypes.byref(g), layer, b, kvh, _p(qh), _p(pos), R, d,
                                         int(W), int(S), float(gamma), _p(O), _p(sp))
    if rc != 0:
        raise ValueError("oracle_sink_attention_gen failed (%d)" % rc)
    return O, sp


def sink_attention_bf16(Q, pos, Kp, Vp, W, S, gamma):
    Q = np.ascontiguousarray(Q, dtype=np.uint16)
    Kp = np.ascontiguousarray(Kp, dtype=np.uint16)
    Vp = np.ascontiguousarray(Vp, dtype=np.uint16)
    pos = np.ascontiguousarray(pos, dtype=np.int64)
    R, d = Q.shape
    O = np.zeros((R, d))
    sp = np.zeros(R)
    rc = lib().oracle_sink_attention_bf16(_p(Q), d, _p(pos), R, _p(Kp), _p(Vp), d, Kp.shape[0], d,
                                          int(W), int(S), float(gamma), _p(O), _p(sp))
    if rc != 0:
        raise ValueError("oracle_sink_attention_bf16 failed (%d)" % rc)
    return O, sp


def sink_ring_positions(t, W, S):
    out = np.zeros(S + W, dtype=np.int64)
    if lib().oracle_sink_ring_positions(t, W, S, _p(out)) != 0:
        raise ValueError("bad ring arguments")
    return out


def sink_ring_expected_gen(g, tensor, layer, b, kvh, d, t, W, S):
    out = np.zeros((S + W, d), dtype=np.uint16)
    if lib().oracle_sink_ring_expected_gen(ctypes.byref(g), tensor, layer, b, kvh, d, t, W, S,
                                           _p(out)) != 0:
        raise ValueError("bad ring arguments")
    return out


def sink_retained_tokens(W, S, C):
    return int(lib().oracle_sink_retained_tokens(W, S, C))
