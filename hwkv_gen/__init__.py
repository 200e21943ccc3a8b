"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle.

The definition is in ``hwkv_gen.h``: a counter-based splitmix64 generator,
Irwin-Hall(12) values rounded to bf16, optionally scaled per (layer, KV head).
This package holds none of the attention arithmetic. Arrays are returned as
uint16 bf16 bit patterns in the library's ``[B, n, H, d]`` layout.
"""
import ctypes
import os

import numpy as np

from . import build as _build

Q, K, V = 1, 2, 3


class GenDesc(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("per_head_scale", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


def desc(seed=0, per_head_scale=False):
    return GenDesc(seed, 1 if per_head_scale else 0, 0)


_host = None
_dev = None


def _host_lib():
    global _host
    if _host is None:
        _build.build(device=False)
        lib = ctypes.CDLL(_build.HOST_LIB)
        lib.hwkv_gen_fill_host.argtypes = [ctypes.POINTER(GenDesc), ctypes.c_uint32,
                                           ctypes.c_uint32, ctypes.c_int32, ctypes.c_int64,
                                           ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                           ctypes.c_void_p]
        lib.hwkv_gen_fill_host.restype = ctypes.c_int
        lib.hwkv_gen_fill_host_sub.argtypes = [
            ctypes.POINTER(GenDesc), ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
            ctypes.c_int32, ctypes.c_void_p]
        lib.hwkv_gen_fill_host_sub.restype = ctypes.c_int
        lib.hwkv_gen_one.argtypes = [ctypes.POINTER(GenDesc), ctypes.c_uint32, ctypes.c_uint32,
                                     ctypes.c_uint32, ctypes.c_uint32, ctypes.c_int64,
                                     ctypes.c_uint32]
        lib.hwkv_gen_one.restype = ctypes.c_uint16
        lib.hwkv_gen_scale.argtypes = [ctypes.POINTER(GenDesc), ctypes.c_uint32,
                                       ctypes.c_uint32, ctypes.c_uint32]
        lib.hwkv_gen_scale.restype = ctypes.c_float
        lib.hwkv_gen_splitmix64_out.argtypes = [ctypes.c_uint64, ctypes.c_uint32]
        lib.hwkv_gen_splitmix64_out.restype = ctypes.c_uint64
        _host = lib
    return _host


def _dev_lib():
    global _dev
    if _dev is None:
        _build.build(device=True)
        lib = ctypes.CDLL(_build.DEV_LIB)
        lib.hwkv_gen_fill_device.argtypes = [ctypes.POINTER(GenDesc), ctypes.c_uint32,
                                             ctypes.c_uint32, ctypes.c_int32, ctypes.c_int64,
                                             ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                             ctypes.c_void_p, ctypes.c_void_p]
        lib.hwkv_gen_fill_device.restype = ctypes.c_int
        _dev = lib
    return _dev


def fill_host(g, tensor, layer, B, pos0, n, H, d):
    """uint16 array [B, n, H, d] of bf16 bits for positions pos0 .. pos0+n-1."""
    out = np.empty((B, n, H, d), dtype=np.uint16)
    rc = _host_lib().hwkv_gen_fill_host(ctypes.byref(g), tensor, layer, B, pos0, n, H, d,
                                        out.ctypes.data_as(ctypes.c_void_p))
    if rc != 0:
        raise ValueError("hwkv_gen_fill_host: bad arguments")
    return out


def fill_host_sub(g, tensor, layer, b, pos0, n, head0, H, d):
    """uint16 array [n, H, d]: batch row b and heads head0 .. head0+H-1 only."""
    out = np.empty((1, n, H, d), dtype=np.uint16)
    rc = _host_lib().hwkv_gen_fill_host_sub(ctypes.byref(g), tensor, layer, b, 1, pos0, n, head0,
                                            H, d, out.ctypes.data_as(ctypes.c_void_p))
    if rc != 0:
        raise ValueError("hwkv_gen_fill_host_sub: bad arguments")
    return out[0]


def one(g, tensor, layer, b, head, pos, dim):
    return int(_host_lib().hwkv_gen_one(ctypes.byref(g), tensor, layer, b, head, pos, dim))


def head_scale(g, tensor, layer, head):
    return float(_host_lib().hwkv_gen_scale(ctypes.byref(g), tensor, layer, head))


def splitmix64_out(state, j):
    """j-th output of splitmix64 seeded with `state` (the generator's core)."""
    return int(_host_lib().hwkv_gen_splitmix64_out(state, j))


def fill_device(g, tensor, layer, B, pos0, n, H, d, out_ptr, stream_ptr=0):
    """Fill device memory at out_ptr ([B, n, H, d] bf16) on the given CUDA stream."""
    rc = _dev_lib().hwkv_gen_fill_device(ctypes.byref(g), tensor, layer, B, pos0, n, H, d,
                                         ctypes.c_void_p(out_ptr), ctypes.c_void_p(stream_ptr))
    if rc != 0:
        raise RuntimeError("hwkv_gen_fill_device failed (rc=%d)" % rc)


def bf16_bits_to_float(a):
    """Exact widening of uint16 bf16 bit patterns to float64."""
    a = np.asarray(a, dtype=np.uint16)
    return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
