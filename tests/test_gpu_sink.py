"""Sink + recent window heads (the static sink--recent policy of the paper's
StreamingLLM control: S sink tokens plus a W-token window) through the C ABI:
prefill chunks that start below, inside and past the sink region, appends that
wrap the window region, decode (plain, fused, captured graph), ring contents
bit-exact against the oracle's ring, residency by the retained-count closed
form, and 8-bit rings and prefill of sink heads."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv
from harness import RunS, assert_close

pytestmark = pytest.mark.gpu


def test_sink_prefill_decode_and_rings():
    r = RunS(windows=[64, 0], sinks=[5, 0], seed=4)
    try:
        r.prefill(3)     # the whole chunk lies in the sink region
        r.check_rings()
        r.prefill(100)   # starts inside the sinks, fills and wraps the window region
        r.check_rings()
        r.prefill(257)   # long past the sinks, chunk longer than the window
        r.check_rings()
        r.check_residency()
        r.step(fused=False)
        for _ in range(3):
            r.step(fused=True)
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings()
        r.check_residency()
    finally:
        r.close()


@pytest.mark.parametrize("fmt", [hwkv.HWKV_KV_BF16, hwkv.HWKV_KV_FP8_E4M3])
def test_sink_prefill_head_dim_256(fmt):
    # d = 256, 24 query / 4 KV heads (G = 6: 126 rows per 128-row tile): the kernel with one
    # query tile per CTA and separate K and V copy threads, over sink tiles, wrapped window
    # regions, a plain window and a full head, with chunks shorter and longer than windows
    r = RunS(windows=[100, 33, 0, 200], sinks=[4, 31, 0, 0], n_q_heads=24, n_kv_heads=4,
             head_dim=256, max_ctx=1200, seed=9, kv_format=fmt)
    try:
        r.prefill(20)    # inside head 1's sinks
        r.check_rings()
        r.prefill(150)   # past every sink region; the window regions wrap
        r.check_rings()
        r.prefill(333)   # one chunk longer than every window
        r.check_rings()
        r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_sink_appends_and_graph_step():
    import torch
    # d = 256, 24 query / 4 KV heads: sink heads with several (S, W), a plain window, a full head
    r = RunS(windows=[100, 33, 0, 700], sinks=[4, 31, 0, 0], n_q_heads=24, n_kv_heads=4,
             head_dim=256, max_ctx=3000, seed=8)
    try:
        r.append(2)      # below every sink count
        r.append(600)    # one call longer than S + W: only the last window's worth written
        r.check_rings()
        q = torch.empty((r.B, r.Hq, r.d), dtype=torch.bfloat16, device="cuda")
        k = torch.empty((r.B, r.Hkv, r.d), dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        out = torch.empty((r.B, r.Hq, r.d), dtype=torch.float32, device="cuda")
        graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            hwkv.hwkv_decode_step_graph(r.cache, 0, q, k, v, r.scale, out,
                                        torch.cuda.current_stream())
        for t in (602, 603):
            q.copy_(r.gen(hwkv_gen.Q, t, 1, r.Hq).view(r.B, r.Hq, r.d))
            k.copy_(r.gen(hwkv_gen.K, t, 1, r.Hkv).view(r.B, r.Hkv, r.d))
            v.copy_(r.gen(hwkv_gen.V, t, 1, r.Hkv).view(r.B, r.Hkv, r.d))
            graph.replay()
            want = np.zeros((r.B, r.Hq, r.d))
            for b in range(r.B):
                for qh in range(r.Hq):
                    want[b, qh] = r.oracle_rows(b, qh, [t])[0]
            assert_close(out.cpu().numpy(), want, "graph step t=%d" % t)
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings()
        r.check_residency()
    finally:
        r.close()


def test_sink_rings_in_8_bits():
    r = RunS(windows=[50, 0], sinks=[7, 0], head_dim=128, max_ctx=800, seed=6,
             kv_format=hwkv.HWKV_KV_FP8_E4M3)
    try:
        r.append(3)
        r.append(180)
        for _ in range(2):
            t = hwkv.hwkv_seq_len(r.cache, 0)
            out = torch_step_fp8(r, t)
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings()
        r.check_residency()
    finally:
        r.close()


def test_sink_prefill_8_bits():
    r = RunS(windows=[48, 0], sinks=[5, 0], head_dim=128, max_ctx=700, seed=12,
             kv_format=hwkv.HWKV_KV_FP8_E4M3)
    try:
        r.prefill(3, sample=1)   # inside the sink region
        r.prefill(100)           # through the sinks, wraps the window region
        r.prefill(150)
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings()
        r.check_residency()
    finally:
        r.close()


def torch_step_fp8(r, t):
    out = r.torch.empty((r.B, r.Hq, r.d), dtype=r.torch.float32, device="cuda")
    q = r.gen(hwkv_gen.Q, t, 1, r.Hq).view(r.B, r.Hq, r.d)
    hwkv.hwkv_decode_step(r.cache, 0, q, r.gen(hwkv_gen.K, t, 1, r.Hkv),
                          r.gen(hwkv_gen.V, t, 1, r.Hkv), r.scale, out, r.stream)
    assert r.torch.isfinite(out).all()
    return out
