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
from harness import assert_close

pytestmark = pytest.mark.gpu


class RunS:
    def __init__(self, windows, sinks, n_q_heads=8, n_kv_heads=2, head_dim=128, batch=2,
                 max_ctx=2000, seed=0, kv_format=hwkv.HWKV_KV_BF16):
        import torch
        self.torch = torch
        self.B, self.Hq, self.Hkv, self.d = batch, n_q_heads, n_kv_heads, head_dim
        self.G = n_q_heads // n_kv_heads
        self.windows, self.sinks, self.max_ctx = list(windows), list(sinks), max_ctx
        self.fmt = kv_format
        self.g = hwkv_gen.desc(seed, True)
        self.scale = 1.0 / np.sqrt(head_dim)
        self.pol = hwkv.make_policy(1, n_kv_heads, n_q_heads, head_dim, batch, max_ctx, windows,
                                    kv_format=kv_format, sinks=sinks)
        nb = hwkv.hwkv_required_bytes(self.pol)
        self.arena = torch.empty(nb, dtype=torch.uint8, device="cuda")
        self.stream = torch.cuda.current_stream()
        self.cache = hwkv.hwkv_alloc(self.pol, self.arena, nb, self.stream)

    def close(self):
        hwkv.hwkv_free(self.cache)

    def gen(self, tensor, pos0, n, heads):
        t = self.torch.empty((self.B, n, heads, self.d), dtype=self.torch.bfloat16, device="cuda")
        hwkv_gen.fill_device(self.g, tensor, 0, self.B, pos0, n, heads, self.d, t.data_ptr(),
                             self.stream.cuda_stream)
        return t

    def oracle_rows(self, b, qh, positions):
        h = qh // self.G
        W, S = self.windows[h], self.sinks[h]
        O, sp = oracle.sink_attention_gen(self.g, 0, b, h, [qh] * len(positions), positions,
                                          self.d, W, S, self.scale)
        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
        return O

    def oracle_rows_fp8(self, b, qh, positions):
        """8-bit format: attention (the plain definition over J) over the rows as
        stored, quantized and dequantized, every key of J included."""
        h = qh // self.G
        W, S = self.windows[h], self.sinks[h]
        out = np.zeros((len(positions), self.d))
        for i, p in enumerate(positions):
            J = oracle.sink_positions(p, W, S)
            rows = {}
            for tensor in (hwkv_gen.K, hwkv_gen.V):
                X = np.stack([hwkv_gen.fill_host_sub(self.g, tensor, 0, b, int(k), 1, h, 1, self.d)[0, 0]
                              for k in J])
                codes, scales = oracle.quantize_rows_e4m3(X)
                rows[tensor] = oracle.dequantize_rows_e4m3(codes, scales)
            qb = hwkv_gen.fill_host_sub(self.g, hwkv_gen.Q, 0, b, p, 1, qh, 1, self.d)[0, 0]
            q = (qb.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
            out[i], pi = oracle.attend(q, rows[hwkv_gen.K], rows[hwkv_gen.V], self.scale)
            np.testing.assert_allclose(pi.sum(), 1.0, atol=1e-12)
        return out

    def prefill(self, n, sample=17):
        t0 = hwkv.hwkv_seq_len(self.cache, 0)
        q, k, v = self.gen(hwkv_gen.Q, t0, n, self.Hq), self.gen(hwkv_gen.K, t0, n, self.Hkv), \
            self.gen(hwkv_gen.V, t0, n, self.Hkv)
        out = self.torch.empty((self.B, n, self.Hq, self.d), dtype=self.torch.float32,
                               device="cuda")
        hwkv.hwkv_prefill(self.cache, 0, q, k, v, n, self.scale, out, self.stream)
        got = out.cpu().numpy()
        pos = sorted(set(list(range(t0, t0 + n, sample)) + [t0, t0 + n - 1]))
        for b in range(self.B):
            for qh in range(0, self.Hq, 3):
                want = (self.oracle_rows(b, qh, pos) if self.fmt == hwkv.HWKV_KV_BF16 else
                        self.oracle_rows_fp8(b, qh, pos))
                assert_close(got[b, [p - t0 for p in pos], qh], want,
                             "prefill t0=%d b=%d qh=%d" % (t0, b, qh))

    def append(self, n):
        t0 = hwkv.hwkv_seq_len(self.cache, 0)
        hwkv.hwkv_append(self.cache, 0, self.gen(hwkv_gen.K, t0, n, self.Hkv),
                         self.gen(hwkv_gen.V, t0, n, self.Hkv), n, self.stream)

    def step(self, fused=True):
        t = hwkv.hwkv_seq_len(self.cache, 0)
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        p = t if fused else t - 1
        q = self.gen(hwkv_gen.Q, p, 1, self.Hq).view(self.B, self.Hq, self.d)
        if fused:
            hwkv.hwkv_decode_step(self.cache, 0, q, self.gen(hwkv_gen.K, t, 1, self.Hkv),
                                  self.gen(hwkv_gen.V, t, 1, self.Hkv), self.scale, out, self.stream)
        else:
            hwkv.hwkv_decode_attn(self.cache, 0, q, self.scale, out, self.stream)
        want = np.zeros((self.B, self.Hq, self.d))
        for b in range(self.B):
            for qh in range(self.Hq):
                want[b, qh] = self.oracle_rows(b, qh, [p])[0]
        assert_close(out.cpu().numpy(), want, "decode p=%d" % p)

    def check_rings(self):
        t = hwkv.hwkv_seq_len(self.cache, 0)
        for b in range(self.B):
            for h in range(self.Hkv):
                W, S = self.windows[h], self.sinks[h]
                kr, vr = hwkv.hwkv_debug_copy_ring(self.cache, 0, b, h, self.d, self.fmt)
                cap = kr.shape[0]
                sink_head = W != 0 and S > 0 and S + W < self.max_ctx
                if self.fmt == hwkv.HWKV_KV_BF16:
                    for tensor, ring in ((hwkv_gen.K, kr), (hwkv_gen.V, vr)):
                        want = (oracle.sink_ring_expected_gen(self.g, tensor, 0, b, h, self.d, t, W, S)
                                if sink_head else
                                oracle.ring_expected_gen(self.g, tensor, 0, b, h, self.d, t, cap))
                        assert np.array_equal(ring, want), "ring b=%d h=%d t=%d" % (b, h, t)
                else:
                    ks, vs = hwkv.hwkv_debug_copy_scales(self.cache, 0, b, h)
                    held = (oracle.sink_ring_positions(t, W, S) if sink_head else
                            oracle.ring_positions(t, cap))
                    for tensor, ring, sc in ((hwkv_gen.K, kr, ks), (hwkv_gen.V, vr, vs)):
                        for j, p in enumerate(held):
                            if p < 0:
                                continue
                            row = hwkv_gen.fill_host_sub(self.g, tensor, 0, b, int(p), 1, h, 1,
                                                         self.d)[0, 0]
                            codes, s = oracle.quantize_row_e4m3(row)
                            assert np.array_equal(ring[j], codes) and sc[j] == s, (b, h, j, p)

    def check_residency(self):
        t = hwkv.hwkv_seq_len(self.cache, 0)
        per = 4 * self.d if self.fmt == hwkv.HWKV_KV_BF16 else 2 * (self.d + 4)
        want = sum(oracle.sink_retained_tokens(W, S, t) for W, S in zip(self.windows, self.sinks))
        assert hwkv.hwkv_residency_bytes(self.cache, 0) == want * per * self.B


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
