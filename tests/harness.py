"""GPU test helpers: build a cache for a shape, feed it generator inputs through
the C ABI, and compare with the oracle. Inputs come only from hwkv_gen."""
import numpy as np

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv

MAX_ABS = 2e-2   # attention outputs, bf16 inputs with fp32 accumulation
MEAN_ABS = 2e-3


class Run:
    """One cache plus the device buffers needed to drive it."""

    def __init__(self, n_layers, batch, n_q_heads, n_kv_heads, head_dim, max_ctx, windows,
                 seed=0, per_head_scale=False, kv_format=hwkv.HWKV_KV_BF16):
        import torch
        self.torch = torch
        self.L, self.B, self.Hq, self.Hkv, self.d = n_layers, batch, n_q_heads, n_kv_heads, head_dim
        self.G = n_q_heads // n_kv_heads
        self.max_ctx = max_ctx
        self.windows = list(windows)
        self.g = hwkv_gen.desc(seed, per_head_scale)
        self.scale = 1.0 / np.sqrt(head_dim)
        self.pol = hwkv.make_policy(n_layers, n_kv_heads, n_q_heads, head_dim, batch, max_ctx,
                                    windows, kv_format=kv_format)
        self.nbytes = hwkv.hwkv_required_bytes(self.pol)
        self.arena = torch.empty(self.nbytes, dtype=torch.uint8, device="cuda")
        self.stream = torch.cuda.current_stream()
        self.s = self.stream.cuda_stream
        self.cache = hwkv.hwkv_alloc(self.pol, self.arena, self.nbytes, self.stream)

    @classmethod
    def for_workload(cls, wl):
        return cls(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.max_ctx,
                   wl.windows, wl.seed, wl.per_head_scale)

    def close(self):
        if self.cache is not None:
            hwkv.hwkv_free(self.cache)
            self.cache = None

    def window(self, layer, h):
        return self.windows[layer * self.Hkv + h]

    def gen(self, tensor, layer, pos0, n, heads):
        t = self.torch.empty((self.B, n, heads, self.d), dtype=self.torch.bfloat16, device="cuda")
        hwkv_gen.fill_device(self.g, tensor, layer, self.B, pos0, n, heads, self.d, t.data_ptr(),
                             self.s)
        return t

    def append(self, layer, n):
        t0 = hwkv.hwkv_seq_len(self.cache, layer)
        k = self.gen(hwkv_gen.K, layer, t0, n, self.Hkv)
        v = self.gen(hwkv_gen.V, layer, t0, n, self.Hkv)
        hwkv.hwkv_append(self.cache, layer, k, v, n, self.stream)

    def fill(self, layer, n, chunk=8192):
        done = 0
        while done < n:
            m = min(chunk, n - done)
            self.append(layer, m)
            done += m

    def prefill(self, layer, n):
        t0 = hwkv.hwkv_seq_len(self.cache, layer)
        q = self.gen(hwkv_gen.Q, layer, t0, n, self.Hq)
        k = self.gen(hwkv_gen.K, layer, t0, n, self.Hkv)
        v = self.gen(hwkv_gen.V, layer, t0, n, self.Hkv)
        out = self.torch.empty((self.B, n, self.Hq, self.d), dtype=self.torch.float32,
                               device="cuda")
        hwkv.hwkv_prefill(self.cache, layer, q, k, v, n, self.scale, out, self.stream)
        return out

    def decode_step(self, layer):
        """Append the token at position t and attend from it; returns out [B, Hq, d]."""
        self.append(layer, 1)
        p = hwkv.hwkv_seq_len(self.cache, layer) - 1
        q = self.gen(hwkv_gen.Q, layer, p, 1, self.Hq).view(self.B, self.Hq, self.d)
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        hwkv.hwkv_decode_attn(self.cache, layer, q, self.scale, out, self.stream)
        return out

    def decode_step_fused(self, layer):
        """hwkv_decode_step: append the token at position t and attend, in one call."""
        t = hwkv.hwkv_seq_len(self.cache, layer)
        k = self.gen(hwkv_gen.K, layer, t, 1, self.Hkv)
        v = self.gen(hwkv_gen.V, layer, t, 1, self.Hkv)
        q = self.gen(hwkv_gen.Q, layer, t, 1, self.Hq).view(self.B, self.Hq, self.d)
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        hwkv.hwkv_decode_step(self.cache, layer, q, k, v, self.scale, out, self.stream)
        return out

    def oracle_rows(self, layer, b, qh, positions):
        h = qh // self.G
        O, sp = oracle.window_attention_gen(self.g, layer, b, h, [qh] * len(positions),
                                            positions, self.d, self.window(layer, h), self.scale)
        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
        return O

    def check_rings(self, layer):
        t = hwkv.hwkv_seq_len(self.cache, layer)
        for b in range(self.B):
            for h in range(self.Hkv):
                kr, vr = hwkv.hwkv_debug_copy_ring(self.cache, layer, b, h, self.d)
                cap = kr.shape[0]
                ek = oracle.ring_expected_gen(self.g, hwkv_gen.K, layer, b, h, self.d, t, cap)
                ev = oracle.ring_expected_gen(self.g, hwkv_gen.V, layer, b, h, self.d, t, cap)
                assert np.array_equal(kr, ek), "K ring (layer %d, b %d, h %d) differs" % (layer, b, h)
                assert np.array_equal(vr, ev), "V ring (layer %d, b %d, h %d) differs" % (layer, b, h)

    def check_residency(self):
        for layer in range(self.L):
            t = hwkv.hwkv_seq_len(self.cache, layer)
            w = self.windows[layer * self.Hkv:(layer + 1) * self.Hkv]
            assert hwkv.hwkv_residency_bytes(self.cache, layer) == \
                oracle.nominal_storage(w, t, self.d, self.d, 2, 2, self.B)


def assert_close(got, want, what=""):
    err = np.abs(np.asarray(got, dtype=np.float64) - want)
    assert np.isfinite(got).all(), "%s: non-finite output" % what
    assert err.max() <= MAX_ABS, "%s: max abs err %.4g > %g" % (what, err.max(), MAX_ABS)
    assert err.mean() <= MEAN_ABS, "%s: mean abs err %.4g > %g" % (what, err.mean(), MEAN_ABS)
    return err.max(), err.mean()


def oracle_unit_decode(run, layer, b, h, p):
    """Oracle outputs [G, d] of the G query heads of KV head h at position p, from
    host-generated inputs (array form: the K/V window is generated once)."""
    W = run.window(layer, h)
    Weff = 0 if (W == 0 or W >= run.max_ctx) else W
    lo = oracle.window_lo(p, Weff)
    K = hwkv_gen.fill_host_sub(run.g, hwkv_gen.K, layer, b, lo, p - lo + 1, h, 1, run.d)[:, 0]
    V = hwkv_gen.fill_host_sub(run.g, hwkv_gen.V, layer, b, lo, p - lo + 1, h, 1, run.d)[:, 0]
    Q = hwkv_gen.fill_host_sub(run.g, hwkv_gen.Q, layer, b, p, 1, h * run.G, run.G, run.d)[0]
    O, sp = oracle.window_attention_bf16(Q, [p - lo] * run.G, K, V, 0, run.scale)
    np.testing.assert_allclose(sp, 1.0, atol=1e-12)
    return O


def check_ring_unit(run, layer, b, h):
    t = hwkv.hwkv_seq_len(run.cache, layer)
    kr, vr = hwkv.hwkv_debug_copy_ring(run.cache, layer, b, h, run.d)
    cap = kr.shape[0]
    assert np.array_equal(kr, oracle.ring_expected_gen(run.g, hwkv_gen.K, layer, b, h, run.d, t, cap))
    assert np.array_equal(vr, oracle.ring_expected_gen(run.g, hwkv_gen.V, layer, b, h, run.d, t, cap))


class RunS:
    """One layer of sink + recent-window heads (windows[h], sinks[h] per KV head) plus
    generator-driven inputs, with ring and residency checks against the oracle's sink
    layout; both cache formats."""
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
