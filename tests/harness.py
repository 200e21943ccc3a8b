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
