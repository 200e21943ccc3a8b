"""The 8-bit cache format (E4M3 codes + one fp32 scale per stored row) through
the C ABI, against the oracle's encoding written from the format definition:
ring codes and scales bit-exact (the quantisation decisions are taken in fp32
on both sides), decode and prefill outputs within the attention tolerance of the
oracle's attention over the dequantised rows (Sec. 3.1: with a format that
changes execution, the compared outputs all use it; a prefill chunk's own keys
are read as stored too)."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv
from harness import MAX_ABS, MEAN_ABS, assert_close

pytestmark = pytest.mark.gpu
FP8 = hwkv.HWKV_KV_FP8_E4M3


class Run8:
    """A cache in the 8-bit format plus generator-driven inputs."""

    def __init__(self, n_layers, batch, n_q_heads, n_kv_heads, head_dim, max_ctx, windows, seed=0,
                 per_head_scale=True):
        import torch
        self.torch = torch
        self.L, self.B, self.Hq, self.Hkv, self.d = n_layers, batch, n_q_heads, n_kv_heads, head_dim
        self.G = n_q_heads // n_kv_heads
        self.max_ctx = max_ctx
        self.windows = list(windows)
        self.g = hwkv_gen.desc(seed, per_head_scale)
        self.scale = 1.0 / np.sqrt(head_dim)
        self.pol = hwkv.make_policy(n_layers, n_kv_heads, n_q_heads, head_dim, batch, max_ctx,
                                    windows, kv_format=FP8)
        self.nbytes = hwkv.hwkv_required_bytes(self.pol)
        self.arena = torch.empty(self.nbytes, dtype=torch.uint8, device="cuda")
        self.stream = torch.cuda.current_stream()
        self.cache = hwkv.hwkv_alloc(self.pol, self.arena, self.nbytes, self.stream)

    def close(self):
        hwkv.hwkv_free(self.cache)

    def gen(self, tensor, layer, pos0, n, heads):
        t = self.torch.empty((self.B, n, heads, self.d), dtype=self.torch.bfloat16, device="cuda")
        hwkv_gen.fill_device(self.g, tensor, layer, self.B, pos0, n, heads, self.d, t.data_ptr(),
                             self.stream.cuda_stream)
        return t

    def fill(self, layer, n, chunk=4096):
        done = 0
        while done < n:
            m = min(chunk, n - done)
            t0 = hwkv.hwkv_seq_len(self.cache, layer)
            hwkv.hwkv_append(self.cache, layer, self.gen(hwkv_gen.K, layer, t0, m, self.Hkv),
                             self.gen(hwkv_gen.V, layer, t0, m, self.Hkv), m, self.stream)
            done += m

    def step(self, layer, fused=True):
        t = hwkv.hwkv_seq_len(self.cache, layer)
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        if fused:
            q = self.gen(hwkv_gen.Q, layer, t, 1, self.Hq).view(self.B, self.Hq, self.d)
            hwkv.hwkv_decode_step(self.cache, layer, q, self.gen(hwkv_gen.K, layer, t, 1, self.Hkv),
                                  self.gen(hwkv_gen.V, layer, t, 1, self.Hkv), self.scale, out,
                                  self.stream)
        else:
            q = self.gen(hwkv_gen.Q, layer, t - 1, 1, self.Hq).view(self.B, self.Hq, self.d)
            hwkv.hwkv_decode_attn(self.cache, layer, q, self.scale, out, self.stream)
        return out

    def window(self, layer, h):
        return self.windows[layer * self.Hkv + h]

    def oracle_unit(self, layer, b, h, p):
        """[G, d]: the G query heads of KV head h at position p over the 8-bit rows."""
        W = self.window(layer, h)
        Weff = 0 if (W == 0 or W >= self.max_ctx) else W
        lo = oracle.window_lo(p, Weff)
        K = hwkv_gen.fill_host_sub(self.g, hwkv_gen.K, layer, b, lo, p - lo + 1, h, 1, self.d)[:, 0]
        V = hwkv_gen.fill_host_sub(self.g, hwkv_gen.V, layer, b, lo, p - lo + 1, h, 1, self.d)[:, 0]
        Q = hwkv_gen.fill_host_sub(self.g, hwkv_gen.Q, layer, b, p, 1, h * self.G, self.G,
                                   self.d)[0]
        Kc, Ks = oracle.quantize_rows_e4m3(K)
        Vc, Vs = oracle.quantize_rows_e4m3(V)
        O, sp = oracle.window_attention_fp8(Q, [p - lo] * self.G, Kc, Ks, Vc, Vs, 0, self.scale)
        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
        return O

    def oracle_step(self, layer, p, heads=None):
        want = np.zeros((self.B, self.Hq, self.d))
        for b in range(self.B):
            for h in (heads if heads is not None else range(self.Hkv)):
                want[b, h * self.G:(h + 1) * self.G] = self.oracle_unit(layer, b, h, p)
        return want

    def check_rings(self, layer):
        t = hwkv.hwkv_seq_len(self.cache, layer)
        for b in range(self.B):
            for h in range(self.Hkv):
                kr, vr = hwkv.hwkv_debug_copy_ring(self.cache, layer, b, h, self.d, FP8)
                ks, vs = hwkv.hwkv_debug_copy_scales(self.cache, layer, b, h)
                cap = kr.shape[0]
                ek, eks = oracle.ring_expected_fp8_gen(self.g, hwkv_gen.K, layer, b, h, self.d, t, cap)
                ev, evs = oracle.ring_expected_fp8_gen(self.g, hwkv_gen.V, layer, b, h, self.d, t, cap)
                assert np.array_equal(kr, ek), "K codes (layer %d, b %d, h %d)" % (layer, b, h)
                assert np.array_equal(vr, ev), "V codes (layer %d, b %d, h %d)" % (layer, b, h)
                assert np.array_equal(ks.view(np.uint32), eks.view(np.uint32)), "K scales"
                assert np.array_equal(vs.view(np.uint32), evs.view(np.uint32)), "V scales"


@pytest.mark.parametrize("d", [128, 256])
def test_fp8_rings_bit_exact_and_decode(d):
    r = Run8(1, 2, 8, 2, d, 700, [0, 100], seed=7)
    try:
        r.fill(0, 37)             # below the window: nothing wrapped
        r.check_rings(0)
        r.fill(0, 230)            # the 100-token ring wraps
        r.check_rings(0)
        out = r.step(0, fused=False)  # decode of the last appended token
        assert_close(out.cpu().numpy(), r.oracle_step(0, 266), "fp8 decode_attn d=%d" % d)
        for _ in range(3):        # fused steps: the new row is quantised inside the split kernel
            t = hwkv.hwkv_seq_len(r.cache, 0)
            out = r.step(0, fused=True)
            assert_close(out.cpu().numpy(), r.oracle_step(0, t), "fp8 decode_step d=%d" % d)
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings(0)
        w = r.windows
        t = hwkv.hwkv_seq_len(r.cache, 0)
        # residency: r_C(w) rows of (d codes + one 4-byte scale) for K and V (effective
        # precision (d + 4) / d bytes per element in Eq. nominal-storage)
        assert hwkv.hwkv_residency_bytes(r.cache, 0) == oracle.nominal_storage(w, t, d + 4, d + 4, 1, 1, r.B)
    finally:
        r.close()


def test_fp8_zero_row():
    import torch
    r = Run8(1, 2, 4, 1, 256, 300, [0], seed=2)
    try:
        r.fill(0, 20)
        z = torch.zeros((r.B, 1, r.Hkv, r.d), dtype=torch.bfloat16, device="cuda")
        hwkv.hwkv_append(r.cache, 0, z, z, 1, r.stream)  # stored as scale 0, zero codes
        kr, vr = hwkv.hwkv_debug_copy_ring(r.cache, 0, 1, 0, r.d, FP8)
        ks, vs = hwkv.hwkv_debug_copy_scales(r.cache, 0, 1, 0)
        assert not kr[20].any() and not vr[20].any() and ks[20] == 0.0 and vs[20] == 0.0
        assert ks[19] > 0.0
    finally:
        r.close()


def test_fp8_graph_step():
    import torch
    r = Run8(2, 3, 8, 2, 128, 600, [64, 0, 0, 200], seed=3)
    try:
        for layer in range(2):
            r.fill(layer, 150)
        q = [torch.empty((r.B, r.Hq, r.d), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        k = [torch.empty((r.B, r.Hkv, r.d), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
        v = [torch.empty_like(x) for x in k]
        outs = [torch.empty((r.B, r.Hq, r.d), dtype=torch.float32, device="cuda") for _ in range(2)]
        graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            st = torch.cuda.current_stream()
            for layer in range(2):
                hwkv.hwkv_decode_step_graph(r.cache, layer, q[layer], k[layer], v[layer], r.scale,
                                            outs[layer], st)
        for t in (150, 151, 152):
            for layer in range(2):
                q[layer].copy_(r.gen(hwkv_gen.Q, layer, t, 1, r.Hq).view(r.B, r.Hq, r.d))
                k[layer].copy_(r.gen(hwkv_gen.K, layer, t, 1, r.Hkv).view(r.B, r.Hkv, r.d))
                v[layer].copy_(r.gen(hwkv_gen.V, layer, t, 1, r.Hkv).view(r.B, r.Hkv, r.d))
            graph.replay()
            for layer in range(2):
                assert_close(outs[layer].cpu().numpy(), r.oracle_step(layer, t),
                             "fp8 graph step layer %d t %d" % (layer, t))
        hwkv.hwkv_sync_check(r.cache)
        for layer in range(2):
            assert hwkv.hwkv_seq_len(r.cache, layer) == 153
            r.check_rings(layer)
    finally:
        r.close()


def test_fp8_larger_sampled():
    # d = 256, 24 query / 4 KV heads, windows {full, 16384, 4096, 1024}, 20K tokens
    r = Run8(1, 2, 24, 4, 256, 20600, [0, 16384, 4096, 1024], seed=19)
    try:
        r.fill(0, 20000, chunk=8192)
        for _ in range(2):
            t = hwkv.hwkv_seq_len(r.cache, 0)
            out = r.step(0, fused=True)
            assert_close(out.cpu().numpy(), r.oracle_step(0, t), "fp8 20K step")
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_fp8_unsupported_head_dim():
    with pytest.raises(hwkv.HwkvError) as e:
        pol = hwkv.make_policy(1, 1, 1, 64, 1, 100, [0], kv_format=FP8)
        hwkv.hwkv_required_bytes(pol)
    assert e.value.status == hwkv.HWKV_EUNSUPPORTED


def prefill_chunk(r, layer, n, row0=None, n_rows=None):
    """Prefill n tokens of the generator's q/k/v into rows [row0, row0 + n_rows)."""
    import torch
    row0 = 0 if row0 is None else row0
    n_rows = r.B if n_rows is None else n_rows
    t0 = hwkv.hwkv_row_len(r.cache, layer, row0)
    def gen(tensor, heads):
        full = r.gen(tensor, layer, t0, n, heads)
        return full[row0:row0 + n_rows].contiguous()
    q, k, v = gen(hwkv_gen.Q, r.Hq), gen(hwkv_gen.K, r.Hkv), gen(hwkv_gen.V, r.Hkv)
    out = torch.empty((n_rows, n, r.Hq, r.d), dtype=torch.float32, device="cuda")
    if n_rows == r.B:
        hwkv.hwkv_prefill(r.cache, layer, q, k, v, n, r.scale, out, r.stream)
    else:
        hwkv.hwkv_prefill_rows(r.cache, layer, row0, n_rows, q, k, v, n, r.scale, out, r.stream)
    return t0, out.cpu().numpy()


def check_prefill(r, layer, t0, n, got, row0=0, stride=13):
    pos = sorted(set(range(t0, t0 + n, stride)) | {t0, t0 + n - 1})
    for bi in range(got.shape[0]):
        for h in range(r.Hkv):
            for p in pos:
                want = r.oracle_unit(layer, row0 + bi, h, p)
                assert_close(got[bi, p - t0, h * r.G:(h + 1) * r.G], want,
                             "fp8 prefill b=%d h=%d p=%d" % (row0 + bi, h, p))


@pytest.mark.parametrize("d", [128, 256])
def test_fp8_prefill_parity_and_rings(d):
    # a full head and a 100-token window; chunks from an empty cache, past the
    # window (the ring wraps inside the call) and after appended history
    r = Run8(1, 2, 8, 2, d, 1400, [0, 100], seed=23)
    try:
        for n in (70, 333):
            t0, got = prefill_chunk(r, 0, n)
            check_prefill(r, 0, t0, n, got)
            r.check_rings(0)
        r.fill(0, 41)
        t0, got = prefill_chunk(r, 0, 150)
        check_prefill(r, 0, t0, 150, got)
        r.check_rings(0)
        t = hwkv.hwkv_seq_len(r.cache, 0)
        out = r.step(0, fused=True)
        assert_close(out.cpu().numpy(), r.oracle_step(0, t), "fp8 decode after prefill d=%d" % d)
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_fp8_prefill_rows_ragged():
    # rows of one cache at different lengths: a row range prefilled on its own
    r = Run8(1, 3, 8, 2, 128, 900, [0, 64], seed=29)
    try:
        t0, got = prefill_chunk(r, 0, 90)
        t0, got = prefill_chunk(r, 0, 130, row0=1, n_rows=2)
        assert [hwkv.hwkv_row_len(r.cache, 0, b) for b in range(3)] == [90, 220, 220]
        check_prefill(r, 0, t0, 130, got, row0=1, stride=11)
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_prefill64k_fp8_sampled():
    """The bench's 8-bit prefill (prefill64k: 8 chunks of 8,192 tokens, B2, 32q/8kv, d128,
    windows drawn per KV head) on sampled rows of the first and the last chunk, for one
    full-history and one windowed KV head per batch row."""
    from hwkv_gen import workloads
    wl = workloads.make("prefill64k")
    r = Run8(wl.n_layers, wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.max_ctx,
             wl.windows, seed=wl.seed, per_head_scale=wl.per_head_scale)
    rng = np.random.default_rng(5)
    try:
        n = wl.chunk
        kept = {}
        for c in range(wl.prompt // n):
            t0, got = prefill_chunk(r, 0, n)
            if c in (0, wl.prompt // n - 1):
                kept[c] = (t0, got)
        hwkv.hwkv_sync_check(r.cache)
        full = [h for h in range(r.Hkv) if r.window(0, h) == 0 or r.window(0, h) >= r.max_ctx]
        win = [h for h in range(r.Hkv) if h not in full]
        heads = ([full[0]] if full else []) + ([win[0]] if win else [])
        for c, (t0, got) in kept.items():
            rows = sorted({0, n - 1} | set(rng.integers(0, n, size=6).tolist()))
            pos = [t0 + i for i in rows]
            for b in range(r.B):
                for h in heads:
                    T = pos[-1] + 1
                    K = hwkv_gen.fill_host_sub(r.g, hwkv_gen.K, 0, b, 0, T, h, 1, r.d)[:, 0]
                    V = hwkv_gen.fill_host_sub(r.g, hwkv_gen.V, 0, b, 0, T, h, 1, r.d)[:, 0]
                    Kc, Ks = oracle.quantize_rows_e4m3(K)
                    Vc, Vs = oracle.quantize_rows_e4m3(V)
                    W = r.window(0, h)
                    W = 0 if W >= r.max_ctx else W
                    for qg in range(r.G):
                        qh = h * r.G + qg
                        Q = np.stack([hwkv_gen.fill_host_sub(r.g, hwkv_gen.Q, 0, b, p, 1, qh, 1, r.d)[0, 0]
                                      for p in pos])
                        O, sp = oracle.window_attention_fp8(Q, pos, Kc, Ks, Vc, Vs, W, r.scale)
                        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
                        assert_close(got[b, rows, qh], O, "fp8 prefill64k chunk %d b%d q%d" % (c, b, qh))
    finally:
        r.close()
