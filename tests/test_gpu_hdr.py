"""Parity on high-dynamic-range logits (Sec. 3.2, Eq. conditional-attention-weight
and Eq. conditional-attention over J_t(w)), both cache formats, head_dim 128 and 256.

The inputs are explicit host arrays: the seeded generator's q, K and V, with the
K row of position s multiplied by a ramp 1 + s / T and a few spike positions by
4 more, and logits taken with gamma = 1 (sqrt(d) times the usual 1 / sqrt(d)).
The logits then have a standard deviation of sqrt(d) (11 to 16) and the spikes
reach several times that, so a row's softmax is dominated by a handful of keys
and its running maximum jumps by tens of units when a late key tile holds a
spike. That drives the branches benign inputs never reach: the prefill's lazy
rescale of O (taken only when a row's maximum grows by more than 2^8) and, in
decode, a log-sum-exp merge of ring segments whose maxima differ by tens of
units. Every output is compared with the fp64 oracle on the same arrays (for the
8-bit format, over the rows as the 8-bit cache stores them), at the attention
tolerance of every other parity test; the rings are checked bit-exactly."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv
from harness import assert_close

pytestmark = pytest.mark.gpu
BF16, FP8 = hwkv.HWKV_KV_BF16, hwkv.HWKV_KV_FP8_E4M3


def to_bf16_bits(x):
    """float32 -> bf16 bits, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def bf16_bits_to_f32(b):
    return (np.asarray(b, dtype=np.uint32) << 16).view(np.float32)


class ArrayRun:
    """One layer's cache driven from host arrays Q [B][T][Hq][d], K and V
    [B][T][Hkv][d] (bf16 bits)."""

    def __init__(self, B, Hq, Hkv, d, windows, T, fmt, seed, spikes, gamma=1.0):
        import torch
        self.torch = torch
        self.B, self.Hq, self.Hkv, self.d, self.T, self.fmt = B, Hq, Hkv, d, T, fmt
        self.G = Hq // Hkv
        self.windows = list(windows)
        self.gamma = gamma
        g = hwkv_gen.desc(seed)
        self.Q = hwkv_gen.fill_host(g, hwkv_gen.Q, 0, B, 0, T, Hq, d)
        k = bf16_bits_to_f32(hwkv_gen.fill_host(g, hwkv_gen.K, 0, B, 0, T, Hkv, d))
        k *= (1.0 + np.arange(T, dtype=np.float32) / T)[None, :, None, None]
        for s in spikes:
            k[:, s] *= 4.0
        self.K = to_bf16_bits(k)
        self.V = hwkv_gen.fill_host(g, hwkv_gen.V, 0, B, 0, T, Hkv, d)
        self.pol = hwkv.make_policy(1, Hkv, Hq, d, B, T, windows, kv_format=fmt)
        nbytes = hwkv.hwkv_required_bytes(self.pol)
        self.arena = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        self.stream = torch.cuda.current_stream()
        self.cache = hwkv.hwkv_alloc(self.pol, self.arena, nbytes, self.stream)
        if fmt == FP8:  # what the 8-bit cache stores for every row
            self.Kq = [[oracle.quantize_rows_e4m3(self.K[b, :, h]) for h in range(Hkv)]
                       for b in range(B)]
            self.Vq = [[oracle.quantize_rows_e4m3(self.V[b, :, h]) for h in range(Hkv)]
                       for b in range(B)]

    def close(self):
        hwkv.hwkv_free(self.cache)

    def dev(self, a):
        t = self.torch.from_numpy(np.ascontiguousarray(a).view(np.int16))
        return t.view(self.torch.bfloat16).cuda()

    def t(self):
        return hwkv.hwkv_seq_len(self.cache, 0)

    def prefill(self, n):
        t0 = self.t()
        out = self.torch.empty((self.B, n, self.Hq, self.d), dtype=self.torch.float32,
                               device="cuda")
        hwkv.hwkv_prefill(self.cache, 0, self.dev(self.Q[:, t0:t0 + n]),
                          self.dev(self.K[:, t0:t0 + n]), self.dev(self.V[:, t0:t0 + n]), n,
                          self.gamma, out, self.stream)
        return out.cpu().numpy()

    def append(self, n):
        t0 = self.t()
        hwkv.hwkv_append(self.cache, 0, self.dev(self.K[:, t0:t0 + n]),
                         self.dev(self.V[:, t0:t0 + n]), n, self.stream)

    def decode_step(self):
        """Fused append of the token at position t and its decode."""
        t = self.t()
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        hwkv.hwkv_decode_step(self.cache, 0, self.dev(self.Q[:, t]), self.dev(self.K[:, t]),
                              self.dev(self.V[:, t]), self.gamma, out, self.stream)
        return out.cpu().numpy()

    def decode_attn(self):
        """Decode of the last appended token over the current rings."""
        p = self.t() - 1
        out = self.torch.empty((self.B, self.Hq, self.d), dtype=self.torch.float32, device="cuda")
        hwkv.hwkv_decode_attn(self.cache, 0, self.dev(self.Q[:, p]), self.gamma, out, self.stream)
        return out.cpu().numpy()

    def oracle(self, b, qh, positions):
        """[len(positions), d] outputs of query head qh of row b."""
        h = qh // self.G
        W = self.windows[h]
        hi = max(positions) + 1
        Qr = self.Q[b, positions, qh]
        if self.fmt == BF16:
            O, sp = oracle.window_attention_bf16(Qr, positions, self.K[b, :hi, h],
                                                 self.V[b, :hi, h], W, self.gamma)
        else:
            (Kc, Ks), (Vc, Vs) = self.Kq[b][h], self.Vq[b][h]
            O, sp = oracle.window_attention_fp8(Qr, positions, Kc[:hi], Ks[:hi], Vc[:hi], Vs[:hi],
                                                W, self.gamma)
        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
        return O

    def check_rings(self):
        t = self.t()
        for b in range(self.B):
            for h in range(self.Hkv):
                cap = hwkv.hwkv_ring_capacity(self.cache, 0, h)
                pos = oracle.ring_positions(t, cap)
                kr, vr = hwkv.hwkv_debug_copy_ring(self.cache, 0, b, h, self.d, self.fmt)
                held = pos >= 0
                if self.fmt == BF16:
                    assert np.array_equal(kr[held], self.K[b, pos[held], h])
                    assert np.array_equal(vr[held], self.V[b, pos[held], h])
                else:
                    ks, vs = hwkv.hwkv_debug_copy_scales(self.cache, 0, b, h)
                    (Kc, Ks), (Vc, Vs) = self.Kq[b][h], self.Vq[b][h]
                    assert np.array_equal(kr[held], Kc[pos[held]])
                    assert np.array_equal(vr[held], Vc[pos[held]])
                    assert np.array_equal(ks[held].view(np.uint32), Ks[pos[held]].view(np.uint32))
                    assert np.array_equal(vs[held].view(np.uint32), Vs[pos[held]].view(np.uint32))
                assert not kr[~held].any() and not vr[~held].any(), "unwritten slots stay zero"


@pytest.mark.parametrize("d,fmt", [(128, BF16), (256, BF16), (128, FP8), (256, FP8)])
def test_prefill_high_dynamic_range(d, fmt):
    # two chunks, the second longer than the 300-token window; spikes late in each
    # chunk (a row's maximum jumps inside a late key tile) and one early one
    chunks = [600, 520]
    T = sum(chunks)
    r = ArrayRun(1, 8, 2, d, [0, 300], T, fmt, seed=31, spikes=[37, 455, 590, 1001, 1100])
    try:
        t0 = 0
        for n in chunks:
            out = r.prefill(n)
            pos = list(range(t0, t0 + n))
            for qh in range(r.Hq):
                assert_close(out[0, :, qh], r.oracle(0, qh, pos),
                             "hdr prefill d%d fmt%d q%d chunk@%d" % (d, fmt, qh, t0))
            t0 += n
        r.check_rings()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


@pytest.mark.parametrize("d,fmt", [(128, BF16), (256, BF16), (128, FP8), (256, FP8)])
def test_decode_high_dynamic_range(d, fmt):
    # a 5,000-token full ring split over many CTAs (segments whose maxima differ by
    # tens of units, two of them holding spikes) beside a 2,000-token window ring
    prompt, steps = 5000, 3
    Hq = 12 if d == 256 else 16
    r = ArrayRun(2, Hq, 2, d, [0, 2000], prompt + steps + 1, fmt, seed=32,
                 spikes=[1500, 3333, 4990])
    try:
        done = 0
        while done < prompt:
            m = min(1024, prompt - done)
            r.append(m)
            done += m
        outs = [r.decode_attn()]           # the last prompt token over the current rings
        pos = [prompt - 1]
        for _ in range(steps):             # fused append + decode
            outs.append(r.decode_step())
            pos.append(r.t() - 1)
        for b in range(r.B):
            for qh in range(r.Hq):
                got = np.stack([o[b, qh] for o in outs])
                assert_close(got, r.oracle(b, qh, pos), "hdr decode d%d fmt%d b%d q%d" % (d, fmt, b, qh))
        r.check_rings()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()
