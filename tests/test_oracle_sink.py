"""Pins of the oracle's sink + recent window (the static sink--recent policy of
the paper's StreamingLLM control: S sink tokens plus a W-token recent window;
a query at p reads J = {0..S-1} U [max(0, p-W+1), p], limited to <= p).
Pinned against the already pinned plain window (S = 0), full attention when
nothing falls outside J, a probe that reads J off the output, the ring holding
exactly what the newest query reads, and the retained-count closed form."""
import numpy as np
import pytest

import hwkv_gen
import oracle


def bf16_bits(x):
    return (np.asarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


@pytest.mark.parametrize("W,p", [(5, 3), (5, 40), (64, 200), (1, 17)])
def test_no_sinks_is_the_plain_window(W, p):
    g = hwkv_gen.desc(3, True)
    a, _ = oracle.sink_attention_gen(g, 0, 1, 2, [4, 5], [p, p], 64, W, 0, 0.125)
    b, _ = oracle.window_attention_gen(g, 0, 1, 2, [4, 5], [p, p], 64, W, 0.125)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-14)


@pytest.mark.parametrize("W,S,p", [(3, 4, 6), (10, 1, 9), (2, 30, 25), (0, 4, 50)])
def test_everything_visible_is_full_attention(W, S, p):
    # p - W + 1 <= S (or W = full): J is the whole prefix [0, p]
    g = hwkv_gen.desc(5, False)
    a, sp = oracle.sink_attention_gen(g, 1, 0, 0, [0], [p], 128, W, S, 0.0884)
    b, _ = oracle.window_attention_gen(g, 1, 0, 0, [0], [p], 128, 0, 0.0884)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-14)
    np.testing.assert_allclose(sp, 1.0, atol=1e-12)


@pytest.mark.parametrize("W,S", [(3, 2), (7, 5), (1, 1), (4, 0), (20, 3)])
def test_uniform_logits_reveal_the_read_set(W, S):
    # q = 0 gives equal logits: o = mean of the V rows in J; with V row k = basis
    # vector k, o[k] = 1/|J| exactly for k in J and 0 elsewhere
    T = 32
    V = bf16_bits(np.eye(T, dtype=np.float32))
    K = bf16_bits(np.random.default_rng(1).standard_normal((T, T)).astype(np.float32))
    Q = np.zeros((T, T), dtype=np.uint16)
    O, _ = oracle.sink_attention_bf16(Q, list(range(T)), K, V, W, S, 0.3)
    for p in range(T):
        lo = oracle.window_lo(p, W)  # the plain window, pinned on its own
        want = {k for k in range(p + 1) if k >= lo} | set(range(min(S, p + 1)))
        got = {k for k in range(T) if O[p, k] != 0.0}
        assert got == want, (p, sorted(got), sorted(want))
        np.testing.assert_allclose(O[p, sorted(want)], 1.0 / len(want), rtol=1e-15)


@pytest.mark.parametrize("W,S", [(3, 4), (5, 1), (1, 3), (16, 16)])
def test_ring_holds_exactly_what_the_newest_query_reads(W, S):
    for t in range(1, 3 * (W + S) + 5):
        held = oracle.sink_ring_positions(t, W, S)
        held = sorted(int(x) for x in held if x >= 0)
        assert held == list(oracle.sink_positions(t - 1, W, S))
        assert len(held) == oracle.sink_retained_tokens(W, S, t)
        # a position never moves: sink slots hold their own index
        ring = oracle.sink_ring_positions(t, W, S)
        for j in range(min(S, t)):
            assert ring[j] == j


def test_retained_closed_form():
    assert oracle.sink_retained_tokens(90364, 4, 131072) == 90368  # the paper's 4 + 90,364 cache
    assert oracle.sink_retained_tokens(90364, 4, 65536) == 65536
    assert oracle.sink_retained_tokens(0, 4, 1000) == 1000          # full history
