"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each check uses a construction independent of the oracle's own loop (dense
masked matrices, closed forms, special cases, brute-force simulation,
printed worked examples), chosen so that a dropped term, a sign error, an
off-by-one in the window, a transposed operand or a missing normalisation
fails at least one of them.
"""
import os

import numpy as np
import pytest

import hwkv_gen
import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _bf16_bits(x):
    """float64 -> bf16 bits by round-to-nearest-even (test-side helper)."""
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def _rand_bf16(rng, shape, scale=1.0):
    return _bf16_bits(rng.standard_normal(shape) * scale)


def _dense_masked(Q, pos, K, V, W, gamma):
    """Brute force: the whole score matrix, masked entries set to -inf.
    Masked iff s > p (causal) or, for a finite window, p - s >= W."""
    Qf = hwkv_gen.bf16_bits_to_float(Q)
    Kf = hwkv_gen.bf16_bits_to_float(K)
    Vf = hwkv_gen.bf16_bits_to_float(V)
    T = Kf.shape[0]
    S = gamma * (Qf @ Kf.T)
    s_idx = np.arange(T)[None, :]
    p_idx = np.asarray(pos)[:, None]
    mask = s_idx > p_idx
    if W != oracle.FULL:
        mask |= (p_idx - s_idx) >= W
    S = np.where(mask, -np.inf, S)
    S = S - S.max(axis=1, keepdims=True)
    P = np.exp(S)
    P /= P.sum(axis=1, keepdims=True)
    return P @ Vf


@pytest.fixture(scope="module")
def data():
    rng = np.random.default_rng(7)
    T, d = 97, 24
    K = _rand_bf16(rng, (T, d))
    V = _rand_bf16(rng, (T, d), 1.5)
    Q = _rand_bf16(rng, (T, d))
    return Q, K, V


GAMMA = 0.37


def test_full_head_equals_dense_causal(data):
    Q, K, V = data
    pos = np.arange(K.shape[0])
    O, sp = oracle.window_attention_bf16(Q, pos, K, V, oracle.FULL, GAMMA)
    ref = _dense_masked(Q, pos, K, V, oracle.FULL, GAMMA)
    np.testing.assert_allclose(O, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(sp, 1.0, rtol=0, atol=1e-12)


@pytest.mark.parametrize("W", [1, 2, 5, 16, 50, 96])
def test_window_head_equals_dense_recent_mask(data, W):
    Q, K, V = data
    pos = np.arange(K.shape[0])
    O, sp = oracle.window_attention_bf16(Q, pos, K, V, W, GAMMA)
    ref = _dense_masked(Q, pos, K, V, W, GAMMA)
    np.testing.assert_allclose(O, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(sp, 1.0, rtol=0, atol=1e-12)


def test_window_ge_context_is_full_bitwise(data):
    """Sec. 3.1: any w >= C is equivalent to full."""
    Q, K, V = data
    T = K.shape[0]
    pos = np.arange(T)
    O0, _ = oracle.window_attention_bf16(Q, pos, K, V, oracle.FULL, GAMMA)
    for W in (T, T + 1, 10 ** 9):
        O1, _ = oracle.window_attention_bf16(Q, pos, K, V, W, GAMMA)
        assert np.array_equal(O0, O1)


def test_window_one_returns_own_value(data):
    """J_p(1) = {p}: the single weight is 1, the output is v_p exactly."""
    Q, K, V = data
    pos = np.arange(K.shape[0])
    O, _ = oracle.window_attention_bf16(Q, pos, K, V, 1, GAMMA)
    np.testing.assert_array_equal(O, hwkv_gen.bf16_bits_to_float(V))


def test_identical_keys_give_window_mean():
    """All keys equal: every weight is 1/|J|, the output is the mean of V over J_p(W)."""
    rng = np.random.default_rng(3)
    T, d, W = 40, 8, 7
    k = _rand_bf16(rng, (1, d))
    K = np.repeat(k, T, axis=0)
    V = _rand_bf16(rng, (T, d))
    Q = _rand_bf16(rng, (T, d))
    pos = np.arange(T)
    O, _ = oracle.window_attention_bf16(Q, pos, K, V, W, 1.0)
    Vf = hwkv_gen.bf16_bits_to_float(V)
    for p in range(T):
        lo = max(0, p - W + 1)
        np.testing.assert_allclose(O[p], Vf[lo:p + 1].mean(axis=0), rtol=0, atol=1e-12)


def test_dominant_logit_selects_its_value():
    """One key aligned with q and large gamma: softmax concentrates on it (sign of z)."""
    rng = np.random.default_rng(5)
    n, d = 30, 16
    q = rng.standard_normal(d)
    K = rng.standard_normal((n, d)) * 0.01
    K[11] = q / np.linalg.norm(q)
    V = rng.standard_normal((n, d))
    o, pi = oracle.attend(q, K, V, 200.0)
    assert pi.argmax() == 11 and pi[11] > 1 - 1e-9
    np.testing.assert_allclose(o, V[11], atol=1e-8)
    o2, pi2 = oracle.attend(q, K, V, -200.0)  # negated logits avoid that key
    assert pi2[11] < 1e-9


def test_gamma_and_operand_orientation():
    """Closed form for two keys: pi_0 = 1 / (1 + exp(gamma q.(k1 - k0)))."""
    q = np.array([1.0, 2.0, -0.5])
    K = np.array([[0.3, -0.1, 0.2], [-0.4, 0.5, 1.0]])
    V = np.array([[1.0, 0.0, 2.0], [0.0, 3.0, -1.0]])
    g = 0.8
    o, pi = oracle.attend(q, K, V, g)
    p0 = 1.0 / (1.0 + np.exp(g * (q @ K[1] - q @ K[0])))
    np.testing.assert_allclose(pi, [p0, 1 - p0], atol=1e-15)
    np.testing.assert_allclose(o, p0 * V[0] + (1 - p0) * V[1], atol=1e-15)


def test_key_order_does_not_matter():
    rng = np.random.default_rng(11)
    n, d = 50, 12
    q, K, V = rng.standard_normal(d), rng.standard_normal((n, d)), rng.standard_normal((n, d))
    perm = rng.permutation(n)
    o1, _ = oracle.attend(q, K, V, 0.5)
    o2, _ = oracle.attend(q, K[perm], V[perm], 0.5)
    np.testing.assert_allclose(o1, o2, atol=1e-13)


@pytest.mark.parametrize("W", [3, 20, 60])
def test_truncation_identity_and_bound(data, W):
    """App. A.1, Eq. local-attention-bound: o_F = (1 - m_w) o_w + m_w mu_wbar and
    ||o_F - o_w|| = m_w ||mu_wbar - mu_w|| <= m_w Delta_V, with the full-history
    weights alpha computed here independently of the oracle."""
    Q, K, V = data
    T = K.shape[0]
    Qf, Kf, Vf = (hwkv_gen.bf16_bits_to_float(x) for x in (Q, K, V))
    for p in (W + 5, T - 1):
        oF, _ = oracle.window_attention_bf16(Q[p:p + 1], [p], K, V, oracle.FULL, GAMMA)
        oW, _ = oracle.window_attention_bf16(Q[p:p + 1], [p], K, V, W, GAMMA)
        z = GAMMA * (Kf[:p + 1] @ Qf[p])
        a = np.exp(z - z.max())
        a /= a.sum()
        lo = p - W + 1
        omitted = np.arange(p + 1) < lo
        m = a[omitted].sum()
        mu_bar = (a[omitted, None] * Vf[:p + 1][omitted]).sum(0) / m
        np.testing.assert_allclose(oF[0], (1 - m) * oW[0] + m * mu_bar, atol=1e-12)
        dV = max(np.linalg.norm(Vf[r] - Vf[s]) for r in range(lo, p + 1) for s in range(lo))
        gap = np.linalg.norm(oF[0] - oW[0])
        np.testing.assert_allclose(gap, m * np.linalg.norm(mu_bar - oW[0]), rtol=1e-9)
        assert gap <= m * dV + 1e-12


def test_generator_backed_oracle_matches_array_oracle():
    """The regenerate-on-demand path computes the same definition as the array path."""
    g = hwkv_gen.desc(seed=9, per_head_scale=True)
    layer, B, T, Hkv, G, d = 2, 2, 70, 2, 3, 32
    K = hwkv_gen.fill_host(g, hwkv_gen.K, layer, B, 0, T, Hkv, d)
    V = hwkv_gen.fill_host(g, hwkv_gen.V, layer, B, 0, T, Hkv, d)
    Q = hwkv_gen.fill_host(g, hwkv_gen.Q, layer, B, 0, T, Hkv * G, d)
    pos = np.array([0, 1, 17, 40, 69])
    for b in range(B):
        for h in range(Hkv):
            for W in (oracle.FULL, 9):
                qh = h * G + 1
                O1, _ = oracle.window_attention_bf16(Q[b, pos, qh], pos, K[b, :, h], V[b, :, h],
                                                     W, 0.2)
                O2, _ = oracle.window_attention_gen(g, layer, b, h, [qh] * len(pos), pos, d, W,
                                                    0.2)
                np.testing.assert_array_equal(O1, O2)


# ------------------------------------------------------------------ rings

@pytest.mark.parametrize("cap", [1, 3, 8, 128])
def test_ring_positions_match_write_simulation(cap):
    """Brute force: write positions 0..t-1 one by one into slot p mod cap."""
    for t in [0, 1, cap - 1, cap, cap + 1, 2 * cap, 3 * cap + 2, 517]:
        if t < 0:
            continue
        sim = [-1] * cap
        for p in range(t):
            sim[p % cap] = p
        assert list(oracle.ring_positions(t, cap)) == sim
        held = sorted(x for x in sim if x >= 0)
        assert held == list(range(max(0, t - cap), t))  # the latest min(t, cap) states


def test_ring_expected_contents_from_generator():
    g = hwkv_gen.desc(seed=1)
    cap, t, d = 5, 12, 8
    ring = oracle.ring_expected_gen(g, hwkv_gen.K, 0, 0, 1, d, t, cap)
    for j in range(cap):
        p = max(q for q in range(t) if q % cap == j)
        assert [hwkv_gen.one(g, hwkv_gen.K, 0, 0, 1, p, i) for i in range(d)] == list(ring[j])
    ring0 = oracle.ring_expected_gen(g, hwkv_gen.K, 0, 0, 1, d, 3, cap)
    assert not ring0[3:].any()


# ------------------------------------------------------------- accounting

def _golden_rows(name):
    rows = []
    for line in open(os.path.join(GOLD, name)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        rows.append([f.strip() for f in line.split("|")])
    return rows


def test_residency_worked_examples():
    rows = _golden_rows("residency_worked_examples.txt")
    assert len(rows) == 4
    for name, wins, C, dims, bytes_, expect in rows:
        W = [int(x) for x in wins.split(",")]
        C = int(C)
        dK, dV = (int(x) for x in dims.split())
        bK, bV = (int(x) for x in bytes_.split())
        key, val = expect.split("=")
        if key == "rate":
            assert oracle.normalized_rate(W, C, dK, dV, bK, bV) == pytest.approx(float(val),
                                                                                 abs=1e-15)
        elif key == "rate_pct_2dp":
            assert round(100 * oracle.normalized_rate(W, C, dK, dV, bK, bV), 2) == float(val)
        elif key == "bytes":
            assert oracle.nominal_storage(W, C, dK, dV, bK, bV) == int(val)
        else:
            raise AssertionError(name)


def test_retained_tokens_definition():
    assert oracle.retained_tokens(oracle.FULL, 1000) == 1000
    assert oracle.retained_tokens(100, 1000) == 100
    assert oracle.retained_tokens(5000, 1000) == 1000
    # Eq. nominal-storage sums units and scales with precision and batch
    W = [0, 16384, 4096, 1024]
    n1 = oracle.nominal_storage(W, 33024, 256, 256, 2, 2, 1)
    assert n1 == (33024 + 16384 + 4096 + 1024) * 1024
    assert oracle.nominal_storage(W, 33024, 256, 256, 1, 1, 3) == 3 * n1 // 2


def test_window_lo():
    assert oracle.window_lo(0, oracle.FULL) == 0
    assert oracle.window_lo(10, 1) == 10
    assert oracle.window_lo(10, 11) == 0
    assert oracle.window_lo(10, 4) == 7


# -------------------------------------------------------------- generator

def test_splitmix64_published_vector():
    vals = [int(x) for x in open(os.path.join(GOLD, "splitmix64_seed1234567.txt"))
            if x.strip() and not x.startswith("#")]
    assert [hwkv_gen.splitmix64_out(1234567, j) for j in range(1, 6)] == vals


def test_generator_distribution_and_scale():
    g = hwkv_gen.desc(seed=0)
    x = hwkv_gen.bf16_bits_to_float(hwkv_gen.fill_host(g, hwkv_gen.K, 0, 2, 0, 4096, 2, 64))
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1) < 0.01
    gs = hwkv_gen.desc(seed=0, per_head_scale=True)
    scales = [hwkv_gen.head_scale(gs, hwkv_gen.K, l, h) for l in range(8) for h in range(8)]
    assert min(scales) >= 0.5 and max(scales) < 2.0
    assert hwkv_gen.head_scale(gs, hwkv_gen.Q, 0, 0) == 1.0
    y = hwkv_gen.bf16_bits_to_float(hwkv_gen.fill_host(gs, hwkv_gen.K, 3, 1, 0, 8192, 4, 32))
    for h in range(4):
        s = hwkv_gen.head_scale(gs, hwkv_gen.K, 3, h)
        assert abs(y[0, :, h].std() / s - 1) < 0.03


def test_generator_sub_fill_matches_full_fill():
    g = hwkv_gen.desc(seed=4, per_head_scale=True)
    full = hwkv_gen.fill_host(g, hwkv_gen.V, 2, 3, 10, 20, 5, 16)
    sub = hwkv_gen.fill_host_sub(g, hwkv_gen.V, 2, 2, 10, 20, 1, 3, 16)
    assert np.array_equal(sub, full[2, :, 1:4])
