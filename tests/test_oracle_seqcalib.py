"""Pins of the oracle's SeqCalib scoring and selection (App. A.2 and Sec. 3.2):
special cases of the stabilized cosine, the conditional similarity against an
independent dense-mask computation, the cosine identity and the trace error
bound, threshold selection and Prop. 1 / Cor. 1 by brute force over every
same-layer assignment, and the lexicographic budget selector by brute force."""
import itertools

import numpy as np
import pytest

import hwkv_gen
import oracle


def test_cos_eval_special_cases():
    e = oracle.EPS_COS
    assert oracle.cos_eval([0, 0, 0], [0, 0, 0]) == 1.0            # both zero
    assert oracle.cos_eval([1e-13, 0, 0], [0, -1e-13, 0]) == 1.0   # both below eps
    assert oracle.cos_eval([0, 0, 0], [1, 2, 3]) == 0.0            # exactly one zero
    assert oracle.cos_eval([3, 4], [1e-13, 0]) == 0.0
    assert oracle.cos_eval([2, 0], [5, 0]) == pytest.approx(1.0, abs=1e-15)
    assert oracle.cos_eval([2, 0], [-5, 0]) == pytest.approx(-1.0, abs=1e-15)
    assert oracle.cos_eval([1, 0], [0, 7]) == 0.0
    rng = np.random.default_rng(0)
    for _ in range(20):
        u, v = rng.standard_normal(16), rng.standard_normal(16)
        ref = u @ v / np.linalg.norm(u) / np.linalg.norm(v)
        assert oracle.cos_eval(u, v) == pytest.approx(ref, abs=1e-14)
        assert oracle.cos_eval(3 * u, 0.5 * v) == pytest.approx(ref, abs=1e-14)  # scale free
    assert oracle.cos_eval([2 * e, 0], [1, 1]) == pytest.approx(1 / np.sqrt(2), abs=1e-12)


def _bf16(x):
    f = np.asarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    return ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)


def _dense_out(Qf, pos, Kf, Vf, W, gamma):
    """Dense masked attention (masked iff s > p or, finite W, p - s >= W)."""
    T = Kf.shape[0]
    S = gamma * (Qf @ Kf.T)
    s_idx = np.arange(T)[None, :]
    p_idx = np.asarray(pos)[:, None]
    mask = s_idx > p_idx
    if W:
        mask |= (p_idx - s_idx) >= W
    S = np.where(mask, -np.inf, S)
    P = np.exp(S - S.max(axis=1, keepdims=True))
    return (P / P.sum(axis=1, keepdims=True)) @ Vf


@pytest.fixture(scope="module")
def trace():
    rng = np.random.default_rng(21)
    T, d, R = 300, 16, 24
    K = _bf16(rng.standard_normal((T, d)))
    V = _bf16(rng.standard_normal((T, d)))
    Q = _bf16(rng.standard_normal((R, d)) * 2.0)
    pos = rng.integers(200, T, size=R)
    return Q, pos, K, V


def test_conditional_similarity_matches_dense_mask(trace):
    Q, pos, K, V = trace
    W = [4, 16, 64, 299, 300, 1000]
    gamma = 0.4
    scores, cos = oracle.conditional_similarity_bf16(Q, pos, K, V, W, gamma)
    Qf, Kf, Vf = (hwkv_gen.bf16_bits_to_float(x) for x in (Q, K, V))
    of = _dense_out(Qf, pos, Kf, Vf, 0, gamma)
    for k, w in enumerate(W):
        ow = _dense_out(Qf, pos, Kf, Vf, w, gamma)
        c = (ow * of).sum(1) / np.linalg.norm(ow, axis=1) / np.linalg.norm(of, axis=1)
        np.testing.assert_allclose(cos[:, k], c, atol=1e-12)
        assert scores[k] == pytest.approx(c.mean(), abs=1e-12)
    # w >= every position + 1 is full: score exactly one (Sec. 3.1 / App. A.2)
    assert scores[W.index(300)] == 1.0 and scores[W.index(1000)] == 1.0
    assert scores.max() <= 1.0 + 1e-12


def test_cosine_identity_and_trace_error_bound(trace):
    """Eq. conditional-empirical-cosine-bound: mean ||y~w - y~F||^2 <= eta^2 + 2 B^2 (1 - S_w),
    from the pointwise ||u - v||^2 = (|u| - |v|)^2 + 2 |u| |v| (1 - cos)."""
    Q, pos, K, V = trace
    gamma = 0.4
    of, _ = oracle.window_attention_bf16(Q, pos, K, V, 0, gamma)
    for w in (2, 8, 40):
        ow, _ = oracle.window_attention_bf16(Q, pos, K, V, w, gamma)
        scores, cos = oracle.conditional_similarity_bf16(Q, pos, K, V, [w], gamma)
        nu, nv = np.linalg.norm(ow, axis=1), np.linalg.norm(of, axis=1)
        lhs = ((ow - of) ** 2).sum(1)
        np.testing.assert_allclose(lhs, (nu - nv) ** 2 + 2 * nu * nv * (1 - cos[:, 0]),
                                   rtol=1e-9, atol=1e-12)
        B = max(nu.max(), nv.max())
        eta = np.abs(nu - nv).max()
        assert lhs.mean() <= eta ** 2 + 2 * B ** 2 * (1 - scores[0]) + 1e-12
        for tau in (0.5, 0.9, 0.99):
            if scores[0] >= tau:
                assert lhs.mean() <= eta ** 2 + 2 * B ** 2 * (1 - tau) + 1e-12


def _brute_select(scores, W, C, tau):
    cands = [(min(w, C), i, w) for i, w in enumerate(W) if scores[i] >= tau]
    cands.append((C, len(W), 0))  # full: score one, last in <_W
    return min(cands)[2]


def test_threshold_selection_brute_force():
    rng = np.random.default_rng(4)
    W = [512, 2048, 8192, 32768]
    for _ in range(200):
        s = rng.uniform(0.9, 1.0, size=len(W))
        tau = rng.uniform(0.9, 1.0)
        C = int(rng.choice([1000, 5000, 20000, 131072]))
        assert oracle.select_window(s, W, C, tau) == _brute_select(list(s), W, C, tau)
    assert oracle.select_window([0.1, 0.2, 0.3, 0.4], W, 131072, 0.999) == 0   # only full
    assert oracle.select_window([1.0, 1.0, 1.0, 1.0], W, 131072, 1.0) == 512   # cheapest
    # equal costs (w >= C all cost C): <_W prefers the smaller finite window
    assert oracle.select_window([0.5, 1.0, 1.0, 1.0], W, 1500, 0.99) == 2048


def test_fixed_prefix_minimality_and_shared_window():
    """Prop. 1 and Cor. 1: per-head selection attains the minimum layer cost over
    every assignment meeting all floors; it never costs more than a shared feasible window."""
    rng = np.random.default_rng(8)
    W = [256, 1024, 4096]
    cand = W + [0]
    C = 8192
    cost = lambda w: C if w == 0 else min(w, C)
    for _ in range(50):
        H = 4
        S = rng.uniform(0.95, 1.0, size=(H, len(W)))
        tau = rng.uniform(0.95, 1.0)
        sel = [oracle.select_window(S[h], W, C, tau) for h in range(H)]
        feas = lambda h, w: w == 0 or S[h, W.index(w)] >= tau
        assert all(feas(h, sel[h]) for h in range(H))
        best = min(sum(cost(a) for a in assign)
                   for assign in itertools.product(cand, repeat=H)
                   if all(feas(h, a) for h, a in enumerate(assign)))
        assert sum(cost(a) for a in sel) == best
        for w in cand:
            if all(feas(h, w) for h in range(H)):
                assert sum(cost(a) for a in sel) <= H * cost(w)


def test_budget_selector_brute_force():
    rng = np.random.default_rng(9)
    for _ in range(300):
        G = int(rng.integers(1, 8))
        beta = rng.choice([0.25, 0.5, 0.69, 0.86, 0.96], size=G)
        phi = rng.choice([0.990, 0.995, 0.998, 0.999], size=G)
        budget = float(rng.choice([0.3, 0.7, 0.9, 1.0, 0.1]))
        feas = [g for g in range(G) if beta[g] <= budget]
        want = min(feas, key=lambda g: (-phi[g], beta[g], g)) if feas else -1
        assert oracle.budget_select(beta, phi, budget) == want
