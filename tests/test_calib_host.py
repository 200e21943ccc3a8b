"""Host-only checks of the library's SeqCalib selection entry points against the
oracle (no GPU): threshold selection (Eq. threshold-selection), the budget
selector (Eq. budget-selector), and calib argument validation."""
import numpy as np
import pytest

import oracle
import paper_2609_02029_gb300 as hwkv


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_02029_gb300 import build
    build.build()


def test_calib_select_matches_oracle():
    rng = np.random.default_rng(1)
    W = [512, 2048, 8192, 32768]
    for _ in range(100):
        H = int(rng.integers(1, 9))
        S = rng.uniform(0.9, 1.0, size=(H, len(W)))
        tau = float(rng.uniform(0.9, 1.0))
        C = int(rng.choice([1000, 10000, 131072]))
        got = hwkv.hwkv_calib_select(S, W, C, tau)
        want = [oracle.select_window(S[h], W, C, tau) for h in range(H)]
        assert list(got) == want


def test_budget_select_matches_oracle():
    rng = np.random.default_rng(2)
    for _ in range(200):
        G = int(rng.integers(0, 7))
        beta = rng.choice([0.3, 0.5, 0.69, 0.86, 0.96], size=G)
        phi = rng.choice([0.99, 0.995, 0.998], size=G)
        budget = float(rng.choice([0.2, 0.6, 0.9, 1.0]))
        assert hwkv.hwkv_budget_select(beta, phi, budget) == oracle.budget_select(beta, phi, budget)


@pytest.mark.parametrize("kw", [
    dict(windows=[100, 50]),           # not increasing
    dict(windows=[0, 50]),             # non-positive
    dict(positions=[[5, 9999]]),       # outside [0, T)
    dict(windows=list(range(1, 10))),  # more than 8 windows
    dict(n_kv_heads=2, n_q_heads=7),   # not a multiple of the KV heads
])
def test_calib_validation(kw):
    args = dict(n_seq=1, n_pos=2, n_kv_heads=1, n_q_heads=4, head_dim=64, T=1000,
                windows=[16, 64], positions=[[5, 900]])
    args.update(kw)
    d = hwkv.make_calib_desc(**args)
    with pytest.raises(hwkv.HwkvError):
        hwkv.hwkv_calib_workspace_bytes(d)
