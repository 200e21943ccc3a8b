"""Full-size parity for the two large workloads, in the launch configuration
bench.py times (hwkv_decode_step: the new token's append fused into the decode
launch, work planned on the GPU): the 112K-context, 16-layer, batch-16 decode
(39 GB of rings) and the 161K-context budget sweep (25/50/75/100% of all-full
residency, up to 43 GB). The whole prompt is appended through the C ABI; decode
steps run over every layer. Seeded samples of (layer, batch row, KV head) units
are checked against the oracle at the first and last step, sampled rings
bit-exactly, and residency exactly at every step."""
import numpy as np
import pytest

import oracle
import paper_2609_02029_gb300 as hwkv
from hwkv_gen import workloads
from harness import Run, assert_close, check_ring_unit, oracle_unit_decode

pytestmark = pytest.mark.gpu


def _units(wl, rng, k):
    picks = {(0, 0, h) for h in range(wl.n_kv_heads)}
    picks |= {(wl.n_layers - 1, wl.batch - 1, h) for h in range(wl.n_kv_heads)}
    while len(picks) < k:
        picks.add((int(rng.integers(wl.n_layers)), int(rng.integers(wl.batch)),
                   int(rng.integers(wl.n_kv_heads))))
    return sorted(picks)


def _run_decode_workload(wl, steps, n_units, seed):
    import torch
    r = Run.for_workload(wl)
    rng = np.random.default_rng(seed)
    try:
        for layer in range(wl.n_layers):
            r.fill(layer, wl.prompt, chunk=4096)
        torch.cuda.synchronize()
        units = _units(wl, rng, n_units)
        for step in range(steps):
            outs = [r.decode_step_fused(layer) for layer in range(wl.n_layers)]
            t = wl.prompt + step + 1
            assert hwkv.hwkv_residency_bytes(r.cache) == oracle.nominal_storage(
                wl.windows, t, wl.head_dim, wl.head_dim, 2, 2, wl.batch)
            if step in (0, steps - 1):
                for (layer, b, h) in units:
                    got = outs[layer][b, h * wl.group:(h + 1) * wl.group].cpu().numpy()
                    want = oracle_unit_decode(r, layer, b, h, t - 1)
                    assert_close(got, want, "%s step %d unit (%d,%d,%d)" % (wl.name, step, layer, b, h))
        for (layer, b, h) in units[:6]:
            check_ring_unit(r, layer, b, h)
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_layers16_112k_decode():
    _run_decode_workload(workloads.make("layers16_112k"), steps=3, n_units=24, seed=3)


@pytest.mark.parametrize("budget", [0.25, 0.5, 0.75, 1.0])
def test_budget161k_decode(budget):
    wl = workloads.make("budget161k", budget)
    assert abs(oracle.normalized_rate(wl.windows, wl.max_ctx, 256, 256) - budget) < 0.02
    _run_decode_workload(wl, steps=2, n_units=10, seed=int(budget * 100))
