"""Full-size parity for the two large decode workloads, at their own lengths, in
the launch configuration bench.py times (hwkv_decode_step: the new token's append
fused into the decode launch, work planned on the GPU):

  - layers16_112k: 16 layers, batch 16, 24q/4kv, head_dim 256, 112K context
    (39 GB of rings), all 128 decode steps;
  - budget161k at 25/50/75/100% of all-full residency: 16 layers, batch 4, 161K
    context (up to 43 GB), all 64 decode steps of each budget.

The whole prompt is appended through the C ABI. Every (layer, batch row, KV
head) unit is checked against the fp64 oracle (all G query heads) at the first
and the last decode step; at every other step 16 seeded (layer, batch row)
pairs with all their KV heads. Residency is exact at every step
and every ring is compared bit-exactly with the oracle's ring at the end. The
oracle runs on the host cores (one oracle thread per worker) while the GPU
steps continue."""
import os
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
import paper_2609_02029_gb300 as hwkv
from hwkv_gen import workloads
from harness import Run, assert_close, check_ring_unit, oracle_unit_decode

pytestmark = pytest.mark.gpu


class OraclePool:
    """Worker threads for oracle checks; each sets its own oracle thread count to
    one (the pool supplies the parallelism)."""

    def __init__(self):
        self.local = threading.local()
        self.ex = ThreadPoolExecutor(max_workers=os.cpu_count() or 1)
        self.futures = []

    def _one_thread(self):
        if not getattr(self.local, "set", False):
            oracle.set_threads(1)
            self.local.set = True

    def submit(self, fn, *args):
        def work():
            self._one_thread()
            return fn(*args)
        self.futures.append(self.ex.submit(work))

    def drain(self):
        try:
            for f in self.futures:
                f.result()
        finally:
            self.ex.shutdown(wait=True, cancel_futures=True)


def _check_unit(r, wl, layer, b, h, p, got, what):
    want = oracle_unit_decode(r, layer, b, h, p)
    assert_close(got, want, "%s unit (%d,%d,%d) p%d" % (what, layer, b, h, p))


def _run_decode_workload(wl, pairs_per_step, seed):
    import torch
    r = Run.for_workload(wl)
    rng = np.random.default_rng(seed)
    pool = OraclePool()
    L, B, H, G = wl.n_layers, wl.batch, wl.n_kv_heads, wl.group
    all_units = [(l, b, h) for l in range(L) for b in range(B) for h in range(H)]
    try:
        for layer in range(L):
            r.fill(layer, wl.prompt, chunk=4096)
        torch.cuda.synchronize()
        steps = wl.decode_steps
        for step in range(steps):
            outs = torch.stack([r.decode_step_fused(layer) for layer in range(L)])
            t = wl.prompt + step + 1
            assert hwkv.hwkv_residency_bytes(r.cache) == oracle.nominal_storage(
                wl.windows, t, wl.head_dim, wl.head_dim, 2, 2, B), "residency at t=%d" % t
            if step in (0, steps - 1):
                units = all_units
            else:
                picks = rng.choice(L * B, size=pairs_per_step, replace=False)
                units = [(int(x) // B, int(x) % B, h) for x in picks for h in range(H)]
            host = outs.cpu().numpy()
            for (layer, b, h) in units:
                pool.submit(_check_unit, r, wl, layer, b, h, t - 1,
                            host[layer, b, h * G:(h + 1) * G].copy(), "%s step %d" % (wl.name, step))
        hwkv.hwkv_sync_check(r.cache)
        for (layer, b, h) in all_units:
            pool.submit(check_ring_unit, r, layer, b, h)
        pool.drain()
    finally:
        r.close()


def test_layers16_112k_decode():
    wl = workloads.make("layers16_112k")
    assert wl.decode_steps == 128
    _run_decode_workload(wl, pairs_per_step=16, seed=3)


@pytest.mark.parametrize("budget", [0.25, 0.5, 0.75, 1.0])
def test_budget161k_decode(budget):
    wl = workloads.make("budget161k", budget)
    assert wl.decode_steps == 64
    assert abs(oracle.normalized_rate(wl.windows, wl.max_ctx, 256, 256) - budget) < 0.02
    _run_decode_workload(wl, pairs_per_step=16, seed=int(budget * 100))
