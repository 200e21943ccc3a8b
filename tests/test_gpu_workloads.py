"""Parity on the full-size workloads, through the C ABI, in the launch
configuration the benchmark times. Every decode output of the small workloads
is checked; prefill rows and the large workloads are sampled (seeded)."""
import numpy as np
import pytest

import paper_2609_02029_gb300 as hwkv
from hwkv_gen import workloads
from harness import Run, assert_close

pytestmark = pytest.mark.gpu


def _prefill_rows(n, t0, W_list, rng, k=48):
    rows = {0, 1, 2, n - 1, n - 2, n // 2}
    for W in W_list:
        if W:
            for x in (W - 2, W - 1, W, W + 1):
                if 0 <= x < n:
                    rows.add(x)
    rows |= set(rng.integers(0, n, size=k).tolist())
    return sorted(r for r in rows if 0 <= r < n)


@pytest.mark.parametrize("name", ["tiny", "single32k"])
def test_prompt_then_every_decode_output(name):
    wl = workloads.make(name)
    r = Run.for_workload(wl)
    rng = np.random.default_rng(0)
    try:
        done = 0
        while done < wl.prompt:
            n = min(wl.chunk, wl.prompt - done)
            out = r.prefill(0, n).cpu().numpy()
            rows = _prefill_rows(n, done, wl.windows, rng, k=16)
            for qh in range(0, wl.n_q_heads, max(1, wl.group // 2)):
                assert_close(out[0, rows, qh], r.oracle_rows(0, 0, qh, [done + i for i in rows]),
                             "%s prefill q%d chunk@%d" % (name, qh, done))
            done += n
        r.check_rings(0)
        outs = []
        for i in range(wl.decode_steps):
            outs.append(r.decode_step(0).cpu().numpy())
            assert hwkv.hwkv_residency_bytes(r.cache, 0) == __import__("oracle").nominal_storage(
                wl.windows, wl.prompt + i + 1, wl.head_dim, wl.head_dim, 2, 2, wl.batch)
        pos = list(range(wl.prompt, wl.prompt + wl.decode_steps))
        for qh in range(wl.n_q_heads):
            got = np.stack([o[0, qh] for o in outs])
            assert_close(got, r.oracle_rows(0, 0, qh, pos), "%s decode q%d" % (name, qh))
        r.check_rings(0)
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_prefill64k_sampled_rows():
    wl = workloads.make("prefill64k")
    r = Run.for_workload(wl)
    rng = np.random.default_rng(1)
    try:
        done = 0
        while done < wl.prompt:
            n = wl.chunk
            out = r.prefill(0, n).cpu().numpy()
            rows = _prefill_rows(n, done, wl.windows, rng, k=8) if done else list(range(0, n, 61))
            for b in range(wl.batch):
                heads = [int(x) for x in rng.choice(wl.n_q_heads, size=6, replace=False)]
                for qh in heads:
                    # chunk 0: every row for two of the sampled heads
                    rr = list(range(n)) if (done == 0 and qh in heads[:2]) else rows
                    assert_close(out[b, rr, qh],
                                 r.oracle_rows(0, b, qh, [done + i for i in rr]),
                                 "prefill64k b%d q%d chunk@%d" % (b, qh, done))
            done += n
        r.check_rings(0)
        r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()
