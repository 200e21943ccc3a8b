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


def test_prefill64k_rows():
    """prefill64k (64K prompt in 8 chunks of 8,192, batch 2, 32q/8kv, head_dim 128):
    every row of chunk 0 for every (batch row, query head); on each later chunk
    the rows within 2 of the chunk's first and last position and of each window
    edge, plus 512 seeded random rows per (batch row, query head). The oracle runs
    over host arrays of each KV head's whole history (generated once), one oracle
    thread per worker, while the GPU continues."""
    import os
    import threading
    from concurrent.futures import ThreadPoolExecutor

    import hwkv_gen
    import oracle
    wl = workloads.make("prefill64k")
    r = Run.for_workload(wl)
    rng = np.random.default_rng(1)
    B, Hq, Hkv, d, G, n = wl.batch, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.group, wl.chunk
    K = [[hwkv_gen.fill_host_sub(r.g, hwkv_gen.K, 0, b, 0, wl.prompt, h, 1, d)[:, 0]
          for h in range(Hkv)] for b in range(B)]
    V = [[hwkv_gen.fill_host_sub(r.g, hwkv_gen.V, 0, b, 0, wl.prompt, h, 1, d)[:, 0]
          for h in range(Hkv)] for b in range(B)]
    local = threading.local()

    def check(b, qh, rows, t0, got, Q):
        if not getattr(local, "set", False):
            oracle.set_threads(1)
            local.set = True
        h = qh // G
        pos = [t0 + i for i in rows]
        want, sp = oracle.window_attention_bf16(Q, pos, K[b][h], V[b][h], r.window(0, h), r.scale)
        np.testing.assert_allclose(sp, 1.0, atol=1e-12)
        assert_close(got, want, "prefill64k b%d q%d chunk@%d (%d rows)" % (b, qh, t0, len(rows)))

    ex = ThreadPoolExecutor(max_workers=os.cpu_count() or 1)
    futures = []
    try:
        done = 0
        while done < wl.prompt:
            out = r.prefill(0, n).cpu().numpy()
            Qc = hwkv_gen.fill_host(r.g, hwkv_gen.Q, 0, B, done, n, Hq, d)
            edges = _prefill_rows(n, done, wl.windows, rng, k=0)
            for b in range(B):
                for qh in range(Hq):
                    if done == 0:
                        rows = list(range(n))
                    else:
                        rows = sorted(set(edges) | set(rng.choice(n, size=512, replace=False).tolist()))
                    futures.append(ex.submit(check, b, qh, rows, done, out[b, rows, qh].copy(),
                                             Qc[b, rows, qh].copy()))
            done += n
        r.check_rings(0)
        r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
        for f in futures:
            f.result()
    finally:
        ex.shutdown(wait=True, cancel_futures=True)
        r.close()
