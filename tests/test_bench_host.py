"""Host-side pins for the quantities bench.py divides by: the algorithmic flops of a
prefill chunk (every visible (query, key) pair, Sec. 3.2's window J_t(w) per KV head)
and the algorithmic bytes of a decode step (every resident K/V row read once, which is
the residency of Sec. 3.1, Eq. nominal-storage). Each is checked against an independent
count: brute-force enumeration of visible pairs, and the oracle's storage formula."""
import numpy as np
import pytest

import bench
import oracle
from hwkv_gen import workloads


class _Wl:
    """A minimal workload description with the fields bench's counters read."""

    def __init__(self, windows, n_kv_heads, group, head_dim, batch, max_ctx, n_layers=1):
        self.windows, self.n_kv_heads, self.group = list(windows), n_kv_heads, group
        self.head_dim, self.batch, self.max_ctx, self.n_layers = head_dim, batch, max_ctx, n_layers
        self.n_q_heads = n_kv_heads * group


def _brute_prefill_flops(wl, t0, n):
    """4 d G flops (QK^T and PV, multiply-add = 2) per visible pair, pairs enumerated."""
    total = 0
    for h in range(wl.n_kv_heads):
        W = wl.windows[h]
        full = W == 0 or W >= wl.max_ctx
        pairs = 0
        for p in range(t0, t0 + n):
            lo = 0 if full else max(0, p - W + 1)
            pairs += sum(1 for s in range(lo, p + 1))  # keys s in [lo, p]
        total += pairs * wl.group * 4 * wl.head_dim * wl.batch
    return total


def _vector_prefill_flops(wl, t0, n):
    """The same count with numpy, for full-size prompts."""
    p = np.arange(t0, t0 + n, dtype=np.int64)
    total = 0
    for h in range(wl.n_kv_heads):
        W = wl.windows[h]
        full = W == 0 or W >= wl.max_ctx
        keys = p + 1 if full else np.minimum(p + 1, W)
        total += int(keys.sum()) * wl.group * 4 * wl.head_dim * wl.batch
    return total


@pytest.mark.parametrize("windows,t0,n", [
    ([0, 1], 0, 7),            # full head and a one-token window
    ([5, 0, 3], 0, 12),        # chunk longer than the windows
    ([5, 16, 40], 9, 20),      # window edges inside the chunk
    ([64, 200], 100, 1),       # one query, window < t0 < max_ctx
    ([300, 7], 250, 50),       # W >= max_ctx counts as full
])
def test_prefill_flops_matches_enumeration(windows, t0, n):
    wl = _Wl(windows, len(windows), group=3, head_dim=8, batch=2, max_ctx=300)
    assert bench.prefill_flops(wl, t0, n) == _brute_prefill_flops(wl, t0, n)


@pytest.mark.parametrize("name", ["prefill64k", "single32k"])
def test_prefill_flops_full_prompts(name):
    wl = workloads.make(name)
    total = sum(bench.prefill_flops(wl, c * wl.chunk, wl.chunk) for c in range(wl.prompt // wl.chunk))
    want = sum(_vector_prefill_flops(wl, c * wl.chunk, wl.chunk) for c in range(wl.prompt // wl.chunk))
    assert total == want
    if name == "prefill64k":
        assert total == 49959781007360  # the figure the prefill lines divide by


@pytest.mark.parametrize("t", [1, 511, 512, 513, 114688])
def test_decode_bytes_equal_residency(t):
    wl = workloads.make("layers16_112k")
    per_layer = bench.decode_bytes(wl, wl.max_ctx, t)
    d = wl.head_dim
    assert sum(per_layer) == oracle.nominal_storage(wl.windows, t, d, d, 2, 2, wl.batch)
    for layer in range(wl.n_layers):
        ws = wl.windows[layer * wl.n_kv_heads:(layer + 1) * wl.n_kv_heads]
        assert per_layer[layer] == oracle.nominal_storage(ws, t, d, d, 2, 2, wl.batch)
    # the oracle sample's key count is the same sum, in rows
    keys = sum(u[4] for u in bench.step_keys(wl, wl.max_ctx, t))
    assert keys * 4 * d == sum(per_layer)


def test_decode_bytes_8_bit_format():
    wl = workloads.make("layers16_112k")
    t = 100000
    bf16 = sum(bench.decode_bytes(wl, wl.max_ctx, t))
    fp8 = sum(bench.decode_bytes(wl, wl.max_ctx, t, fp8=True))
    d = wl.head_dim
    # E4M3 codes (1 byte per channel) plus one fp32 scale per K and per V row
    assert fp8 * 4 * d == bf16 * 2 * (d + 4)


def test_oracle_layer_steps_cover_every_unit():
    """The oracle baseline times whole layer-steps: every (batch row, KV head) unit
    of the layer, each over its whole retained window at position p."""
    import oracle
    wl = workloads.make("tiny")
    orc = bench.OracleLayerSteps(wl, wl.max_ctx)
    p = 300
    sec, units, keys = orc.run_layer(0, p)
    assert units == wl.batch * wl.n_kv_heads
    assert keys == wl.batch * sum(p - oracle.window_lo(p, 0 if W >= wl.max_ctx else W) + 1
                                  for W in wl.windows)
    assert sec > 0


def test_secondary_line_rates():
    """The secondary workload line divides each step's bytes by the replayed graph's
    step time and reports it against the copy bandwidth (graph_frac) beside the one
    eager layer launch (frac); the GPU run is replaced by fixed timings."""
    import argparse
    fake = {"value": 100.0, "ms": 80.0, "graph_value": 110.0, "graph_ms": 40.0, "graph_steps": 8,
            "e2e_value": 90.0, "achieved_gbs": 5000.0, "bytes_avg": 1.0e9, "dec_avg_ms": 0.2,
            "step_bytes": 3.0e9, "flush": False, "resid_bytes": 123}
    saved = bench.run_gpu
    bench.run_gpu = lambda a, wl, world, rank, local: fake
    try:
        args = argparse.Namespace(steps=96, e2e_steps=32)
        line = bench.run_secondary(args, "budget161k_r25", 1, 0, 0, 6000.0)
    finally:
        bench.run_gpu = saved
    assert line["steps"] == 32
    assert line["graph_ms_per_step"] == 40.0 / 8
    assert abs(line["graph_step_gbs"] - 3.0e9 / (5.0e-3) / 1e9) < 1e-9
    assert abs(line["graph_frac"] - line["graph_step_gbs"] / 6000.0) < 1e-12
    assert abs(line["frac"] - 5000.0 / 6000.0) < 1e-12
