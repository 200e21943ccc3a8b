"""Per-row lengths through the C ABI: ragged and idle rows, row-range append and
prefill, and the graph-mode decode step replayed from a captured CUDA graph.

Every row is an independent sequence, so the oracle is the same window
attention (Sec. 3.2) evaluated per row at that row's own position, and the ring
contents / residency (Sec. 3.3, Eq. nominal-storage) per row at its own length."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv
from harness import MAX_ABS, MEAN_ABS, Run, assert_close, oracle_unit_decode

pytestmark = pytest.mark.gpu


def rows_at(run, tensor, layer, positions, heads):
    """[B, heads, d] bf16: row b holds the generator's token at positions[b]
    (zeros for rows given None)."""
    torch = run.torch
    out = torch.zeros((run.B, heads, run.d), dtype=torch.bfloat16, device="cuda")
    for p in sorted({p for p in positions if p is not None}):
        full = run.gen(tensor, layer, p, 1, heads)  # every row at position p
        for b, pb in enumerate(positions):
            if pb == p:
                out[b] = full[b, 0]
    return out


def append_row(run, layer, b, n, chunk=8192):
    """Append the generator's next n tokens of row b through hwkv_append_rows."""
    done = 0
    while done < n:
        m = min(chunk, n - done)
        t = hwkv.hwkv_row_len(run.cache, layer, b)
        k = run.gen(hwkv_gen.K, layer, t, m, run.Hkv)[b:b + 1].contiguous()
        v = run.gen(hwkv_gen.V, layer, t, m, run.Hkv)[b:b + 1].contiguous()
        hwkv.hwkv_append_rows(run.cache, layer, b, 1, k, v, m, run.stream)
        done += m


def expected_step(run, layer, lens, heads_sample=None):
    """Oracle outputs [B, Hq, d] of a fused step from lengths `lens` (None = idle)."""
    want = np.zeros((run.B, run.Hq, run.d))
    for b, t in enumerate(lens):
        if t is None:
            continue
        for h in range(run.Hkv):
            if heads_sample is not None and h not in heads_sample:
                continue
            want[b, h * run.G:(h + 1) * run.G] = oracle_unit_decode(run, layer, b, h, t)
    return want


def check_rows_state(run, lens):
    for layer in range(run.L):
        for b, t in enumerate(lens[layer]):
            assert hwkv.hwkv_row_len(run.cache, layer, b) == (-1 if t is None else t)
            if t is None:
                continue
            for h in range(run.Hkv):
                kr, vr = hwkv.hwkv_debug_copy_ring(run.cache, layer, b, h, run.d)
                cap = kr.shape[0]
                r = min(t, cap)  # resident slots; a reset row keeps stale, unreachable ones
                ek = oracle.ring_expected_gen(run.g, hwkv_gen.K, layer, b, h, run.d, t, cap)
                ev = oracle.ring_expected_gen(run.g, hwkv_gen.V, layer, b, h, run.d, t, cap)
                assert np.array_equal(kr[:r], ek[:r]), "K ring (%d, %d, %d)" % (layer, b, h)
                assert np.array_equal(vr[:r], ev[:r]), "V ring (%d, %d, %d)" % (layer, b, h)
        w = run.windows[layer * run.Hkv:(layer + 1) * run.Hkv]
        want = sum(oracle.nominal_storage(w, t, run.d, run.d, 2, 2, 1)
                   for t in lens[layer] if t is not None)
        assert hwkv.hwkv_residency_bytes(run.cache, layer) == want


def test_ragged_eager_then_graph():
    # rows: fresh (0), 1, 63, 700, 1500 tokens, and one idle row
    start = [0, 1, 63, 700, 1500, None]
    run = Run(n_layers=2, batch=6, n_q_heads=8, n_kv_heads=2, head_dim=128, max_ctx=3000,
              windows=[0, 256, 64, 0], seed=11)
    torch = run.torch
    try:
        hwkv.hwkv_reset_rows(run.cache, 5, 1, idle=True, stream=run.stream)
        for layer in range(run.L):
            for b, n in enumerate(start):
                if n:
                    append_row(run, layer, b, n)
        with pytest.raises(hwkv.HwkvError):  # rows differ: no single t
            hwkv.hwkv_seq_len(run.cache, 0)
        lens = [list(start) for _ in range(run.L)]
        check_rows_state(run, lens)

        def step_inputs(layer):
            pos = lens[layer]
            return (rows_at(run, hwkv_gen.Q, layer, pos, run.Hq),
                    rows_at(run, hwkv_gen.K, layer, pos, run.Hkv),
                    rows_at(run, hwkv_gen.V, layer, pos, run.Hkv))

        # eager fused steps over ragged rows (device tile plan)
        for _ in range(2):
            for layer in range(run.L):
                q, k, v = step_inputs(layer)
                out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
                hwkv.hwkv_decode_step(run.cache, layer, q, k, v, run.scale, out, run.stream)
                got = out.cpu().numpy()
                assert_close(got, expected_step(run, layer, lens[layer]), "eager ragged step")
                assert not got[5].any()  # idle row
                lens[layer] = [None if t is None else t + 1 for t in lens[layer]]
        hwkv.hwkv_sync_check(run.cache)
        check_rows_state(run, lens)

        # one step of both layers captured once, replayed three times
        qs = [torch.empty((run.B, run.Hq, run.d), dtype=torch.bfloat16, device="cuda")
              for _ in range(run.L)]
        ks = [torch.empty((run.B, run.Hkv, run.d), dtype=torch.bfloat16, device="cuda")
              for _ in range(run.L)]
        vs = [torch.empty_like(k) for k in ks]
        outs = [torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
                for _ in range(run.L)]
        graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            st = torch.cuda.current_stream()
            for layer in range(run.L):
                hwkv.hwkv_decode_step_graph(run.cache, layer, qs[layer], ks[layer], vs[layer],
                                            run.scale, outs[layer], st)
        # capture does not run the kernels: the device lengths are unchanged
        hwkv.hwkv_sync_lens(run.cache, run.stream)
        check_rows_state(run, lens)
        for _ in range(3):
            for layer in range(run.L):
                q, k, v = step_inputs(layer)
                qs[layer].copy_(q)
                ks[layer].copy_(k)
                vs[layer].copy_(v)
            graph.replay()
            for layer in range(run.L):
                got = outs[layer].cpu().numpy()
                assert_close(got, expected_step(run, layer, lens[layer]), "graph ragged step")
                assert not got[5].any()
                lens[layer] = [None if t is None else t + 1 for t in lens[layer]]
        # the replays advanced the lengths on the device only; host reads re-fetch them
        assert [hwkv.hwkv_row_len(run.cache, 0, b) for b in range(run.B)] == \
            [-1 if t is None else t for t in lens[0]]
        hwkv.hwkv_sync_lens(run.cache, run.stream)
        hwkv.hwkv_sync_check(run.cache)
        check_rows_state(run, lens)

        # a finished request's slot restarts empty; the next step sees only its new token
        hwkv.hwkv_reset_rows(run.cache, 3, 1, idle=False, stream=run.stream)
        for layer in range(run.L):
            lens[layer][3] = 0
        for layer in range(run.L):
            q, k, v = step_inputs(layer)
            out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
            hwkv.hwkv_decode_step(run.cache, layer, q, k, v, run.scale, out, run.stream)
            assert_close(out.cpu().numpy(), expected_step(run, layer, lens[layer]), "after reset")
            lens[layer] = [None if t is None else t + 1 for t in lens[layer]]
        hwkv.hwkv_sync_check(run.cache)
        # row 3 now holds position 0 again (same generator token as before)
        check_rows_state(run, lens)
    finally:
        run.close()


def test_prefill_rows_and_ragged_plain_decode():
    run = Run(n_layers=1, batch=3, n_q_heads=8, n_kv_heads=2, head_dim=64, max_ctx=4096,
              windows=[0, 300], seed=5)
    torch = run.torch
    try:
        # row 1 gets a 600-token prompt through prefill_rows in two chunks; row 0 by append
        append_row(run, 0, 0, 257)
        for t0, n in ((0, 400), (400, 200)):
            q = run.gen(hwkv_gen.Q, 0, t0, n, run.Hq)[1:2].contiguous()
            k = run.gen(hwkv_gen.K, 0, t0, n, run.Hkv)[1:2].contiguous()
            v = run.gen(hwkv_gen.V, 0, t0, n, run.Hkv)[1:2].contiguous()
            out = torch.empty((1, n, run.Hq, run.d), dtype=torch.float32, device="cuda")
            hwkv.hwkv_prefill_rows(run.cache, 0, 1, 1, q, k, v, n, run.scale, out, run.stream)
            got = out.cpu().numpy()[0]
            pos = list(range(t0, t0 + n, 37)) + [t0 + n - 1]
            for qh in (0, 5):
                assert_close(got[[p - t0 for p in pos], qh], run.oracle_rows(0, 1, qh, pos),
                             "prefill_rows")
        with pytest.raises(hwkv.HwkvError):  # rows 0 and 1 hold different lengths
            hwkv.hwkv_prefill_rows(run.cache, 0, 0, 2, q, k, v, 1, run.scale, out, run.stream)
        # plain decode over ragged rows: row 2 holds nothing and reads as zeros
        lens = [257, 600, 0]
        q = rows_at(run, hwkv_gen.Q, 0, [256, 599, None], run.Hq)
        out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
        hwkv.hwkv_decode_attn(run.cache, 0, q, run.scale, out, run.stream)
        got = out.cpu().numpy()
        want = np.zeros_like(got, dtype=np.float64)
        for b in (0, 1):
            for h in range(run.Hkv):
                want[b, h * run.G:(h + 1) * run.G] = oracle_unit_decode(run, 0, b, h, lens[b] - 1)
        assert_close(got, want, "ragged plain decode")
        assert not got[2].any()
        hwkv.hwkv_sync_check(run.cache)
        check_rows_state(run, [lens])
    finally:
        run.close()


def test_graph_large_ragged_sampled():
    # d = 256, 24 query / 4 KV heads, windows {full, 16384, 4096, 1024}; rows far apart
    start = [33000, 9000, 100, 20000]
    run = Run(n_layers=1, batch=4, n_q_heads=24, n_kv_heads=4, head_dim=256, max_ctx=40000,
              windows=[0, 16384, 4096, 1024], seed=3, per_head_scale=True)
    torch = run.torch
    try:
        for b, n in enumerate(start):
            append_row(run, 0, b, n)
        lens = list(start)
        q = torch.empty((run.B, run.Hq, run.d), dtype=torch.bfloat16, device="cuda")
        k = torch.empty((run.B, run.Hkv, run.d), dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
        graph = torch.cuda.CUDAGraph()
        torch.cuda.synchronize()
        with torch.cuda.graph(graph):
            hwkv.hwkv_decode_step_graph(run.cache, 0, q, k, v, run.scale, out,
                                        torch.cuda.current_stream())
        for _ in range(2):
            q.copy_(rows_at(run, hwkv_gen.Q, 0, lens, run.Hq))
            k.copy_(rows_at(run, hwkv_gen.K, 0, lens, run.Hkv))
            v.copy_(rows_at(run, hwkv_gen.V, 0, lens, run.Hkv))
            graph.replay()
            assert_close(out.cpu().numpy(), expected_step(run, 0, lens), "large graph step")
            lens = [t + 1 for t in lens]
        hwkv.hwkv_sync_lens(run.cache, run.stream)
        hwkv.hwkv_sync_check(run.cache)
        assert [hwkv.hwkv_row_len(run.cache, 0, b) for b in range(run.B)] == lens
        w = run.windows
        assert hwkv.hwkv_residency_bytes(run.cache, 0) == sum(
            oracle.nominal_storage(w, t, run.d, run.d, 2, 2, 1) for t in lens)
    finally:
        run.close()


def test_graph_row_at_capacity_is_skipped():
    run = Run(n_layers=1, batch=2, n_q_heads=2, n_kv_heads=1, head_dim=64, max_ctx=200,
              windows=[0], seed=9)
    torch = run.torch
    try:
        append_row(run, 0, 0, 199)
        append_row(run, 0, 1, 10)
        lens = [199, 10]
        out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
        for step in range(2):
            q = rows_at(run, hwkv_gen.Q, 0, lens, run.Hq)
            k = rows_at(run, hwkv_gen.K, 0, lens, run.Hkv)
            v = rows_at(run, hwkv_gen.V, 0, lens, run.Hkv)
            hwkv.hwkv_decode_step_graph(run.cache, 0, q, k, v, run.scale, out, run.stream)
            got = out.cpu().numpy()
            if step == 0:  # row 0 reaches max_ctx
                assert_close(got, expected_step(run, 0, lens), "last fitting step")
                lens = [200, 11]
            else:  # row 0 is full: skipped with zeros, row 1 goes on
                assert not got[0].any()
                assert_close(got[1], expected_step(run, 0, [None, 11])[1], "row beside a full row")
                lens = [200, 12]
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_sync_check(run.cache)
        assert e.value.status == hwkv.HWKV_EKERNEL
        hwkv.hwkv_sync_lens(run.cache, run.stream)
        assert [hwkv.hwkv_row_len(run.cache, 0, b) for b in range(2)] == lens
        # the host-checked step refuses the full row outright
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_decode_step(run.cache, 0, q, k, v, run.scale, out, run.stream)
        assert e.value.status == hwkv.HWKV_ECAPACITY
    finally:
        run.close()


def test_device_plan_many_units():
    # 80 rows x 4 KV heads = 320 units: more than the 256 the plan keeps in registers
    rng = np.random.default_rng(17)
    B = 80
    start = [int(x) for x in rng.integers(0, 500, size=B)]
    idle = {3, 40, 77}
    run = Run(n_layers=1, batch=B, n_q_heads=8, n_kv_heads=4, head_dim=64, max_ctx=600,
              windows=[0, 128, 64, 0], seed=21)
    torch = run.torch
    try:
        for b in sorted(idle):
            hwkv.hwkv_reset_rows(run.cache, b, 1, idle=True, stream=run.stream)
        # rows of equal length are appended together (one call per length)
        by_len = {}
        for b, n in enumerate(start):
            if b not in idle:
                by_len.setdefault(n, []).append(b)
        for n, rows in by_len.items():
            if n == 0:
                continue
            k_all = run.gen(hwkv_gen.K, 0, 0, n, run.Hkv)
            v_all = run.gen(hwkv_gen.V, 0, 0, n, run.Hkv)
            for b in rows:
                hwkv.hwkv_append_rows(run.cache, 0, b, 1, k_all[b:b + 1].contiguous(),
                                      v_all[b:b + 1].contiguous(), n, run.stream)
        lens = [None if b in idle else start[b] for b in range(B)]
        out = torch.empty((run.B, run.Hq, run.d), dtype=torch.float32, device="cuda")
        for step in range(2):
            q = rows_at(run, hwkv_gen.Q, 0, lens, run.Hq)
            k = rows_at(run, hwkv_gen.K, 0, lens, run.Hkv)
            v = rows_at(run, hwkv_gen.V, 0, lens, run.Hkv)
            hwkv.hwkv_decode_step_graph(run.cache, 0, q, k, v, run.scale, out, run.stream)
            got = out.cpu().numpy()
            assert_close(got, expected_step(run, 0, lens), "320-unit device plan step %d" % step)
            for b in idle:
                assert not got[b].any()
            lens = [None if t is None else t + 1 for t in lens]
        hwkv.hwkv_sync_check(run.cache)
        check_rows_state(run, [lens])
    finally:
        run.close()
