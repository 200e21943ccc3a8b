"""Parity at the edges of the supported sizes, through the C ABI against the oracle:
the largest KV-head count (64) and the largest GQA group (8), each with 256 query
heads (the input generator keys at most 256 heads), the largest batch (256 rows)
through prefill and the fused decode step, and empty calls (n = 0 appends and
prefills change nothing)."""
import numpy as np
import pytest

import hwkv_gen
import paper_2609_02029_gb300 as hwkv
from harness import Run, assert_close, check_ring_unit, oracle_unit_decode

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("Hkv,G", [(64, 4), (32, 8)])
def test_most_kv_heads_and_largest_group(Hkv, G):
    windows = [0 if h % 4 == 0 else (17 * h + 3) for h in range(Hkv)]
    Hq = Hkv * G
    r = Run(1, 1, Hq, Hkv, 64, 420, windows, seed=41)
    try:
        out = r.prefill(0, 390).cpu().numpy()
        rows = [0, 1, 100, 257, 388, 389]
        for qh in range(0, Hq, 37):
            assert_close(out[0, rows, qh], r.oracle_rows(0, 0, qh, rows), "prefill q%d" % qh)
        for _ in range(3):
            got = r.decode_step_fused(0).cpu().numpy()
        p = hwkv.hwkv_seq_len(r.cache, 0) - 1
        for h in range(Hkv):
            assert_close(got[0, h * G:(h + 1) * G], oracle_unit_decode(r, 0, 0, h, p), "decode h%d" % h)
        for h in (0, 1, Hkv - 1):
            check_ring_unit(r, 0, 0, h)
        r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_256_batch_rows_prefill_and_decode():
    r = Run(1, 256, 8, 2, 128, 200, [0, 45], seed=42)
    try:
        out = r.prefill(0, 150).cpu().numpy()
        rows = [0, 44, 45, 46, 149]
        for b in (0, 1, 127, 255):
            for qh in (0, 3, 4, 7):
                assert_close(out[b, rows, qh], r.oracle_rows(0, b, qh, rows), "prefill b%d q%d" % (b, qh))
        for _ in range(2):
            got = r.decode_step_fused(0).cpu().numpy()
        p = hwkv.hwkv_seq_len(r.cache, 0) - 1
        for b in (0, 5, 200, 255):
            for h in range(2):
                assert_close(got[b, h * 4:(h + 1) * 4], oracle_unit_decode(r, 0, b, h, p), "decode b%d" % b)
                check_ring_unit(r, 0, b, h)
        r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_empty_calls_change_nothing():
    import torch
    r = Run(1, 2, 8, 2, 64, 100, [0, 10], seed=43)
    try:
        r.fill(0, 30)
        before = [hwkv.hwkv_debug_copy_ring(r.cache, 0, b, h, r.d) for b in range(2) for h in range(2)]
        k = torch.empty((2, 1, 2, 64), dtype=torch.bfloat16, device="cuda")
        q = torch.empty((2, 1, 8, 64), dtype=torch.bfloat16, device="cuda")
        out = torch.full((2, 1, 8, 64), 7.0, dtype=torch.float32, device="cuda")
        hwkv.hwkv_append(r.cache, 0, k, k, 0, r.stream)
        hwkv.hwkv_prefill(r.cache, 0, q, k, k, 0, r.scale, out, r.stream)
        hwkv.hwkv_append_rows(r.cache, 0, 1, 1, k, k, 0, r.stream)
        hwkv.hwkv_sync_check(r.cache)
        assert hwkv.hwkv_seq_len(r.cache, 0) == 30
        assert bool((out == 7.0).all())  # nothing written
        after = [hwkv.hwkv_debug_copy_ring(r.cache, 0, b, h, r.d) for b in range(2) for h in range(2)]
        for (k0, v0), (k1, v1) in zip(before, after):
            assert np.array_equal(k0, k1) and np.array_equal(v0, v1)
        r.check_rings(0)
    finally:
        r.close()
