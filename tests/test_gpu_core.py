"""GPU parity of the C-ABI path against the fp64 oracle on small shapes that
still span several tiles and ragged tails: generator device/host identity,
append/wrap bit-exactness, decode and prefill outputs within tolerance,
residency exact, error codes."""
import numpy as np
import pytest

import hwkv_gen
import paper_2609_02029_gb300 as hwkv
from harness import Run, assert_close

pytestmark = pytest.mark.gpu


def test_device_generator_matches_host():
    import torch
    for g in (hwkv_gen.desc(0), hwkv_gen.desc(5, per_head_scale=True)):
        for tensor, layer, B, pos0, n, H, d in [(hwkv_gen.K, 3, 2, 1000, 37, 4, 256),
                                                 (hwkv_gen.Q, 0, 1, 0, 65, 8, 64),
                                                 (hwkv_gen.V, 15, 3, 114000, 9, 2, 128)]:
            t = torch.empty((B, n, H, d), dtype=torch.bfloat16, device="cuda")
            hwkv_gen.fill_device(g, tensor, layer, B, pos0, n, H, d, t.data_ptr(),
                                 torch.cuda.current_stream().cuda_stream)
            dev = t.view(torch.int16).cpu().numpy().view(np.uint16)
            assert np.array_equal(dev, hwkv_gen.fill_host(g, tensor, layer, B, pos0, n, H, d))


@pytest.mark.parametrize("cap_w,steps", [
    (5, [1, 1, 3, 2, 7, 1, 5, 11]),        # wraps, n < cap, n = cap, n > cap
    (64, [63, 1, 64, 130, 1, 1]),          # exact multiples and long chunks
    (0, [17, 1, 100]),                      # full head
])
def test_append_wrap_bit_exact(cap_w, steps):
    max_ctx = sum(steps) + 3
    r = Run(2, 3, 4, 2, 64, max_ctx, [cap_w, 7, 0, cap_w], seed=3)
    try:
        for n in steps:
            for layer in range(2):
                r.append(layer, n)
                r.check_rings(layer)
                r.check_residency()
    finally:
        r.close()


@pytest.mark.parametrize("d,Hq,Hkv,B,windows,prompt,steps", [
    (64, 8, 2, 1, [0, 128], 300, 5),                 # tiny-like, G=4
    (128, 8, 8, 2, [0, 1, 2, 63, 64, 65, 200, 4096], 333, 4),  # G=1, W=1 and tails
    (256, 24, 4, 2, [0, 1000, 257, 70], 1500, 3),    # G=6, several tiles per ring
    (128, 16, 2, 3, [0, 513], 2100, 2),              # G=8
])
def test_decode_parity(d, Hq, Hkv, B, windows, prompt, steps):
    r = Run(1, B, Hq, Hkv, d, prompt + steps, windows, seed=11, per_head_scale=True)
    try:
        r.fill(0, prompt, chunk=777)
        for i in range(steps):
            out = r.decode_step(0).cpu().numpy()
            p = prompt + i
            for b in range(B):
                for qh in range(Hq):
                    assert_close(out[b, qh], r.oracle_rows(0, b, qh, [p])[0],
                                 "decode b%d q%d p%d" % (b, qh, p))
        hwkv.hwkv_sync_check(r.cache)
        r.check_rings(0)
        r.check_residency()
    finally:
        r.close()


@pytest.mark.parametrize("d,Hq,Hkv,B,windows,prompt,steps", [
    (64, 8, 2, 1, [0, 128], 120, 14),                 # crosses the window and wraps
    (128, 8, 8, 2, [0, 1, 2, 63, 64, 65, 200, 4096], 60, 8),
    (256, 24, 4, 2, [0, 1000, 257, 70], 1500, 3),
    (128, 16, 2, 3, [0, 513], 2100, 2),
])
def test_fused_decode_step(d, Hq, Hkv, B, windows, prompt, steps):
    """hwkv_decode_step equals append + decode_attn (oracle, twin cache, ring bytes)."""
    r = Run(1, B, Hq, Hkv, d, prompt + steps, windows, seed=13, per_head_scale=True)
    twin = Run(1, B, Hq, Hkv, d, prompt + steps, windows, seed=13, per_head_scale=True)
    try:
        r.fill(0, prompt, chunk=511)
        twin.fill(0, prompt, chunk=511)
        for i in range(steps):
            got = r.decode_step_fused(0).cpu().numpy()
            ref = twin.decode_step(0).cpu().numpy()
            p = prompt + i
            assert hwkv.hwkv_seq_len(r.cache, 0) == p + 1
            assert_close(got, ref.astype(np.float64), "fused vs separate p%d" % p)
            for b in range(B):
                for qh in range(Hq):
                    assert_close(got[b, qh], r.oracle_rows(0, b, qh, [p])[0],
                                 "fused b%d q%d p%d" % (b, qh, p))
            r.check_rings(0)
            r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()
        twin.close()


def test_decode_multi_layer_independent_state():
    r = Run(3, 2, 12, 2, 256, 900, [0, 64, 300, 0, 0, 5], seed=2)
    try:
        r.fill(0, 700)
        r.fill(1, 200)
        r.fill(2, 5)
        for layer in (2, 0, 1):
            out = r.decode_step(layer).cpu().numpy()
            p = hwkv.hwkv_seq_len(r.cache, layer) - 1
            for b in range(2):
                for qh in range(12):
                    assert_close(out[b, qh], r.oracle_rows(layer, b, qh, [p])[0], "layer %d" % layer)
        r.check_residency()
    finally:
        r.close()


@pytest.mark.parametrize("d,Hq,Hkv,B,windows,chunks", [
    (64, 8, 2, 1, [0, 128], [512]),                        # tiny prompt in one chunk
    (128, 8, 4, 2, [0, 1, 50, 100], [100, 37, 200, 64]),   # chunk > window, ragged
    (256, 12, 2, 1, [0, 130], [70, 130, 129, 1]),          # wrap inside history
    (128, 4, 1, 2, [64], [64, 64, 65, 63]),
    (64, 3, 3, 1, [0, 200, 7], [300, 129]),                # G=1: 128 positions per tile
    (128, 16, 2, 1, [0, 90], [257, 100]),                  # G=8
    (64, 9, 3, 2, [0, 150, 33], [190, 70]),                # G=3: 126 valid rows of 128
    (256, 10, 2, 1, [0, 77], [140, 60]),                   # G=5: 125 valid rows
])
def test_prefill_parity(d, Hq, Hkv, B, windows, chunks):
    total = sum(chunks)
    r = Run(1, B, Hq, Hkv, d, total, windows, seed=7, per_head_scale=True)
    try:
        t0 = 0
        for n in chunks:
            out = r.prefill(0, n).cpu().numpy()
            rows = sorted(set([0, 1, n // 2, n - 2, n - 1]) & set(range(n)))
            pos = [t0 + i for i in rows]
            for b in range(B):
                for qh in range(Hq):
                    assert_close(out[b, rows, qh], r.oracle_rows(0, b, qh, pos),
                                 "prefill b%d q%d chunk@%d" % (b, qh, t0))
            t0 += n
            r.check_rings(0)
            r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_prefill_every_row_small():
    r = Run(1, 1, 4, 2, 64, 300, [0, 33], seed=1)
    try:
        out1 = r.prefill(0, 170).cpu().numpy()
        out2 = r.prefill(0, 130).cpu().numpy()
        for qh in range(4):
            assert_close(out1[0, :, qh], r.oracle_rows(0, 0, qh, list(range(170))), "chunk 1")
            assert_close(out2[0, :, qh], r.oracle_rows(0, 0, qh, list(range(170, 300))), "chunk 2")
    finally:
        r.close()


def test_error_codes():
    import torch
    r = Run(2, 1, 4, 2, 64, 10, [0, 3, 4, 0])
    try:
        q = torch.zeros((1, 4, 64), dtype=torch.bfloat16, device="cuda")
        out = torch.empty((1, 4, 64), dtype=torch.float32, device="cuda")
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_decode_attn(r.cache, 0, q, 1.0, out, r.stream)  # empty layer
        assert e.value.status == hwkv.HWKV_EINVAL
        r.fill(0, 10)
        with pytest.raises(hwkv.HwkvError) as e:
            r.append(0, 1)  # beyond max_ctx
        assert e.value.status == hwkv.HWKV_ECAPACITY
        assert hwkv.hwkv_seq_len(r.cache, 0) == 10
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_seq_len(r.cache, 2)
        assert e.value.status == hwkv.HWKV_EINVAL
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def test_library_allocated_arena():
    import torch
    pol = hwkv.make_policy(1, 2, 4, 128, 2, 100, [0, 10])
    c = hwkv.hwkv_alloc(pol, None, 0, torch.cuda.current_stream())
    try:
        assert hwkv.hwkv_allocated_ring_bytes(c) == 2 * (100 + 10) * 128 * 4
        assert hwkv.hwkv_residency_bytes(c) == 0
    finally:
        hwkv.hwkv_free(c)


def test_bounded_wait_gives_up_and_reports():
    """The kernels' bounded mbarrier wait, run out on purpose (an mbarrier nothing
    arrives at, a 50 ms limit, nothing asynchronous in flight): the error word
    reaches the host as HWKV_EKERNEL, the word is cleared, and the cache and the
    context keep working."""
    import time
    import torch
    r = Run(1, 1, 8, 2, 64, 400, [0, 128], seed=1)
    try:
        r.fill(0, 200)
        hwkv.hwkv_sync_check(r.cache)
        t0 = time.perf_counter()
        hwkv.hwkv_debug_wait_probe(r.cache, 50_000_000, r.stream)
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_sync_check(r.cache)
        assert e.value.status == hwkv.HWKV_EKERNEL
        assert "0x1" in str(e.value)
        assert time.perf_counter() - t0 >= 0.05
        hwkv.hwkv_sync_check(r.cache)  # cleared
        out = r.decode_step(0).cpu().numpy()
        p = hwkv.hwkv_seq_len(r.cache, 0) - 1
        for qh in range(8):
            assert_close(out[0, qh], r.oracle_rows(0, 0, qh, [p])[0], "decode after the probe")
        hwkv.hwkv_sync_check(r.cache)
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_debug_wait_probe(r.cache, 10, r.stream)  # below the 1 ms floor
        assert e.value.status == hwkv.HWKV_EINVAL
        torch.cuda.synchronize()
    finally:
        r.close()
