"""Chunk appends against the oracle's rings (Sec. 3.3: a head keeps only its latest W
states, S sink positions first where it has sinks).

Of a chunk's tokens only the sink positions and the last W of the window region land,
in at most three runs of consecutive ring slots: the sinks, the window tokens up to the
ring's end, and those that wrap to its first window slot. The chunk sizes here sit
around multiples of a block's row count (R - 1, R, R + 1, 3R + 5, 5R for R = 8192 / d),
the windows wrap inside chunks, some are shorter than R or one slot long, sink regions
are shorter and longer than R, and one multi-row call has rows at different positions.
Rings are compared bit-exactly in both cache formats after every call, together with
the resident bytes."""
import numpy as np
import pytest

import hwkv_gen
import oracle
import paper_2609_02029_gb300 as hwkv
from harness import Run, RunS

pytestmark = pytest.mark.gpu
BF16, FP8 = hwkv.HWKV_KV_BF16, hwkv.HWKV_KV_FP8_E4M3


@pytest.mark.parametrize("d,fmt", [(64, BF16), (128, BF16), (256, BF16), (128, FP8), (256, FP8)])
def test_chunk_append_around_block_sizes(d, fmt):
    R = 8192 // d
    chunks = [R - 1, R, R + 1, 3 * R + 5, 1, 2 * R + 7, 5 * R]
    windows = [0, R + 3, 40, 2 * R - 1, 3 * R + 5, 1]
    sinks = [0, 0, 0, 5, R + 1, 0]
    r = RunS(windows=windows, sinks=sinks, n_q_heads=12, n_kv_heads=6, head_dim=d, batch=3,
             max_ctx=sum(chunks) + 16, seed=21 + d, kv_format=fmt)
    try:
        for n in chunks:
            r.append(n)
            r.check_rings()
            r.check_residency()
        hwkv.hwkv_sync_check(r.cache)
    finally:
        r.close()


def _chunk_rows(run, tensor, layer, starts, n):
    """[len(starts), n, Hkv, d] bf16: row i holds the generator's tokens of batch row
    starts[i][0] from position starts[i][1]."""
    parts = [run.gen(tensor, layer, t, n, run.Hkv)[b:b + 1] for b, t in starts]
    return run.torch.cat(parts).contiguous()


@pytest.mark.parametrize("fmt", [BF16, FP8])
def test_chunk_append_ragged_rows_in_one_call(fmt):
    d, R = 128, 64
    windows = [0, 100, 7, 300]
    B = 5
    run = Run(1, B, 8, 4, d, 1200, windows, seed=31, kv_format=fmt)
    try:
        # rows at different lengths, then one call over rows 1..4 with a chunk of 3R + 9
        for b, n in enumerate([10, 0, 65, 130, 299]):
            for m in ([n] if n else []):
                k = run.gen(hwkv_gen.K, 0, 0, m, 4)[b:b + 1].contiguous()
                v = run.gen(hwkv_gen.V, 0, 0, m, 4)[b:b + 1].contiguous()
                hwkv.hwkv_append_rows(run.cache, 0, b, 1, k, v, m, run.stream)
        lens = [hwkv.hwkv_row_len(run.cache, 0, b) for b in range(B)]
        n = 3 * R + 9
        starts = [(b, lens[b]) for b in range(1, B)]
        k = _chunk_rows(run, hwkv_gen.K, 0, starts, n)
        v = _chunk_rows(run, hwkv_gen.V, 0, starts, n)
        hwkv.hwkv_append_rows(run.cache, 0, 1, B - 1, k, v, n, run.stream)
        hwkv.hwkv_sync_check(run.cache)
        lens = [lens[0]] + [t + n for t in lens[1:]]
        for b, t in enumerate(lens):
            assert hwkv.hwkv_row_len(run.cache, 0, b) == t
            for h in range(4):
                kr, vr = hwkv.hwkv_debug_copy_ring(run.cache, 0, b, h, d, fmt)
                cap = kr.shape[0]
                held = min(t, cap)
                if fmt == BF16:
                    ek = oracle.ring_expected_gen(run.g, hwkv_gen.K, 0, b, h, d, t, cap)
                    ev = oracle.ring_expected_gen(run.g, hwkv_gen.V, 0, b, h, d, t, cap)
                    assert np.array_equal(kr[:held], ek[:held]), ("K", b, h)
                    assert np.array_equal(vr[:held], ev[:held]), ("V", b, h)
                else:
                    ks, vs = hwkv.hwkv_debug_copy_scales(run.cache, 0, b, h)
                    ek, eks = oracle.ring_expected_fp8_gen(run.g, hwkv_gen.K, 0, b, h, d, t, cap)
                    ev, evs = oracle.ring_expected_fp8_gen(run.g, hwkv_gen.V, 0, b, h, d, t, cap)
                    assert np.array_equal(kr[:held], ek[:held]) and np.array_equal(ks[:held], eks[:held]), ("K", b, h)
                    assert np.array_equal(vr[:held], ev[:held]) and np.array_equal(vs[:held], evs[:held]), ("V", b, h)
    finally:
        run.close()
