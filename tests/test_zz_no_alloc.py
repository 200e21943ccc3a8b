"""hwkv_decode_attn_static: decode for callers that cannot allocate device memory.

Such callers (a plugin inside another engine whose allocator owns the GPU, code
that must not synchronize the device, code issued during stream capture) are
handed their cache arena, q and out, but cannot create scratch buffers. This
entry point keeps its tile partials in a fixed array inside the library. The
tests call it through the C ABI and check it against hwkv_decode_attn, within
the tolerance of the other parity tests, on two decode calls in a row (the
array keeps the first call's contents when the second one runs), and against
the fp64 oracle; with bf16 and 8-bit caches; after graph-mode steps (where the
call must not wait for the device to re-read the lengths); and with the
device's free memory unchanged across the calls. The file name makes pytest
collect it last.
"""
import numpy as np
import pytest

import hwkv_gen
import paper_2609_02029_gb300 as hwkv
from harness import Run, assert_close, oracle_unit_decode

pytestmark = pytest.mark.gpu


def test_static_scratch_decode_matches_allocating_decode():
    import torch
    r = Run(2, 3, 24, 4, 256, 6000, [0, 4096, 1000, 129, 0, 64, 5000, 1], seed=21,
            per_head_scale=True)
    try:
        for layer in range(2):
            r.fill(layer, 5300, chunk=2048)
        for step in range(2):  # two calls in a row on the shared array
            for layer in range(2):
                r.append(layer, 1)
                p = hwkv.hwkv_seq_len(r.cache, layer) - 1
                q = r.gen(1, layer, p, 1, r.Hq).view(r.B, r.Hq, r.d)
                ref = torch.empty((r.B, r.Hq, r.d), dtype=torch.float32, device="cuda")
                got = torch.full_like(ref, float("nan"))
                hwkv.hwkv_decode_attn(r.cache, layer, q, r.scale, ref, r.stream)
                hwkv.hwkv_decode_attn_static(r.cache, layer, q, r.scale, got, r.stream)
                hwkv.hwkv_sync_check(r.cache)
                got = got.cpu().numpy()
                assert_close(got, ref.cpu().numpy().astype(np.float64),
                             "static vs allocating decode, step %d layer %d" % (step, layer))
                for b in range(r.B):
                    for h in range(r.Hkv):
                        assert_close(got[b, h * r.G:(h + 1) * r.G],
                                     oracle_unit_decode(r, layer, b, h, p),
                                     "static vs oracle, step %d layer %d b%d h%d" % (step, layer, b, h))
    finally:
        r.close()


def test_static_scratch_serves_the_largest_batches():
    import torch
    # 256 batch rows x 4 KV heads: the work plan and partials (two per CTA) still fit
    r = Run(1, 256, 8, 4, 256, 300, [0, 4, 0, 64], seed=4)
    try:
        r.fill(0, 200)
        q = r.gen(hwkv_gen.Q, 0, 199, 1, r.Hq).view(r.B, r.Hq, r.d)
        ref = torch.empty((256, 8, 256), dtype=torch.float32, device="cuda")
        got = torch.empty_like(ref)
        hwkv.hwkv_decode_attn(r.cache, 0, q, r.scale, ref, r.stream)
        for _ in range(2):
            hwkv.hwkv_decode_attn_static(r.cache, 0, q, r.scale, got, r.stream)
            hwkv.hwkv_sync_check(r.cache)
            assert_close(got.cpu().numpy(), ref.cpu().numpy().astype(np.float64),
                         "static vs allocating decode, 256 rows")
        for b in (0, 128, 255):
            for h in range(r.Hkv):
                assert_close(got[b, h * r.G:(h + 1) * r.G].cpu().numpy(),
                             oracle_unit_decode(r, 0, b, h, 199), "static vs oracle b%d h%d" % (b, h))
    finally:
        r.close()


def test_static_scratch_decode_8bit_cache():
    import torch
    d, B, Hq, Hkv = 128, 2, 16, 2
    pol = hwkv.make_policy(1, Hkv, Hq, d, B, 4000, [0, 700], kv_format=hwkv.HWKV_KV_FP8_E4M3)
    nbytes = hwkv.hwkv_required_bytes(pol)
    arena = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    cache = hwkv.hwkv_alloc(pol, arena, nbytes, stream)
    g = hwkv_gen.desc(9, per_head_scale=True)

    def gen(tensor, pos0, n, heads):
        t = torch.empty((B, n, heads, d), dtype=torch.bfloat16, device="cuda")
        hwkv_gen.fill_device(g, tensor, 0, B, pos0, n, heads, d, t.data_ptr(), stream.cuda_stream)
        return t

    try:
        hwkv.hwkv_append(cache, 0, gen(hwkv_gen.K, 0, 3100, Hkv), gen(hwkv_gen.V, 0, 3100, Hkv),
                         3100, stream)
        for step in range(2):
            p = hwkv.hwkv_seq_len(cache, 0) - 1
            q = gen(hwkv_gen.Q, p, 1, Hq).view(B, Hq, d)
            ref = torch.empty((B, Hq, d), dtype=torch.float32, device="cuda")
            got = torch.full_like(ref, float("nan"))
            hwkv.hwkv_decode_attn(cache, 0, q, 1.0 / np.sqrt(d), ref, stream)
            hwkv.hwkv_decode_attn_static(cache, 0, q, 1.0 / np.sqrt(d), got, stream)
            hwkv.hwkv_sync_check(cache)
            assert_close(got.cpu().numpy(), ref.cpu().numpy().astype(np.float64),
                         "8-bit static vs allocating decode, call %d" % step)
            hwkv.hwkv_append(cache, 0, gen(hwkv_gen.K, p + 1, 1, Hkv), gen(hwkv_gen.V, p + 1, 1, Hkv),
                             1, stream)
    finally:
        hwkv.hwkv_free(cache)


def test_static_scratch_after_graph_mode_steps_and_without_allocating():
    """After hwkv_decode_step_graph the device owns the layer's lengths; the static
    call plans from them without waiting for the device. Two calls after a warm-up
    one leave the device's free memory and torch's allocation count unchanged."""
    import torch
    r = Run(1, 2, 12, 2, 256, 3000, [0, 500], seed=5)
    try:
        r.fill(0, 2000)
        for _ in range(3):  # graph-mode steps (issued eagerly): the device owns the lengths
            t = hwkv.hwkv_row_len(r.cache, 0, 0)
            q = r.gen(hwkv_gen.Q, 0, t, 1, r.Hq).view(r.B, r.Hq, r.d)
            out = torch.empty((r.B, r.Hq, r.d), dtype=torch.float32, device="cuda")
            hwkv.hwkv_decode_step_graph(r.cache, 0, q, r.gen(hwkv_gen.K, 0, t, 1, r.Hkv),
                                        r.gen(hwkv_gen.V, 0, t, 1, r.Hkv), r.scale, out, r.stream)
        p = 2002
        q = r.gen(hwkv_gen.Q, 0, p, 1, r.Hq).view(r.B, r.Hq, r.d)
        got = torch.full((r.B, r.Hq, r.d), float("nan"), dtype=torch.float32, device="cuda")
        hwkv.hwkv_decode_attn_static(r.cache, 0, q, r.scale, got, r.stream)  # warm-up call
        torch.cuda.synchronize()
        free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
        for _ in range(2):
            hwkv.hwkv_decode_attn_static(r.cache, 0, q, r.scale, got, r.stream)
        torch.cuda.synchronize()
        assert torch.cuda.mem_get_info()[0] == free0
        assert torch.cuda.memory_allocated() == alloc0
        ref = torch.empty_like(got)
        hwkv.hwkv_decode_attn(r.cache, 0, q, r.scale, ref, r.stream)  # re-reads the lengths
        hwkv.hwkv_sync_check(r.cache)
        assert hwkv.hwkv_row_len(r.cache, 0, 1) == p + 1
        got = got.cpu().numpy()
        assert_close(got, ref.cpu().numpy().astype(np.float64), "static after graph-mode steps")
        for b in range(r.B):
            for h in range(r.Hkv):
                assert_close(got[b, h * r.G:(h + 1) * r.G], oracle_unit_decode(r, 0, b, h, p),
                             "static after graph-mode steps vs oracle b%d h%d" % (b, h))
    finally:
        r.close()
