"""hwkv_decode_attn_static: decode for callers that cannot allocate device memory.

Such callers (a plugin inside another engine whose allocator owns the GPU, code
that must not synchronize the device, code issued during stream capture) are
handed their cache arena, q and out, but cannot create scratch buffers. This
entry point keeps its tile partials in a fixed array inside the library. The
test calls it through the C ABI and checks it against hwkv_decode_attn, within
the tolerance of the other parity tests, on two decode calls in a row (the
array keeps the first call's contents when the second one runs). The file name
makes pytest collect it last.
"""
import numpy as np
import pytest

import hwkv_gen
import paper_2609_02029_gb300 as hwkv
from harness import Run, assert_close

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
                assert_close(got.cpu().numpy(), ref.cpu().numpy().astype(np.float64),
                             "static vs allocating decode, step %d layer %d" % (step, layer))
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
    finally:
        r.close()
