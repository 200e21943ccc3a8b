"""Policy artifact I/O (host-only): the layer x KV-head window matrix with its
artifact id and seed round-trips exactly, and malformed files are rejected with
the offending line."""
import numpy as np
import pytest

import paper_2609_02029_gb300 as hwkv
from hwkv_gen import workloads


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_02029_gb300 import build
    build.build()


def test_round_trip(tmp_path):
    wl = workloads.make("layers16_112k")
    W = np.array(wl.windows, dtype=np.int64).reshape(wl.n_layers, wl.n_kv_heads)
    path = tmp_path / "policy.txt"
    hwkv.hwkv_policy_save(path, "seqcalib-tau0.995-run7", 2 ** 63 + 5, W)
    art, seed, W2 = hwkv.hwkv_policy_load(path)
    assert art == "seqcalib-tau0.995-run7" and seed == 2 ** 63 + 5
    assert np.array_equal(W, W2)
    # the loaded matrix builds the same cache layout
    pol = hwkv.make_policy(wl.n_layers, wl.n_kv_heads, wl.n_q_heads, wl.head_dim, wl.batch,
                           wl.max_ctx, W2)
    assert hwkv.hwkv_required_bytes(pol) == hwkv.hwkv_required_bytes(
        hwkv.make_policy(wl.n_layers, wl.n_kv_heads, wl.n_q_heads, wl.head_dim, wl.batch,
                         wl.max_ctx, wl.windows))


def test_comments_and_blank_lines(tmp_path):
    p = tmp_path / "p.txt"
    p.write_text("# calibration output\nhwkv-policy 1\n\nartifact a1 # id\nseed 0\nshape 2 3\n"
                 "layer 0 0 8192 512\nlayer 1 16384 0 0   # last\n")
    art, seed, W = hwkv.hwkv_policy_load(p)
    assert (art, seed) == ("a1", 0)
    assert W.tolist() == [[0, 8192, 512], [16384, 0, 0]]


@pytest.mark.parametrize("text,msg", [
    ("hwkv-policy 2\nartifact a\nseed 1\nshape 1 1\nlayer 0 5\n", ":1:"),
    ("hwkv-policy 1\nartifact a b\nseed 1\nshape 1 1\nlayer 0 5\n", None),
    ("hwkv-policy 1\nartifact a\nseed -1\nshape 1 1\nlayer 0 5\n", ":3:"),
    ("hwkv-policy 1\nartifact a\nseed 1\nshape 2 1\nlayer 0 5\n", "incomplete"),
    ("hwkv-policy 1\nartifact a\nseed 1\nshape 1 2\nlayer 0 5\n", ":5:"),
    ("hwkv-policy 1\nartifact a\nseed 1\nshape 1 1\nlayer 0 -5\n", ":5:"),
    ("hwkv-policy 1\nartifact a\nseed 1\nshape 1 1\nlayer 1 5\n", ":5:"),
    ("hwkv-policy 1\nartifact a\nseed 1\nshape 1 1\nlayer 0 5 6\n", ":5:"),
])
def test_malformed(tmp_path, text, msg):
    p = tmp_path / "bad.txt"
    p.write_text(text)
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_policy_load(p)
    assert e.value.status == hwkv.HWKV_EINVAL
    if msg:
        assert msg in str(e.value)


def test_save_rejects_bad_inputs(tmp_path):
    with pytest.raises(hwkv.HwkvError):
        hwkv.hwkv_policy_save(tmp_path / "x", "has space", 1, [[1, 2]])
    with pytest.raises(hwkv.HwkvError):
        hwkv.hwkv_policy_save(tmp_path / "x", "ok", 1, [[1, -2]])
