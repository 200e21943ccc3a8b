"""Host-side checks of the C-ABI library that need no GPU: it loads, exports
every entry point include/hwkv.h declares, and its pure-host calls
(arena sizing, policy validation) behave as documented."""
import pytest

import paper_2609_02029_gb300 as hwkv


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_02029_gb300 import build
    build.build()


def test_exports_every_declared_entry_point():
    names = hwkv.declared_symbols()
    assert len(names) >= 13
    for n in names:
        assert hasattr(hwkv.lib(), n), n


def test_required_bytes_counts_rings_and_workspace():
    pol = hwkv.make_policy(2, 2, 8, 64, 3, 1000, [0, 100, 2000, 5])
    n = hwkv.hwkv_required_bytes(pol)
    rings = 3 * (1000 + 100 + 1000 + 5) * 64 * 2 * 2  # W >= max_ctx is stored as full
    assert n >= rings
    assert n - rings < 2048 * 8 * 64 * 4 + 2048 * 8 * 8 + 4096


@pytest.mark.parametrize("kw,status", [
    (dict(windows=[0, -1]), hwkv.HWKV_EINVAL),
    (dict(n_q_heads=7), hwkv.HWKV_EINVAL),
    (dict(batch=0), hwkv.HWKV_EINVAL),
    (dict(max_ctx=0), hwkv.HWKV_EINVAL),
    (dict(head_dim=96), hwkv.HWKV_EUNSUPPORTED),
    (dict(n_q_heads=18), hwkv.HWKV_EUNSUPPORTED),  # GQA group of 9
])
def test_policy_validation(kw, status):
    args = dict(n_layers=1, n_kv_heads=2, n_q_heads=8, head_dim=64, batch=1, max_ctx=100,
                windows=[0, 10])
    args.update(kw)
    pol = hwkv.make_policy(**args)
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_required_bytes(pol)
    assert e.value.status == status
    assert hwkv.hwkv_last_error()


def test_null_arguments_rejected_without_device():
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_append(None, 0, 0, 0, 1, 0)
    assert e.value.status == hwkv.HWKV_EINVAL
    with pytest.raises(hwkv.HwkvError):
        hwkv.hwkv_residency_bytes(None)
    hwkv.hwkv_free(None)
