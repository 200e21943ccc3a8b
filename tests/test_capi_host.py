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


def test_arena_smaller_than_required_is_enomem_before_any_device_call():
    """hwkv_alloc checks a caller-owned arena's size before touching the device:
    one byte short of hwkv_required_bytes gives HWKV_ENOMEM (the pointer is never
    dereferenced, so a made-up aligned address is enough here)."""
    pol = hwkv.make_policy(2, 2, 8, 128, 3, 5000, [0, 100, 4096, 0])
    need = hwkv.hwkv_required_bytes(pol)
    fake_arena = 1 << 40  # 256-byte aligned, never touched
    for short in (need - 1, need // 2, 0):
        with pytest.raises(hwkv.HwkvError) as e:
            hwkv.hwkv_alloc(pol, fake_arena, short, 0)
        assert e.value.status == hwkv.HWKV_ENOMEM
        assert "required" in hwkv.hwkv_last_error()


def _static_need(grid, d, batch, hkv):
    """The size rule written out independently: two partial slots per CTA of
    kMaxGroup (8) query heads x d fp32 outputs, then 8 (max, sum) pairs of fp32,
    then the int64 plan table (4 + 2 per ring), each rounded up to 256 bytes."""
    up = lambda x: (x + 255) // 256 * 256
    return up(2 * grid * 8 * d * 4) + up(2 * grid * 8 * 8) + up((4 + 2 * batch * hkv) * 8)


@pytest.mark.parametrize("sms,batch,hkv,d", [
    (152, 256, 64, 256),   # the largest valid policy on this GPU's SM count
    (160, 256, 64, 256),   # a few more SMs still fit
    (148, 1, 1, 64),
    (152, 16, 4, 128),
])
def test_static_decode_scratch_fits(sms, batch, hkv, d):
    pol = hwkv.make_policy(1, hkv, hkv * 8, d, batch, 1000, [0] * hkv)
    got = hwkv.hwkv_decode_static_scratch_bytes(pol, sms)
    assert got == _static_need(sms, d, batch, hkv)
    assert got <= 4 << 20


def test_static_decode_scratch_too_small_is_einval():
    # 256 SMs (the decode's slot limit) at head_dim 256 and the largest plan: > 4 MiB
    pol = hwkv.make_policy(1, 64, 512, 256, 256, 1000, [0] * 64)
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_decode_static_scratch_bytes(pol, 256)
    assert e.value.status == hwkv.HWKV_EINVAL
    assert _static_need(256, 256, 256, 64) > 4 << 20
    with pytest.raises(hwkv.HwkvError) as e:
        hwkv.hwkv_decode_static_scratch_bytes(pol, 0)
    assert e.value.status == hwkv.HWKV_EINVAL
