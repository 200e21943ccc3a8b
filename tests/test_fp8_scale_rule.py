"""The kernels take the 8-bit format's power-of-two row scale from the bits of the row
maximum instead of dividing: for amax = (1 + f) 2^e (a bf16 value), s = 2^(e-8) when
1 + f <= 1.75 and 2^(e-7) otherwise (448 = 1.75 2^8), for every amax whose scale is a
normal float. This checks that rule, written out here from its statement, against the
oracle's scale (the format's definition: the smallest power of two at or above
amax / 448 in fp32) for every positive finite bf16 value on that path."""
import numpy as np

import oracle


def rule_scale(bits16):
    b = np.uint32(bits16) << np.uint32(16)
    e = b >> np.uint32(23)
    f = b & np.uint32(0x7FFFFF)
    se = e - np.uint32(8) if f <= 0x600000 else e - np.uint32(7)
    return float(np.array([se << np.uint32(23)], dtype=np.uint32).view(np.float32)[0])


def test_exponent_rule_equals_the_definition_for_every_bf16_maximum():
    checked = 0
    for bits in range(0x0001, 0x7F80):  # positive finite bf16
        if (bits << 16) >> 23 <= 8:
            continue  # the scale would be subnormal: the kernels divide there
        _, s = oracle.quantize_row_e4m3(np.array([bits], dtype=np.uint16))
        assert rule_scale(bits) == float(s), hex(bits)
        checked += 1
    assert checked == 31488
