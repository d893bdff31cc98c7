"""Host-side checks of the exact arithmetic the tcgen05 (kind::mxf4) packed product rests on (the
reformulated forward of Sec. 3.2, Eq. def:forward_x, with codes and activation digits as e2m1 operands):
every operand value is exact in e2m1, the balanced base-8 digit split reconstructs every rounded
activation, the fp32 accumulators cannot round, and the codes' nibble order matches the digits' K order.
The digit table is read from the kernel source, so a wrong constant there fails here before any GPU run."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "paper_2606_10531_gb300", "csrc", "gemv_fp4.cu")


def e2m1(nib):
    """Value of a 4-bit e2m1 pattern: sign bit 3, exponent bits 2-1 (bias 1), mantissa bit 0."""
    s, e, m = (nib >> 3) & 1, (nib >> 1) & 3, nib & 1
    v = 0.5 * m if e == 0 else 2.0 ** (e - 1) * (1.0 + 0.5 * m)
    return -v if s else v


def kernel_constant(name):
    m = re.search(name + r"\s*=\s*(0x[0-9A-Fa-f]+)u", open(SRC).read())
    assert m, name
    return int(m.group(1), 16)


def test_digit_table_holds_each_balanced_digit_exactly():
    lo, hi = kernel_constant("kE2m1BytesLo"), kernel_constant("kE2m1BytesHi")
    table = [(lo >> (8 * f)) & 0xFF for f in range(4)] + [(hi >> (8 * f)) & 0xFF for f in range(4)]
    for f, byte in enumerate(table):          # byte f (the octal field) carries digit f - 4
        assert byte < 16
        assert e2m1(byte) == f - 4


def test_a_code_in_the_low_half_of_a_nibble_is_half_the_code():
    for z in range(4):
        assert e2m1(z) == z / 2


def test_balanced_octal_digits_reconstruct_every_rounded_activation():
    qmax, bias = 8191, 4 * (1 + 8 + 64 + 512 + 4096)
    assert bias == kernel_constant_int("kF4DigitBias")
    assert re.search(r"constexpr float kF4QMax\s*=\s*8191\.0f;", open(SRC).read())   # |q| <= 8191
    q = np.arange(-qmax, qmax + 1)
    u = q + bias
    assert u.min() >= 0 and u.max() < 8 ** 5
    d = [((u >> (3 * j)) & 7) - 4 for j in range(5)]
    assert all(((dj >= -4) & (dj <= 3)).all() for dj in d)
    assert np.array_equal(sum(dj * 8 ** j for j, dj in enumerate(d)), q)


def kernel_constant_int(name):
    m = re.search(r"constexpr int " + name + r"\s*=\s*(\d+);", open(SRC).read())
    assert m, name
    return int(m.group(1))


def test_accumulators_hold_exact_sums():
    """sum_c (z/2) d over K <= 32768 columns: multiples of 1/2 bounded by 32768 * 1.5 * 4, so twice the
    bound stays below 2^24 and every partial sum is an exact fp32 value."""
    assert kernel_constant_int("kF4Digits") == 5
    kmax = 32768
    assert 2 * kmax * 1.5 * 4 < 2 ** 24


def test_code_nibbles_follow_the_digit_k_order():
    """w & 0x33333333 puts code 2i of a 16-code word in nibble i (K positions 0-7), (w >> 2) & 0x33333333
    code 2i + 1 (K positions 8-15): K position 8 p + i carries column 2 i + p, the order the prep gives
    the digits."""
    rng = np.random.default_rng(0)
    for w in rng.integers(0, 2 ** 32, 64, dtype=np.uint64).tolist():
        codes = [(w >> (2 * c)) & 3 for c in range(16)]
        even, odd = w & 0x33333333, (w >> 2) & 0x33333333
        kpos = [(even >> (4 * i)) & 0xF for i in range(8)] + [(odd >> (4 * i)) & 0xF for i in range(8)]
        for p in range(2):
            for i in range(8):
                assert kpos[8 * p + i] == codes[2 * i + p]
