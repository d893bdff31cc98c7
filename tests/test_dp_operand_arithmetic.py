"""Host-side checks of the integer arithmetic of the one-token packed product (dp2a kernel; the
reformulated forward of Sec. 3.2, Eq. def:forward_x, with int16 activations): the rounding of X' to
int16 by one fma with 1.5 * 2^23, the pairing of the int16 activation words with the code masks of
dp_word (read from the kernel source), the quarter-scale odd columns, and the int32 bound. A wrong
constant or pairing in the source fails here before any GPU run."""
import os
import re
from fractions import Fraction

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "paper_2606_10531_gb300", "csrc", "gemv_packed.cu")


def source():
    return open(SRC).read()


def function_body(name):
    text = source()
    start = text.index(name + "(")
    open_brace = text.index("{", start)
    depth, i = 0, open_brace
    while True:
        depth += {"{": 1, "}": -1}.get(text[i], 0)
        if depth == 0:
            return text[open_brace:i + 1]
        i += 1


def round_half_even(x: Fraction) -> int:
    f = x.numerator // x.denominator
    r = x - f
    if r > Fraction(1, 2) or (r == Fraction(1, 2) and f % 2 == 1):
        f += 1
    return f


def _f32_exact(x: Fraction) -> float:
    """x rounded once to fp32 (to nearest, ties to even), for x in fp32's normal range."""
    e = int(np.floor(np.log2(abs(float(x)))))
    ulp = Fraction(2) ** (e - 23)
    return float(round_half_even(x / ulp) * ulp)


def test_magic_rounding_gives_the_int16_of_round_half_even():
    """fl32(v + 1.5 * 2^23) keeps round(v) (ties to even) in its low mantissa bits for |v| < 2^22: the
    low 16 bits of its pattern are the two's-complement int16 of round(v), for every |round(v)| <= 32767."""
    assert re.search(r"constexpr float kMagic\s*=\s*12582912\.0f;", function_body("dp_quantize"))
    magic = Fraction(12582912)
    rng = np.random.default_rng(0)
    vals = [Fraction(k) + Fraction(1, 2) for k in range(-32768, 32767, 97)]            # exact ties
    vals += [Fraction(float(v)) for v in rng.uniform(-32767.49, 32767.49, 4000)]    # everything else
    vals += [Fraction(k) for k in (-32767, -1, 0, 1, 32767)]
    for v in vals:
        r = round_half_even(v)
        if abs(r) > 32767:
            continue
        bits = int(np.array(_f32_exact(v + magic), dtype=np.float32).view(np.uint32))
        assert (bits & 0xFFFF) == (r & 0xFFFF), (v, r)


def dp2a(a: int, b: int, hi: bool) -> int:
    h = [a & 0xFFFF, (a >> 16) & 0xFFFF]
    h = [x - 0x10000 if x & 0x8000 else x for x in h]                      # signed int16 halves
    by = [(b >> (8 * k)) & 0xFF for k in range(4)]                          # unsigned bytes
    o = 2 if hi else 0
    return h[0] * by[o] + h[1] * by[o + 1]


def test_activation_words_pair_with_the_code_masks():
    """One 16-column block: int16 activations q (odd columns at a quarter scale) packed as the kernel
    packs them, multiplied by a 16-code word through dp_word's masks and dp2a calls, give
    sum_even z q + 4 sum_odd z q exactly."""
    quant = function_body("dp_quantize")
    first = [int(v) for v in re.search(r"kFirst\[8\]\s*=\s*\{([^}]*)\}", quant).group(1).split(",")]
    assert sorted(first + [c + 4 for c in first]) == list(range(16))
    assert "0x5410" in quant                                  # low halves of (column cc, column cc + 4)
    assert re.search(r"\(cc & 1\) \? 0\.25f \* inv : inv", quant)   # odd columns at a quarter scale
    body = function_body("dp_word")
    masks = dict(re.findall(r"(s\d) = (w4? & 0x[0-9A-Fa-f]+)u", body))
    assert sorted(masks) == ["s0", "s1", "s2", "s3"]
    assert re.search(r"w4 = w >> 4;", body)
    calls = re.findall(r"dp2a_(lo|hi)\((x[ab])\.([xyzw]), (s\d), (acc\d)\);", body)
    assert len(calls) == 8
    rng = np.random.default_rng(1)
    for _ in range(200):
        z = rng.integers(0, 4, 16)
        q = rng.integers(-32767, 32768, 16)
        q[1::2] = rng.integers(-8192, 8192, 8)                 # the quarter-scale columns
        w = sum(int(z[c]) << (2 * c) for c in range(16))
        words = [((int(q[cc + 4]) & 0xFFFF) << 16) | (int(q[cc]) & 0xFFFF) for cc in first]
        regs = {"xa": dict(zip("xyzw", words[:4])), "xb": dict(zip("xyzw", words[4:]))}
        env = {"w": w, "w4": w >> 4}
        s = {}
        for name, expr in masks.items():
            var, mask = expr.split(" & ")
            s[name] = env[var] & int(mask, 16)
        acc = {"acc0": 0, "acc1": 0}
        for mode, reg, comp, sname, accn in calls:
            acc[accn] += dp2a(regs[reg][comp], s[sname], mode == "hi")
        want = int(sum(int(z[c]) * int(q[c]) * (4 if c % 2 else 1) for c in range(16)))
        assert acc["acc0"] + acc["acc1"] == want


def test_each_accumulator_stays_in_int32():
    """Each accumulator takes 8 of a block's 16 columns; at n <= 32768 its sum is below 2^31."""
    assert re.search(r"constexpr int64_t kDpMaxN = 32768;", source())
    per_column = max(3 * 32767, 4 * 3 * 8192)
    assert (32768 // 2) * per_column < 2 ** 31
