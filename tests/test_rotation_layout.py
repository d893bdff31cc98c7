"""Host-side check of the index arithmetic of the rotation inside the tcgen05 product's prep kernel
(the block Walsh-Hadamard rotation of Sec. 2.2 / App. Inference Speed, read as in the oracle).

The prep holds column (t + 512 gg) * 16 + i of a token's row in register i of group gg of thread t.
The kernel combines index bits 0-3 in registers, bits 4-8 (the lane) by shuffles, and bits 9 .. lb-1 in
passes over the row in shared memory, where element e sits at word e ^ (((e >> 5) & 3) << 2). These
tests replay that schedule in NumPy, with the kernel's own shared-memory addresses, for every block
size the kernel takes (2^6 .. 2^15), compare the result with the oracle's rotation, and check the
bank-conflict claims of the kernel's comments. They test the layout and addressing, not the compiled
kernel (the GPU parity tests do that)."""
import numpy as np
import pytest

import oracle

THREADS, GROUPS = 512, 4


def swz(e):
    return e ^ (((e >> 5) & 3) << 2)


def butterfly_bit(v, bit):
    """(u, v) -> (u + v, u - v) over index bit `bit` of a vector (index with that bit clear first)."""
    idx = np.arange(v.size)
    lo = idx[(idx >> bit) & 1 == 0]
    hi = lo | (1 << bit)
    u, w = v[lo].copy(), v[hi].copy()
    v[lo], v[hi] = u + w, u - w


def prep_rotation(x_row, lb):
    """The kernel's schedule on one row (fp64): registers, lane shuffles, swizzled shared-memory passes."""
    n = x_row.size
    cols = THREADS * GROUPS * 16
    v = np.zeros(cols)
    v[:n] = x_row
    for bit in range(4):                                   # registers: bits 0-3
        butterfly_bit(v, bit)
    hmax = 32 if lb >= 9 else 1 << (lb - 4)
    h = 1
    while h < hmax:                                        # lanes: t = (c // 16) % 512, lane bit h = column bit 4 + log2 h
        c = np.arange(cols)
        t = (c // 16) % THREADS
        partner = c ^ (h << 4)                             # the same register of lane t ^ h
        sgn = np.where(t & h, -1.0, 1.0)
        v = sgn * v + v[partner]
        h <<= 1
    if lb > 9:
        buf = np.full(n, np.nan)
        c = np.arange(n)
        buf[swz(c)] = v[:n]                                # 16-byte stores at chunk q ^ ((c0 >> 5) & 3)
        bit0 = 9
        while bit0 < lb:
            K = 1 << min(4, lb - bit0)
            low = (1 << bit0) - 1
            g = np.arange(n // K)
            base = swz((g & low) | ((g >> bit0) << bit0) * K)
            addr = base[:, None] + (np.arange(K) << bit0)[None, :]     # [group][k]: one thread's K words
            y = buf[addr]
            hh = 1
            while hh < K:
                k = np.arange(K)
                lo = k[(k & hh) == 0]
                u, w = y[:, lo].copy(), y[:, lo + hh].copy()
                y[:, lo], y[:, lo + hh] = u + w, u - w
                hh <<= 1
            buf[addr] = y
            bit0 += 4
        v[:n] = buf[swz(c)]
    return v[:n] / np.sqrt(2.0 ** lb)


@pytest.mark.parametrize("n", [64, 576, 384, 768, 512, 3072, 14336, 4096, 12288])
def test_prep_rotation_schedule_equals_the_oracle_rotation(n):
    """Blocks 2^6 .. 2^12 (lanes only, one pass of 2, 4 or 8 points): the whole row against the oracle."""
    lb = oracle.hadamard_block(n).bit_length() - 1
    assert 6 <= lb <= 12
    rng = np.random.default_rng(n)
    X = rng.normal(size=(2, n))
    ref = oracle.hadamard_rotate(X, n)
    for r in range(2):
        np.testing.assert_allclose(prep_rotation(X[r], lb), ref[r], rtol=0, atol=1e-12 * np.abs(X).max() * n)


@pytest.mark.parametrize("n", [8192, 24576, 16384, 32768])
def test_prep_rotation_schedule_large_blocks(n):
    """Blocks 2^13 .. 2^15 (one 16-point pass, or 16 + 2 and 16 + 4 points), where the oracle's dense
    block would take gigabytes: sampled outputs against the closed form of the Sylvester matrix,
    H[i][j] = (-1)^popcount(i & j) / sqrt(B), summed over the output's block."""
    lb = oracle.hadamard_block(n).bit_length() - 1
    assert 13 <= lb <= 15
    B = 1 << lb
    rng = np.random.default_rng(n)
    x = rng.normal(size=n)
    out = prep_rotation(x, lb)
    i = np.arange(B)
    for j in rng.integers(0, n, 24):
        blk = (j // B) * B
        sign = 1.0 - 2.0 * (np.vectorize(lambda v: bin(v).count("1"))(i & (j - blk)) & 1)
        assert abs(out[j] - np.dot(x[blk:blk + B], sign) / np.sqrt(B)) <= 1e-12 * np.abs(x).sum()


def test_swizzle_is_a_permutation_within_64_byte_groups():
    e = np.arange(32768)
    p = swz(e)
    assert np.array_equal(np.sort(p), e)
    assert np.array_equal(p >> 4, e >> 4)                  # stays in its 16-element (64-byte) group
    assert np.array_equal(p & 3, e & 3)                    # moves whole 16-byte chunks


def test_prep_stores_are_conflict_free():
    """A 16-byte store of a quarter warp (8 lanes) touches 8 distinct 4-bank groups."""
    for gg in range(GROUPS):
        for warp in range(THREADS // 32):
            for q in range(4):
                for quarter in range(4):
                    lanes = np.arange(8) + 8 * quarter
                    c0 = (warp * 32 + lanes + THREADS * gg) * 16
                    word = c0 + 4 * (q ^ ((c0 >> 5) & 3))
                    assert len(set(((word // 4) % 8).tolist())) == 8


@pytest.mark.parametrize("lb", [10, 11, 12, 13, 14, 15])
def test_pass_accesses_hit_32_banks(lb):
    n = 1 << lb
    bit0 = 9
    while bit0 < lb:
        K = 1 << min(4, lb - bit0)
        low = (1 << bit0) - 1
        groups = n // K
        g = np.arange(groups)
        base = swz((g & low) | ((g >> bit0) << bit0) * K).reshape(-1, 32)   # one row per warp
        for k in range(K):
            banks = np.sort((base + (k << bit0)) % 32, axis=1)
            assert np.array_equal(banks, np.broadcast_to(np.arange(32), banks.shape))
        bit0 += 4
