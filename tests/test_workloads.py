"""The seeded input recipe (CPU): shapes of the benchmarked layers, reproducible and independent
seed streams, bf16 rounding, and the stated distributions, for the NumPy draws that the parity tests
feed to both sides and for the torch draws the benchmark makes on the device (here on the CPU)."""
import numpy as np
import pytest
import torch

from paper_2606_10531_gb300 import workloads as wl


def test_bf16_rounding_is_round_to_nearest_even_like_torch():
    rng = np.random.default_rng(5)
    x = rng.standard_normal(20000).astype(np.float32) * np.float32(10.0) ** rng.integers(-30, 30, 20000)
    # exact ties (low half 0x8000) with even and odd upper halves, and the rounding overflow to inf
    ties = ((rng.integers(0, 0x7F00, 4000).astype(np.uint32) << 16) | 0x8000).view(np.float32)
    edge = np.array([np.finfo(np.float32).max, -np.finfo(np.float32).max, 0.0, -0.0, 1e-45, -1e-45],
                    dtype=np.float32)
    for v in (x, ties, -ties, edge):
        ours = wl.bf16_to_f32(wl.bf16_bits(v))
        ref = torch.from_numpy(v.copy()).to(torch.bfloat16).to(torch.float32).numpy()
        np.testing.assert_array_equal(ours.view(np.uint32), ref.view(np.uint32))


def test_bf16_to_f32_is_exact_on_every_finite_pattern():
    bits = np.arange(0, 1 << 16, dtype=np.uint32).astype(np.uint16)
    f = wl.bf16_to_f32(bits)
    finite = np.isfinite(f)
    np.testing.assert_array_equal(wl.bf16_bits(f[finite]), bits[finite])


def test_llama3_8b_layer_shapes_and_step_flops():
    mats = wl.llama3_8b_layer()
    assert [(m.name, m.m, m.n, m.d, m.N) for m in mats] == [
        ("q", 4096, 4096, 8, 16384), ("k", 1024, 4096, 8, 16384), ("v", 1024, 4096, 8, 16384),
        ("o", 4096, 4096, 8, 16384), ("gate", 14336, 4096, 8, 16384), ("up", 14336, 4096, 8, 16384),
        ("down", 4096, 14336, 8, 16384)]
    assert sum(6.0 * m.N * m.m * m.n for m in mats) == pytest.approx(2.144e13, rel=1e-3)


def test_llama3_70b_shapes():
    enc = wl.llama3_70b_layer_encode()
    assert sum(m.m * m.n for m in enc) == 855_638_016
    assert all(m.heavy_tail and m.w_std == 0.015 and m.d == 8 for m in enc)
    (gate,) = wl.llama3_70b_gate_decode(16)
    assert (gate.m, gate.n, gate.d, gate.N) == (28672, 8192, 8, 16)
    assert gate.m * gate.n // 4 == 58_720_256
    l2 = wl.llama2_7b_projections(4)
    assert [(m.m, m.n) for m in l2] == [(4096, 4096)] * 4 + [(11008, 4096)] * 2 + [(4096, 11008)]


def test_seed_streams_are_reproducible_and_independent():
    (mx,) = wl.tiny_layer()
    W = wl.draw_W(mx, 0, 0)
    np.testing.assert_array_equal(W, wl.draw_W(mx, 0, 0))
    assert not np.array_equal(W, wl.draw_W(mx, 0, 1))
    assert not np.array_equal(W, wl.draw_W(mx, 1, 0))
    # a tensor drawn alone equals the same tensor drawn after the others (one stream per part)
    _ = wl.draw_A(mx, 0, 0), wl.draw_b(mx, 0, 0)
    np.testing.assert_array_equal(wl.draw_X(mx, 0, 0), wl.draw_X(mx, 0, 0))


def test_a_token_sample_is_the_leading_rows_of_the_full_draw():
    """The CPU baseline times the oracle on the first tokens of the benchmarked activations."""
    (mx,) = wl.llama2_7b_projections(8, N=96)[:1]
    full_X, full_dY = wl.draw_X(mx, 3, 2), wl.draw_dY(mx, 3, 2)
    np.testing.assert_array_equal(wl.draw_X(mx, 3, 2, tokens=17), full_X[:17])
    np.testing.assert_array_equal(wl.draw_dY(mx, 3, 2, tokens=17), full_dY[:17])


def test_numpy_draws_follow_the_stated_distributions():
    mx = wl.Matrix("t", 2048, 2048, 8, 64)
    W = wl.draw_W(mx, 0, 0).astype(np.float64)
    assert abs(W.std() / 0.02 - 1) < 0.01 and abs(W.mean()) < 1e-4
    # beyond 6 sigma: ~0.01 expected of a normal 2048^2 draw, ~16 with 0.1% Student-t(4) entries
    # (P(|t_4| > 6) = 0.0039)
    assert int((np.abs(W) > 6 * 0.02).sum()) == 0
    Wh = wl.draw_W(dataclass_replace(mx, w_std=0.015, heavy_tail=True), 0, 0).astype(np.float64)
    assert abs(Wh.std() / 0.015 - 1) < 0.05
    assert 5 <= int((np.abs(Wh) > 6 * 0.015).sum()) <= 40
    A, b = wl.draw_A(mx, 0, 0), wl.draw_b(mx, 0, 0)
    assert A.shape == (8, 8) and A.dtype == np.float32 and b.shape == (8,)
    assert np.all(np.abs(A - 0.01 * np.eye(8)) < 6e-3) and np.all(np.abs(b) < 6e-3)
    assert np.all(np.diag(A) > 0.0)
    X = wl.bf16_to_f32(wl.draw_X(mx, 0, 0)).astype(np.float64)
    assert abs(X.std() - 1) < 0.01


@pytest.mark.parametrize("n,k", [(4096, 41), (11008, 110)])
def test_outlier_channels_are_one_percent_scaled_by_20(n, k):
    mx = wl.Matrix("t", 64, n, 8, 64, outlier_frac=0.01)
    X = wl.bf16_to_f32(wl.draw_X(mx, 0, 0)).astype(np.float64)
    col = X.std(axis=0)
    assert int((col > 5.0).sum()) == k
    assert np.all((col[col > 5.0] > 14) & (col[col > 5.0] < 27)) and np.all(col[col <= 5.0] < 1.6)


def test_hessian_is_symmetric_positive_definite_with_the_stated_dampening():
    n = 256
    H = wl.draw_hessian(n, 0, 0).astype(np.float64)
    np.testing.assert_array_equal(H, H.T)
    lam = np.linalg.eigvalsh(H)
    # H0 is positive semidefinite, so the 1% dampening bounds the spectrum from below
    assert lam[0] >= 0.0098 * np.mean(np.diag(H))
    big = np.diag(H) > 100.0
    assert int(big.sum()) == round(0.01 * n)


def test_device_draws_follow_the_same_recipe_on_the_cpu():
    mx = wl.Matrix("t", 1024, 1024, 8, 64, outlier_frac=0.01)
    big = dataclass_replace(mx, m=2048, n=2048)
    W = wl.torch_W(torch, big, 0, 0, "cpu").double()
    assert abs(W.std().item() / 0.02 - 1) < 0.01 and int((W.abs() > 6 * 0.02).sum()) == 0
    Wh = wl.torch_W(torch, dataclass_replace(big, w_std=0.015, heavy_tail=True), 0, 0, "cpu").double()
    assert abs(Wh.std().item() / 0.015 - 1) < 0.05
    assert 5 <= int((Wh.abs() > 6 * 0.015).sum()) <= 40
    X = wl.torch_X(torch, mx, 0, 0, "cpu").float()
    assert X.dtype == torch.float32 and int((X.std(0) > 5.0).sum()) == round(0.01 * 1024)
    A = wl.torch_A(torch, mx, 0, 0, "cpu")
    assert torch.all((A - 0.01 * torch.eye(8)).abs() < 6e-3)
    H = wl.torch_hessian(torch, 256, 0, 0, "cpu").double()
    assert torch.allclose(H, H.T)
    assert torch.linalg.eigvalsh(H)[0].item() >= 0.0098 * H.diagonal().mean().item()
    codes = wl.torch_packed_codes(torch, mx, 0, 0, "cpu")
    assert codes.dtype == torch.uint8 and codes.shape == (1024, 256)
    # every 2-bit field is uniform over the level set
    fields = torch.stack([(codes >> (2 * q)) & 3 for q in range(4)]).flatten()
    counts = torch.bincount(fields.long(), minlength=4).double() / fields.numel()
    assert torch.all((counts - 0.25).abs() < 0.005)


def dataclass_replace(mx, **kw):
    import dataclasses
    return dataclasses.replace(mx, **kw)
