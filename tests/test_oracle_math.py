"""Pins of the oracle's layer math against closed forms and textbook identities."""
import numpy as np
import pytest
import scipy.special

from oracle import chimera_oracle as co

RNG = np.random.default_rng(7)


def test_rmsnorm_constant_vector():
    # x = c*1: mean(x^2) = c^2, so y = c / sqrt(c^2 + eps) * g exactly
    for c in (3.0, -0.5, 1e-3):
        g = RNG.normal(size=16)
        y = co.rmsnorm(np.full((1, 16), c), g, 1e-6)
        np.testing.assert_allclose(y[0], c / np.sqrt(c * c + 1e-6) * g, rtol=1e-14)


def test_rmsnorm_unit_rms():
    x = RNG.normal(size=(5, 64)) * 7.0
    y = co.rmsnorm(x, np.ones(64), 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=-1)), 1.0, rtol=1e-13)


def test_silu_values():
    x = np.linspace(-20, 20, 101)
    assert co.silu(np.array([0.0]))[0] == 0.0
    np.testing.assert_allclose(co.silu(x), x * scipy.special.expit(x), rtol=1e-13, atol=1e-300)


def test_rope_position_zero_is_identity():
    x = RNG.normal(size=(3, 2, 64))
    np.testing.assert_array_equal(co.rope(x, np.zeros(3), 1e4), x)


def test_rope_matches_complex_rotation():
    # rotate-half pairs (i, i+hd/2) as the complex number x_i + j x_{i+hd/2}
    # multiplied by exp(j * pos * theta^(-2i/hd))
    hd, pos = 16, 37
    x = RNG.normal(size=(1, 1, hd))
    z = x[0, 0, : hd // 2] + 1j * x[0, 0, hd // 2:]
    w = z * np.exp(1j * pos * 10000.0 ** (-np.arange(hd // 2) * 2.0 / hd))
    y = co.rope(x, np.array([pos]), 10000.0)[0, 0]
    np.testing.assert_allclose(y, np.concatenate([w.real, w.imag]), rtol=1e-12, atol=1e-14)


def test_rope_relative_position_invariance():
    q = RNG.normal(size=(1, 1, 128))
    k = RNG.normal(size=(1, 1, 128))
    dots = []
    for p in (0, 5, 1000):
        qa = co.rope(q, np.array([p + 7]), 1e4)
        ka = co.rope(k, np.array([p]), 1e4)
        dots.append(float(np.sum(qa * ka)))
    np.testing.assert_allclose(dots, dots[0], rtol=1e-10)
    # and the rotation keeps the norm
    np.testing.assert_allclose(np.linalg.norm(co.rope(q, np.array([99]), 1e4)), np.linalg.norm(q))


def test_attend_single_key_returns_value():
    q = RNG.normal(size=(4, 8))
    k = RNG.normal(size=(1, 4, 8))
    v = RNG.normal(size=(1, 4, 8))
    np.testing.assert_allclose(co.attend(q, k, v), v[0], rtol=1e-15)


def test_attend_two_keys_sigmoid_weights():
    q = RNG.normal(size=(2, 8))
    k = RNG.normal(size=(2, 2, 8))
    v = RNG.normal(size=(2, 2, 8))
    out = co.attend(q, k, v)
    for h in range(2):
        s = [q[h] @ k[m, h] / np.sqrt(8) for m in range(2)]
        w0 = scipy.special.expit(s[0] - s[1])
        np.testing.assert_allclose(out[h], w0 * v[0, h] + (1 - w0) * v[1, h], rtol=1e-12)


def test_attend_equal_keys_average_values():
    q = RNG.normal(size=(3, 8))
    k = np.repeat(RNG.normal(size=(1, 3, 8)), 5, axis=0)
    v = RNG.normal(size=(5, 3, 8))
    np.testing.assert_allclose(co.attend(q, k, v), v.mean(axis=0), rtol=1e-12)


def test_topk_tie_break_smaller_id():
    z = np.array([1.0, 3.0, 2.0, 3.0, -1.0, 2.0])
    assert list(co.topk_desc(z, 5)) == [1, 3, 2, 5, 0]
    assert co.argmax_desc(np.zeros(7)) == 0


def _cfg(d=32, H=2, hd=16, F=48):
    return dict(n_heads=H, head_dim=hd, d_model=d, ffn_dim=F, rms_eps=1e-6, rope_theta=1e4)


def _block_weights(cfg, prefix="b"):
    d, F = cfg["d_model"], cfg["ffn_dim"]
    g = np.random.default_rng(3)
    return co.OracleWeights({
        f"{prefix}.attn_norm": 1 + 0.1 * g.normal(size=d),
        f"{prefix}.wqkv": 0.2 * g.normal(size=(3 * d, d)),
        f"{prefix}.wo": 0.2 * g.normal(size=(d, d)),
        f"{prefix}.ffn_norm": 1 + 0.1 * g.normal(size=d),
        f"{prefix}.w_gate": 0.2 * g.normal(size=(F, d)),
        f"{prefix}.w_up": 0.2 * g.normal(size=(F, d)),
        f"{prefix}.w_down": 0.2 * g.normal(size=(d, F)),
    })


def test_block_rows_causal_equals_dense_block():
    # two independent attention codes: per-row key gathering vs a dense masked matrix
    cfg = _cfg()
    W = _block_weights(cfg)
    x = RNG.normal(size=(9, cfg["d_model"]))
    empty = np.zeros((0, 2, 16))
    a, _, _ = co.block_rows(W, "b", cfg, x, np.arange(9), empty, empty,
                            np.tril(np.ones((9, 9), dtype=bool)))
    b = co.causal_block_dense(W, "b", cfg, x)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-12)


def test_block_rows_context_split_is_exact():
    # rows 0..4 as context K/V + rows 5..8 as local rows == causal block on 0..8
    cfg = _cfg()
    W = _block_weights(cfg)
    x = RNG.normal(size=(9, cfg["d_model"]))
    empty = np.zeros((0, 2, 16))
    full, k, v = co.block_rows(W, "b", cfg, x, np.arange(9), empty, empty,
                               np.tril(np.ones((9, 9), dtype=bool)))
    part, _, _ = co.block_rows(W, "b", cfg, x[5:], np.arange(5, 9), k[:5], v[:5],
                               np.tril(np.ones((4, 4), dtype=bool)))
    np.testing.assert_allclose(part, full[5:], rtol=1e-12, atol=1e-12)
