"""Pins of oracle.quant (W8A16 per-row symmetric int8 weights, reading R-Q1): a worked row,
the half-step error bound, ties to even, the extremes, zero rows, and which tensors are
quantised."""
import numpy as np

from oracle.quant import dequantise, is_quantised, quantise_rows, w8a16_weights


def test_worked_row():
    w = np.array([[0.5, -1.27, 0.0, 0.01]], dtype=np.float32)
    q, s = quantise_rows(w)
    assert s[0] == np.float32(np.float32(1.27) / np.float32(127.0))
    assert q.tolist() == [[50, -127, 0, 1]]


def test_error_bound_and_extremes():
    rng = np.random.default_rng(0)
    w = (0.02 * rng.standard_normal((64, 300))).astype(np.float32)
    q, s = quantise_rows(w)
    err = np.abs(dequantise(q, s) - w.astype(np.float64))
    assert (err <= s[:, None].astype(np.float64) * 0.5 * (1 + 1e-6)).all()
    # the largest magnitude of every row maps to +-127
    assert (np.max(np.abs(q.astype(np.int32)), axis=1) == 127).all()
    assert q.dtype == np.int8 and (q >= -127).all()


def test_ties_to_even_and_zero_rows():
    s = np.float32(1.0 / 127.0)
    w = np.array([[1.0, 2.5 * s, 3.5 * s, -2.5 * s], [0.0, 0.0, 0.0, 0.0]], dtype=np.float32)
    q, sc = quantise_rows(w)
    r = (w[0] / sc[0]).astype(np.float32)
    assert q[0].tolist() == np.rint(r).astype(int).tolist()
    assert sc[1] == 0 and (q[1] == 0).all()


def test_which_tensors():
    for name in ("layers.0.wq", "layers.4.wd", "head.15", "layers.2.wg"):
        assert is_quantised(name)
    for name in ("embed.3", "layers.0.attn_norm", "offset.1", "final_norm", "layers.1.q_norm"):
        assert not is_quantised(name)
    w = {"layers.0.wq": np.ones((2, 3), dtype=np.float32), "embed.1": np.full((2, 3), 0.3, dtype=np.float32)}
    d = w8a16_weights(w)
    q, sc = quantise_rows(w["layers.0.wq"])
    assert (q == 127).all() and np.array_equal(d["layers.0.wq"], 127 * np.float64(sc[0]) * np.ones((2, 3)))
    assert np.array_equal(d["embed.1"], w["embed.1"].astype(np.float64))
