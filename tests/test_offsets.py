"""Offset-training harness (Sec. 2.2 offsets paragraph, Table 2) on the CPU: the frozen
model's teacher-forced hidden states against the oracle's row-by-row model, the loss
gradient against central finite differences, and Adam lowering the loss."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2609_37007_gb300 import offsets  # noqa: E402
from paper_2609_37007_gb300.synth import MCD, TINY, make_frames, make_weights, weights_as_f32  # noqa: E402
from oracle.model import Model  # noqa: E402


def _tiny_batch(n=3, seed=5):
    cfg = TINY
    w = make_weights(cfg)
    cond, c0, emb = make_frames(cfg, n, first=900)
    rng = np.random.default_rng(seed)
    codes = rng.integers(0, cfg.vocab, size=(n, cfg.n_pos)).astype(np.int32)
    return cfg, w, cond, c0, emb, codes


def test_teacher_forced_hidden_equals_the_oracle_rows():
    cfg, w, cond, c0, emb, codes = _tiny_batch()
    tw = offsets.torch_weights(cfg, w, "cpu", dtype=torch.float64)
    x = offsets.input_rows(cfg, tw, torch.from_numpy(cond).double(), torch.from_numpy(c0),
                           torch.from_numpy(emb).double(), torch.from_numpy(codes))
    h = offsets.teacher_forced_hidden(cfg, tw, x).numpy()
    model = Model(cfg, weights_as_f32(cfg, w))
    for n in range(len(cond)):
        kv = model.new_kv()
        rows = [np.asarray(cond[n], dtype=np.float64), model.c0_row(int(c0[n]), emb[n])]
        rows += [model.code_row(s, int(codes[n, s - 1])) for s in range(1, cfg.n_pos - 1)]
        for pos, xr in enumerate(rows):
            ref = model.row(kv, xr, pos)
            assert np.max(np.abs(h[n, pos] - ref)) < 1e-9, (n, pos)


def _samples(dtype=torch.float64):
    cfg, w, cond, c0, emb, codes = _tiny_batch(n=4, seed=9)
    tw = offsets.torch_weights(cfg, w, "cpu", dtype=dtype)
    x = offsets.input_rows(cfg, tw, torch.from_numpy(cond).to(dtype), torch.from_numpy(c0),
                           torch.from_numpy(emb).to(dtype), torch.from_numpy(codes))
    h = offsets.teacher_forced_hidden(cfg, tw, x)
    return cfg, w, offsets.OffsetSamples(cfg, tw, h, torch.from_numpy(codes), cfg.draft_len)


def test_samples_cover_every_lookahead_and_target():
    cfg, _, s = _samples()
    P, K = cfg.n_pos, cfg.draft_len
    expect = [(k + j, j) for k in range(1, P) for j in range(1, min(K, P - k) + 1)]
    assert s.blocks == expect
    assert s.base.shape == (len(expect) * s.n, cfg.vocab)


def test_loss_gradient_matches_finite_differences():
    cfg, w, s = _samples()
    b = torch.from_numpy(offsets.offsets_of(cfg, w)).double().requires_grad_(True)
    loss = s.loss(b)
    loss.backward()
    g = b.grad.clone()
    rng = np.random.default_rng(3)
    eps = 1e-6
    for _ in range(6):
        j, i = int(rng.integers(0, cfg.draft_len)), int(rng.integers(0, cfg.hidden))
        bp, bm = b.detach().clone(), b.detach().clone()
        bp[j, i] += eps
        bm[j, i] -= eps
        fd = (float(s.loss(bp)) - float(s.loss(bm))) / (2 * eps)
        assert abs(fd - float(g[j, i])) <= 1e-6 + 1e-4 * abs(fd), (j, i, fd, float(g[j, i]))


def test_adam_lowers_the_teacher_forced_loss():
    cfg, w, s = _samples(dtype=torch.float32)
    b0 = torch.from_numpy(offsets.offsets_of(cfg, w))
    b, hist = offsets.train_offsets(s, b0, steps=40, lr=1e-2)
    assert hist[-1] < hist[0] - 1e-3, hist[::10]
    assert b.shape == b0.shape


def test_offsets_round_trip_through_the_weight_dictionary():
    w = make_weights(MCD)
    b = offsets.offsets_of(MCD, w)
    assert b.shape == (MCD.draft_len, MCD.hidden)
    w2 = offsets.with_offsets(MCD, w, b)
    for j in range(1, MCD.draft_len + 1):
        assert np.array_equal(w2[f"offset.{j}"], w[f"offset.{j}"])          # bf16 values are exact
    w3 = offsets.with_offsets(MCD, w, b + 0.5)
    assert not np.array_equal(w3["offset.1"], w["offset.1"])
    assert w3["layers.0.wq"] is w["layers.0.wq"]                           # nothing else changes
