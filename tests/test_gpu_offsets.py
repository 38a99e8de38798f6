"""Offset-training harness on the GPU (Sec. 2.2 offsets paragraph, Table 2): codes decoded by
the library, teacher-forced cross-entropy training of b_j with Adam (lr 1e-3), tokens per
call measured by the library on frames not used for training.

The synthetic model with a position drift in its embedding tables has the structure the
offsets model (hidden states of position k and k + j differ by a translation that depends on
j), and there the trained offsets raise the acceptance, as in the paper's Table 2."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_trained_offsets_raise_tokens_per_call_on_the_drift_model():
    from paper_2609_37007_gb300 import offsets
    from paper_2609_37007_gb300.synth import TINY_DRIFT, make_weights
    cfg = TINY_DRIFT
    w = make_weights(cfg)
    b, hist = offsets.fit(cfg, w, train_frames=2000, steps=300, lr=1e-3)
    assert hist[-1] < hist[0] - 0.05, (hist[0], hist[-1])
    assert np.isfinite(b).all() and b.shape == (cfg.draft_len, cfg.hidden)
    _, _, st0 = offsets.decode_codes(cfg, w, 2000, 6_000_000, stream_id=1)
    _, _, st1 = offsets.decode_codes(cfg, offsets.with_offsets(cfg, w, b), 2000, 6_000_000, stream_id=1)
    t0, t1 = offsets.tokens_per_call(st0), offsets.tokens_per_call(st1)
    a0 = st0[:, 3].sum() / st0[:, 2].sum()
    a1 = st1[:, 3].sum() / st1[:, 2].sum()
    print("tiny drift model: tokens per call", t0, "->", t1, "accepted per draft", a0, "->", a1)
    assert (st1[:, 1] == cfg.n_pos).all()
    assert t1 > t0 + 0.02 and a1 > a0, (t0, t1, a0, a1)
