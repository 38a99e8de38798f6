"""Planted-model pin of the frame procedure's indexing.

The paper fixes which table and which head each step uses (Sec. 2.1: code c_i is looked
up in table i, the hidden state that LM head i reads emits c_i; Sec. 2.2 / Fig. 3: the
draft of c_{k+j} is LMH_{k+j}(h_k + b_j)).  With every block matrix set to zero the
transformer is the identity on the residual stream, so h_s = RMSNorm(input of row s).
Tables are one-hot, LM head s maps "code c in table s-1" to id (c + s) mod V and maps
offset b_j to id (5 s + 3 j) mod V.  Correct indexing therefore emits
c_s = (c_{s-1} + s) mod V and drafts (5 s + 3 j) mod V for position s at lookahead j;
an off-by-one table, head or offset gives a different sequence.
"""
import numpy as np
import pytest

from paper_2609_37007_gb300.synth import FrameInput, TINY, make_weights, weights_as_f32
from oracle.frame import decode_frame
from oracle.model import Model


def planted(K):
    cfg = TINY.replace(hidden=512, draft_len=K)
    W = {k: np.zeros_like(v) for k, v in weights_as_f32(cfg, make_weights(cfg)).items()}
    V, P = cfg.vocab, cfg.n_pos
    for k in W:
        if k.endswith("norm"):
            W[k][:] = 1.0
    for i in range(1, P):
        for c in range(V):
            W[f"embed.{i}"][c, i * V + c] = 1.0
    for s in range(1, P + 1):
        for c in range(V):
            W[f"head.{s}"][(c + s) % V, (s - 1) * V + c] = 10.0
        for j in range(1, K + 1):
            W[f"head.{s}"][(5 * s + 3 * j) % V, 300 + j] = 10.0
    for j in range(1, K + 1):
        W[f"offset.{j}"][300 + j] = 25.0
    return cfg, Model(cfg, W)


@pytest.mark.parametrize("K", [0, 1, 2, 3])
def test_planted_indexing(K):
    cfg, m = planted(K)
    V, P = cfg.vocab, cfg.n_pos
    c0 = 11
    emb = np.zeros(cfg.hidden, dtype=np.float32)
    emb[c0] = 1.0                                   # "code c0 in table 0" = block 0
    cond = np.zeros(cfg.hidden, dtype=np.float32)
    cond[400] = 1.0
    res = decode_frame(m, FrameInput(cond=cond, c0=-1, c0_emb=emb), frame_idx=0)
    want, prev = [], c0
    for s in range(1, P + 1):
        prev = (prev + s) % V
        want.append(prev)
    assert res.codes == want
    for r in res.rounds:
        a_new = r.a + len(r.emitted)
        assert r.next_drafts == [(5 * (a_new + j) + 3 * j) % V
                                 for j in range(1, min(K, P - a_new) + 1)]
        # the fed rows are the last code and the drafts, at positions a+1..
        if r.rnd:
            assert r.positions == list(range(r.a + 1, r.a + 1 + len(r.positions)))
