"""Parity helpers: replay a GPU frame trace through the CPU oracle.

A traced frame records, for every model call, the rows the GPU fed, the fp32 logits it
computed (verify rows and the draft rows it used) and every decision it took.  The
oracle then (1) recomputes each call's rows in fp64 from the same inputs and compares
the logits, and (2) runs its own sampler on the GPU's fp32 logits with the same Philox
counters; accept decisions, emitted codes and drafts must be identical.  Together this
shows that the GPU frame is the oracle's model composed with the oracle's sampler.
"""
from __future__ import annotations

import numpy as np

from paper_2609_37007_gb300 import mcd
from paper_2609_37007_gb300.synth import DRAFT_NOISY_TARGET
from oracle.frame import Sampling, sample_drafts, to_f32, verify_round


def check_trace_against_oracle(cfg, model, fr, stream_id, frame_idx, trace_u8, codes, n_calls,
                               logit_tol, draft_mode=None):
    recs, vlog, dlog = mcd.parse_trace(np.asarray(trace_u8, dtype=np.uint8), cfg.vocab)
    S = Sampling(cfg, stream_id, frame_idx, draft_mode)
    P, K = cfg.n_pos, cfg.draft_len
    kv = model.new_kv()
    max_err = 0.0
    prev_q = []
    prev_next = []
    emitted_all = []
    for c in range(n_calls):
        r = recs[c]
        a, n_rows, pos0, n_d = int(r["a"]), int(r["n_rows"]), int(r["pos0"]), int(r["n_drafts"])
        assert a == len(emitted_all), (c, a)
        if c == 0:
            assert pos0 == 0 and n_rows == 2 and n_d == 0
            rows = [(0, np.asarray(fr.cond, dtype=np.float64)), (1, model.c0_row(fr.c0, fr.c0_emb))]
            first = 1
        else:
            ids = [int(v) for v in r["input_ids"][:n_rows]]
            assert pos0 == a + 1 and n_rows == min(n_d + 1, P - a), (c, pos0, n_rows, n_d)
            assert ids[0] == emitted_all[-1]
            assert ids[1:] == prev_next[: n_rows - 1]
            assert [int(v) for v in r["drafts"][:n_d]] == prev_next[:n_d]
            rows = [(pos0 + n, model.code_row(pos0 + n - 1, ids[n])) for n in range(n_rows)]
            first = 0
        h = {pos: model.row(kv, x, pos) for pos, x in rows}
        p_rows = []
        for n in range(first, n_rows):
            pos = pos0 + n
            ref = model.verify_logits(pos, h[pos])
            got = vlog[c, n].astype(np.float64)
            err = float(np.max(np.abs(got - ref)))
            max_err = max(max_err, err)
            assert err <= logit_tol, f"call {c} row {n}: verify logits differ by {err}"
            p_rows.append(vlog[c, n].copy())
        drafts = list(zip([int(v) for v in r["drafts"][:n_d]], prev_q))
        n_acc, emitted = verify_round(S, c, a, P, p_rows, drafts)
        assert n_acc == int(r["n_acc"]), (c, n_acc, int(r["n_acc"]))
        assert emitted == [int(v) for v in r["emitted"][: int(r["n_emit"])]], (c, emitted, r["emitted"])
        a_new = a + len(emitted)
        assert int(r["draft_row"]) == a_new - pos0
        n_next = int(r["n_next"])
        assert n_next == min(K, P - a_new)
        z_rows = []
        gpu_next = [int(v) for v in r["next_drafts"][:n_next]]
        if S.mode == DRAFT_NOISY_TARGET:
            # noisy-target rows: one-row passes on a copy of the KV cache, fed the GPU's
            # drafts (Sec. 2.2 chain), plus the counter-based Gaussian noise
            kv2 = kv.copy()
            prev = emitted[-1]
            for j in range(1, n_next + 1):
                s = a_new + j
                hs = model.row(kv2, model.code_row(s - 1, prev), s)
                ref = S.noisy(to_f32(model.verify_logits(s, hs)), c, s).astype(np.float64)
                got = dlog[c, j - 1].astype(np.float64)
                err = float(np.max(np.abs(got - ref)))
                max_err = max(max_err, err)
                assert err <= logit_tol, f"call {c} noisy draft {j}: logits differ by {err}"
                z_rows.append(dlog[c, j - 1].copy())
                prev = gpu_next[j - 1]
        else:
            for j in range(1, n_next + 1):
                ref = model.draft_logits(a_new, j, h[a_new])
                got = dlog[c, j - 1].astype(np.float64)
                err = float(np.max(np.abs(got - ref)))
                max_err = max(max_err, err)
                assert err <= logit_tol, f"call {c} draft {j}: logits differ by {err}"
                z_rows.append(dlog[c, j - 1].copy())
        nd = sample_drafts(S, c, a_new, z_rows)
        prev_next = [d for d, _ in nd]
        assert prev_next == [int(v) for v in r["next_drafts"][:n_next]], (c, prev_next, r["next_drafts"])
        prev_q = [q for _, q in nd]
        emitted_all += emitted
    assert len(emitted_all) == P
    assert emitted_all == [int(v) for v in codes], (emitted_all, list(codes))
    return max_err


def check_tree_trace_against_oracle(cfg, model, fr, stream_id, frame_idx, trace_u8, codes, n_calls, tree,
                                    logit_tol):
    """TREE mode: every call's rows (tree order, ids), every row's verify logits and the draft
    row's draft logits against the oracle (rows recomputed with the tree attention mask on the
    oracle's own cache), then the walk, the kept path, the emitted codes and the next
    candidates identical when the oracle works on the GPU's fp32 logits."""
    from oracle import philox
    from oracle.sampler import draw
    from oracle.tree import ranked, tree_row, walk
    V, P = cfg.vocab, cfg.n_pos
    buf = np.asarray(trace_u8, dtype=np.uint8)
    recs, _, dlog = mcd.parse_trace(buf, V)
    trecs, vall = mcd.parse_tree_trace(buf, V)
    S = Sampling(cfg, stream_id, frame_idx)
    m_need, K = tree.ranks_needed(), tree.max_depth
    kv = model.new_kv()
    max_err = 0.0

    def cmp(got, ref, what):
        nonlocal max_err
        err = float(np.max(np.abs(np.asarray(got, dtype=np.float64) - ref)))
        max_err = max(max_err, err)
        assert err <= logit_tol, f"{what}: logits differ by {err}"

    # call 0: [cond, c0] at positions 0, 1; c1 from LM head 1
    model.row(kv, np.asarray(fr.cond, dtype=np.float64), 0)
    h1 = model.row(kv, model.c0_row(fr.c0, fr.c0_emb), 1)
    t0 = trecs[0]
    assert int(recs[0]["a"]) == 0 and int(t0["n_rows"]) == 2
    cmp(vall[0, 1], model.verify_logits(1, h1), "call 0 row 1")
    c1 = draw(S.dist(vall[0, 1].copy()), S.u(0, 1, philox.PURPOSE_TARGET))
    assert [c1] == [int(v) for v in recs[0]["emitted"][:int(recs[0]["n_emit"])]]
    emitted_all = [c1]
    n_next = int(t0["n_next"])
    assert n_next == min(K, P - 1)
    cand = []
    for d in range(1, n_next + 1):
        cmp(dlog[0, d - 1], model.draft_logits(1, d, h1), f"call 0 draft {d}")
        cand.append(ranked(dlog[0, d - 1], m_need[d - 1]))
        assert cand[-1] == [int(v) for v in t0["next_cand"][d - 1][:m_need[d - 1]]], (cand[-1], t0["next_cand"])
    for c in range(1, n_calls):
        r, t = recs[c], trecs[c]
        a = int(r["a"])
        assert a == len(emitted_all), (c, a)
        codes_map = {i + 1: x for i, x in enumerate(emitted_all)}
        # expected rows: c_a, then the nodes whose candidates exist and a + depth < P
        rows = [(-1, a + 1, codes_map[a])]
        row_of_node = {}
        for i in range(tree.n):
            d = tree.depth[i]
            if d <= len(cand) and a + d < P:
                row_of_node[i] = len(rows)
                rows.append((i, a + 1 + d, cand[d - 1][tree.rank[i]]))
        n_rows = int(t["n_rows"])
        assert n_rows == len(rows), (c, n_rows, len(rows))
        assert [int(v) for v in t["row_node"][:n_rows]] == [x[0] for x in rows]
        assert [int(v) for v in t["row_id"][:n_rows]] == [x[2] for x in rows]
        h, own = {}, {}
        h[0], own[0] = tree_row(model, kv, a + 1, [], model.code_row(a, codes_map[a]), a + 1)
        for n in range(1, n_rows):
            node, pos, x = rows[n]
            anc = [own[0]] + [own[row_of_node[j]] for j in tree.ancestors(node)[:-1]]
            h[n], own[n] = tree_row(model, kv, a + 1, anc, model.code_row(pos - 1, x), pos)
        for n in range(n_rows):
            cmp(vall[c, n], model.verify_logits(rows[n][1], h[n]), f"call {c} row {n}")
        emitted, path, drow = walk(S, c, a, P, tree, cand, lambda n: S.dist(vall[c, n].copy()), row_of_node)
        assert emitted == [int(v) for v in r["emitted"][:int(r["n_emit"])]], (c, emitted, r["emitted"])
        assert path == [int(v) for v in t["path"][:int(t["path_len"])]], (c, path, t["path"])
        assert drow == int(t["draft_row"]), (c, drow, int(t["draft_row"]))
        for i, rr in enumerate([0] + [row_of_node[nn] for nn in path if nn in row_of_node]):
            for l in range(model.cfg.n_layers):
                kv[l, 0, :, a + 1 + i] = own[rr][l][0]
                kv[l, 1, :, a + 1 + i] = own[rr][l][1]
        emitted_all += emitted
        a_new = len(emitted_all)
        n_next = int(t["n_next"])
        assert n_next == min(K, P - a_new)
        cand = []
        for d in range(1, n_next + 1):
            cmp(dlog[c, d - 1], model.draft_logits(rows[drow][1], d, h[drow]), f"call {c} draft {d}")
            cand.append(ranked(dlog[c, d - 1], m_need[d - 1]))
            assert cand[-1] == [int(v) for v in t["next_cand"][d - 1][:m_need[d - 1]]], (c, d, cand[-1])
    assert len(emitted_all) == P
    assert emitted_all == [int(v) for v in codes], (emitted_all, list(codes))
    return max_err
