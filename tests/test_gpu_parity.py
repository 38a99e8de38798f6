"""GPU parity of libmcd against the CPU oracle (all calls go through the C ABI).

  * sampler: top-k sets/order, integer weights and sums, accept decisions, emitted codes
    and drafts bit-exact when fed the same fp32 logits and counters;
  * frames: every call's logits within tolerance of the oracle at the same inputs
    (1e-5 fp32 model, 2e-2 bf16 model) and every decision identical (tests/parity.py);
  * distribution: chi-square of GPU-emitted codes against the exact law.
"""
import math
from collections import Counter

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2609_37007_gb300 import build as _build  # noqa: E402
from paper_2609_37007_gb300 import mcd  # noqa: E402
from paper_2609_37007_gb300.synth import (DRAFT_GREEDY, DRAFT_NOISY_TARGET, MCD, TINY, make_frame,  # noqa: E402
                                          make_weights, random_logits, weights_as_f32)
from oracle.enumeration import PrefixModel, ar_distribution, spec_distribution  # noqa: E402
from oracle.frame import Sampling, decode_frame, verify_round  # noqa: E402
from oracle import accounting  # noqa: E402
from oracle.model import Model  # noqa: E402
from oracle.sampler import topk_dist  # noqa: E402
from parity import check_trace_against_oracle, check_tree_trace_against_oracle  # noqa: E402

DEV = torch.device("cuda:0")
_build.build()


def t(x, dtype=None):
    return torch.from_numpy(np.ascontiguousarray(x)).to(DEV) if dtype is None else \
        torch.from_numpy(np.ascontiguousarray(x)).to(device=DEV, dtype=dtype)


class Env:
    def __init__(self, cfg, weights=None):
        self.cfg = cfg
        self.w = make_weights(cfg) if weights is None else weights
        self.dec = mcd.Decoder(cfg, self.w)
        self._model = None

    @property
    def model(self):
        if self._model is None:
            w = weights_as_f32(self.cfg, self.w)
            if self.cfg.weight_dtype == 2:                 # W8A16: the values the library computes with
                from oracle.quant import w8a16_weights
                w = w8a16_weights(w)
            self._model = Model(self.cfg, w)
        return self._model

    def frame_inputs(self, fr):
        cond = t(fr.cond)
        c0 = t(np.array([fr.c0], dtype=np.int32)) if self.cfg.c0_vocab > 0 else None
        emb = t(fr.c0_emb) if self.cfg.c0_vocab == 0 else None
        return cond, c0, emb

    def decode(self, fr, frame_idx, stream_id=0, trace=False):
        cond, c0, emb = self.frame_inputs(fr)
        codes = torch.full((self.cfg.n_pos,), -1, dtype=torch.int32, device=DEV)
        stats = torch.zeros(8, dtype=torch.int32, device=DEV)
        tr = None
        if trace:
            tr = torch.zeros(mcd.mcd_trace_bytes(self.dec.ctx), dtype=torch.uint8, device=DEV)
        mcd.mcd_set_trace(self.dec.ctx, tr)
        mcd.mcd_decode_frame(self.dec.ctx, stream_id, frame_idx, cond, c0, emb, codes, stats)
        mcd.mcd_sync(self.dec.ctx)
        mcd.mcd_set_trace(self.dec.ctx, None)
        return codes.cpu().numpy(), stats.cpu().numpy(), (tr.cpu().numpy() if trace else None)


@pytest.fixture(scope="module")
def tiny():
    return Env(TINY)


@pytest.fixture(scope="module")
def big():
    return Env(MCD)


# ---------------------------------------------------------------- sampler ----------
@pytest.mark.parametrize("V,k,T,ties", [(2048, 50, 0.9, 0.0), (2048, 50, 0.9, 0.6), (64, 8, 1.0, 0.5),
                                        (64, 64, 1.0, 0.3), (2048, 128, 0.7, 0.2), (3072, 1, 1.3, 0.9),
                                        (2048, 50, 0.05, 0.0), (2000, 50, 0.9, 0.1), (4096, 100, 0.9, 0.2)])
def test_topk_softmax_matches_oracle(V, k, T, ties):
    """Top-k ids, integer weights and their sums are bit-exact (both sides compute the same
    fp32 exp32 and the same integer arithmetic).  Besides random rows: all-equal, signed
    zeros, an outlier that crowds the threshold into one histogram bin, a cluster of nearly
    equal values around the threshold and (T >= 0.7) a value range that overflows fp32."""
    cfg = TINY.replace(vocab=V, top_k=k, temperature=T)
    dec = mcd.Decoder(cfg)                     # sampler entry points need no weights
    rng = np.random.default_rng(V + k)
    rows = 24
    logits = random_logits(rng, rows, V, scale=0.7, tie_frac=ties)
    logits[0] = 0.0                            # all equal: lowest ids win
    logits[1, ::2] = -0.0                      # signed zeros tie
    logits[2, 3] = 1000.0                      # outlier: coarse histogram bins
    n_cl = min(V // 4, 300)                    # nearly equal values around the threshold
    logits[4, :n_cl] = (np.float32(2.0) + np.arange(n_cl, dtype=np.float32) * np.float32(2.0 ** -20))
    if T >= 0.7:
        logits[3, 5], logits[3, 9] = 2e38, -2e38   # max - min overflows fp32
    ids = torch.zeros((rows, k), dtype=torch.int32, device=DEV)
    w = torch.zeros((rows, k), dtype=torch.int32, device=DEV)
    sums = torch.zeros(rows, dtype=torch.int64, device=DEV)
    mcd.mcd_topk_softmax(dec.ctx, rows, t(logits), ids, w, sums)
    mcd.mcd_sync(dec.ctx)
    ids, w, sums = ids.cpu().numpy(), w.cpu().numpy().view(np.uint32), sums.cpu().numpy()
    for r in range(rows):
        d = topk_dist(logits[r], k, T)
        assert ids[r].tolist() == d.ids, r
        assert [int(v) for v in w[r]] == d.W, r
        assert int(sums[r]) == d.S, r
    assert ids[0].tolist() == list(range(k))
    dec.close()


def _begin(dec, cfg, stream_id=0, frame_idx=0):
    fr = make_frame(cfg, 0)
    cond = t(fr.cond)
    c0 = t(np.array([max(fr.c0, 0)], dtype=np.int32))
    emb = t(fr.c0_emb) if fr.c0_emb is not None else None
    mcd.mcd_begin_frame(dec.ctx, stream_id, frame_idx, cond, c0, emb)


@pytest.mark.parametrize("cfg,mode", [(MCD, 0), (TINY, 0), (TINY.replace(draft_len=7, n_pos=15), 0),
                                      (MCD, DRAFT_GREEDY)])
def test_accept_from_logits_is_bit_exact(cfg, mode):
    cfg = cfg.replace(draft_mode=mode)
    dec = mcd.Decoder(cfg)
    rng = np.random.default_rng(11 + mode)
    V, K, P = cfg.vocab, cfg.draft_len, cfg.n_pos
    emitted = torch.zeros(8, dtype=torch.int32, device=DEV)
    out2 = torch.zeros(2, dtype=torch.int32, device=DEV)
    n_cases, n_acc_total = 120, 0
    for case in range(n_cases):
        stream_id, frame_idx, call = int(rng.integers(0, 4)), int(rng.integers(0, 1000)), int(rng.integers(1, 15))
        _begin(dec, cfg, stream_id, frame_idx)
        a = int(rng.integers(1, P))
        n_d = int(rng.integers(0, min(K, P - a) + 1))
        n_p = n_d + 1 if a + 1 + n_d <= P else n_d
        p = random_logits(rng, max(n_p, 1), V, scale=1.0, tie_frac=0.1)
        noise = [0.0, 0.05, 0.5, 3.0][case % 4]     # from q == p (all kept) to unrelated q
        q = (p[:max(n_d, 1)] + noise * rng.standard_normal((max(n_d, 1), V))).astype(np.float32)
        S = Sampling(cfg, stream_id, frame_idx, mode)
        drafts = []
        for i in range(n_d):
            qd = S.dist(q[i]) if mode != DRAFT_GREEDY else None
            from oracle.sampler import greedy_dist, draw
            qd = greedy_dist(q[i]) if mode == DRAFT_GREEDY else qd
            drafts.append((draw(qd, int(rng.integers(0, 2 ** 53))), qd))
        ref_acc, ref_emit = verify_round(S, call, a, P, list(p[:n_p]), drafts)
        mcd.mcd_accept_from_logits(dec.ctx, a, n_d, call, t(p), t(q),
                                   t(np.array([d for d, _ in drafts] or [0], dtype=np.int32)), emitted, out2)
        mcd.mcd_sync(dec.ctx)
        o = out2.cpu().numpy()
        assert int(o[0]) == ref_acc and int(o[1]) == len(ref_emit), (case, o, ref_acc, ref_emit)
        assert emitted.cpu().numpy()[: o[1]].tolist() == ref_emit, case
        n_acc_total += ref_acc
    assert n_acc_total > 0
    dec.close()


# ---------------------------------------------------------------- frames -----------
def test_tiny_frames_trace_parity(tiny):
    cfg = tiny.cfg
    worst = 0.0
    for f in range(12):
        fr = make_frame(cfg, f)
        codes, st, tr = tiny.decode(fr, f, stream_id=f % 3, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        worst = max(worst, check_trace_against_oracle(cfg, tiny.model, fr, f % 3, f, tr, codes, int(st[0]),
                                                      logit_tol=1e-5))
    print("tiny max |dlogit|", worst)


def _first_round_explained_by_a_near_tie(cfg, model, fr, frame_idx, trace, ref):
    """The GPU's decisions are the oracle sampler's on the GPU's fp32 logits (the trace
    check), so a frame whose codes differ from the oracle's own decode must first differ in
    a round fed identical inputs where the two fp32 logit rows -- within the tolerance of
    each other -- give different top-k / temperature distributions (a set or a weight on
    the other side of a boundary).  Returns that round; fails if every distribution of the
    first differing round is the same."""
    recs, vlog, dlog = mcd.parse_trace(np.asarray(trace, dtype=np.uint8), cfg.vocab)
    k, T = cfg.top_k, cfg.temperature
    for c, rd in enumerate(ref.rounds):
        r = recs[c]
        g_emit = [int(v) for v in r["emitted"][: int(r["n_emit"])]]
        g_next = [int(v) for v in r["next_drafts"][: int(r["n_next"])]]
        if g_emit == rd.emitted and g_next == rd.next_drafts:
            continue
        first = 1 if c == 0 else 0
        gp = [topk_dist(vlog[c, n], k, T) for n in range(first, int(r["n_rows"]))]
        op = [topk_dist(rd.verify_logits[pos], k, T) for pos in sorted(rd.verify_logits)]
        gq = [topk_dist(dlog[c, j], k, T) for j in range(len(g_next))]
        oq = [topk_dist(z, k, T) for z in rd.draft_logits]
        assert len(gp) == len(op) and len(gq) == len(oq), c
        differ = [i for i, (a, b) in enumerate(zip(gp + gq, op + oq)) if a.ids != b.ids or a.W != b.W]
        assert differ, f"frame {frame_idx} round {c}: same distributions, different decisions"
        return c
    raise AssertionError(f"frame {frame_idx}: codes differ but every round agrees")


def test_tiny_codes_equal_oracle_end_to_end(tiny):
    """The GPU's codes equal the oracle's own decode (its fp64 rows rounded to fp32); a frame
    may differ only where a near-tie in some distribution explains it."""
    cfg = tiny.cfg
    same = 0
    n = 40
    for f in range(n):
        fr = make_frame(cfg, 100 + f)
        codes, st, _ = tiny.decode(fr, 100 + f)
        ref = decode_frame(tiny.model, fr, frame_idx=100 + f, keep_logits=True)
        if list(codes) == ref.codes:
            same += 1
            assert int(st[0]) == ref.calls
            continue
        codes2, st2, tr = tiny.decode(fr, 100 + f, trace=True)
        assert list(codes2) == list(codes)                        # deterministic
        check_trace_against_oracle(cfg, tiny.model, fr, 0, 100 + f, tr, codes2, int(st2[0]), logit_tol=1e-5)
        _first_round_explained_by_a_near_tie(cfg, tiny.model, fr, 100 + f, tr, ref)
    assert same >= n - 4, f"{n - same} of {n} frames differ from the oracle"


def test_mcd_frame_trace_parity_full_size(big):
    """Eight full-size frames at the bench's launch configuration: every call's verify and
    draft logits within 2e-2 of the oracle's fp64 rows, every decision identical."""
    cfg = big.cfg
    worst = 0.0
    for f in range(8):
        fr = make_frame(cfg, f)
        codes, st, tr = big.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        worst = max(worst, check_trace_against_oracle(cfg, big.model, fr, 0, f, tr, codes, int(st[0]),
                                                      logit_tol=2e-2))
    print("bf16 max |dlogit|", worst)


def test_mcd_frames_are_complete_and_bounded(big):
    cfg = big.cfg
    frames = 50
    calls = 0
    for f in range(frames):
        codes, st, _ = big.decode(make_frame(cfg, f), f)
        assert st[4] == 0 and st[1] == cfg.n_pos
        assert (codes >= 0).all() and (codes < cfg.vocab).all()
        assert 1 + math.ceil((cfg.n_pos - 1) / (cfg.draft_len + 1)) <= st[0] <= cfg.n_pos
        assert st[3] <= st[2]
        calls += int(st[0])
    assert calls <= frames * cfg.n_pos


@pytest.mark.parametrize("variant", ["ar", "k7", "greedy", "topk_all"])
def test_tiny_variants_trace_parity(variant):
    cfg = {"ar": TINY.replace(draft_len=0), "k7": TINY.replace(draft_len=7, n_pos=12),
           "greedy": TINY.replace(draft_mode=DRAFT_GREEDY), "topk_all": TINY.replace(top_k=64)}[variant]
    env = Env(cfg)
    for f in range(4):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        check_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]), logit_tol=1e-5,
                                   draft_mode=cfg.draft_mode)
        if variant == "ar":
            assert int(st[0]) == cfg.n_pos
    env.dec.close()


# ------------------------------------------------- batched streams ---------------------
def decode_many(env, frames, frame_idx, stream_ids):
    """One mcd_decode_frames launch over len(frames) streams, traced."""
    cfg = env.cfg
    n = len(frames)
    ins = [env.frame_inputs(fr) for fr in frames]
    cond = torch.stack([c for c, _, _ in ins])
    c0 = torch.cat([c for _, c, _ in ins]) if cfg.c0_vocab else None
    emb = torch.stack([e for _, _, e in ins]) if not cfg.c0_vocab else None
    codes = torch.full((n, cfg.n_pos), -1, dtype=torch.int32, device=DEV)
    stats = torch.zeros((n, 8), dtype=torch.int32, device=DEV)
    tr = torch.zeros(mcd.mcd_trace_bytes(env.dec.ctx), dtype=torch.uint8, device=DEV)
    mcd.mcd_set_trace(env.dec.ctx, tr)
    mcd.mcd_decode_frames(env.dec.ctx, stream_ids, frame_idx, cond, c0, emb, codes, stats)
    mcd.mcd_sync(env.dec.ctx)
    mcd.mcd_set_trace(env.dec.ctx, None)
    per = tr.numel() // cfg.max_streams
    trh = tr.cpu().numpy()
    return codes.cpu().numpy(), stats.cpu().numpy(), [trh[i * per:(i + 1) * per] for i in range(n)]


@pytest.mark.parametrize("cfg", [TINY.replace(max_streams=2), TINY.replace(draft_len=0, max_streams=4),
                                 TINY.replace(draft_len=1, max_streams=4), TINY.replace(draft_len=3, max_streams=8),
                                 TINY.replace(draft_len=3, max_streams=3)])
def test_batched_streams_trace_parity(cfg):
    """Several streams in one launch, rows re-packed every call: each stream's calls match
    the oracle decoding that stream alone (its own counters and KV cache)."""
    env = Env(cfg)
    for rep in range(3):
        n = cfg.max_streams - (rep % 2)            # also a launch with fewer streams than allowed
        fidx = [10 * rep + s for s in range(n)]
        sids = [7 + s for s in range(n)]
        frames = [make_frame(cfg, f) for f in fidx]
        codes, st, trs = decode_many(env, frames, fidx, sids)
        for s in range(n):
            assert st[s, 4] == 0 and st[s, 1] == cfg.n_pos
            check_trace_against_oracle(cfg, env.model, frames[s], sids[s], fidx[s], trs[s], codes[s], int(st[s, 0]),
                                       logit_tol=1e-5)
    env.dec.close()


@pytest.mark.parametrize("n_streams", [2, 4, 8])
def test_batched_streams_full_size(n_streams):
    """Up to 16 packed rows use the bf16 hi/lo operand, 17..32 a single bf16 operand."""
    cfg = MCD.replace(max_streams=n_streams)
    env = Env(cfg)
    fidx, sids = [4 + 5 * s for s in range(n_streams)], [3 + 2 * s for s in range(n_streams)]
    frames = [make_frame(cfg, f) for f in fidx]
    codes, st, trs = decode_many(env, frames, fidx, sids)
    for s in range(n_streams):
        assert st[s, 4] == 0 and st[s, 1] == cfg.n_pos
        err = check_trace_against_oracle(cfg, env.model, frames[s], sids[s], fidx[s], trs[s], codes[s],
                                         int(st[s, 0]), logit_tol=2e-2)
        print("batched stream", s, "max |dlogit|", err)
    env.dec.close()


def test_batched_streams_reject_shapes_beyond_the_gemm_path():
    for cfg in (MCD.replace(max_streams=128, draft_len=4),         # 640 packed rows > 512
                MCD.replace(max_streams=129),                      # more than 128 streams
                TINY.replace(max_streams=16)):                     # fp32 weights beyond 32 packed rows
        with pytest.raises(mcd.MCDError) as e:
            mcd.Decoder(cfg)
        assert e.value.status == 7


# ------------------------------------------------- batched GEMM path (> 32 rows) ------
TINY_BF16 = TINY.replace(weight_dtype=1)


@pytest.mark.parametrize("cfg", [TINY_BF16.replace(max_streams=16), TINY_BF16.replace(max_streams=24, draft_len=3),
                                 TINY_BF16.replace(max_streams=40, draft_len=1),
                                 TINY_BF16.replace(max_streams=12, draft_len=0, n_pos=6),
                                 TINY_BF16.replace(max_streams=33, draft_len=3, vocab=256)])
def test_gemm_path_trace_parity_tiny_bf16(cfg):
    """More than 32 packed rows per call: the batched GEMM path (one graph launch per frame;
    tensor-core GEMMs for the backbone, and for the LM heads when the vocabulary is a
    multiple of 128).  Every stream's calls match the oracle decoding that stream alone."""
    env = Env(cfg)
    for rep in range(2):
        n = cfg.max_streams - 3 * rep             # also fewer streams than the context allows
        fidx = [100 * rep + 3 * s for s in range(n)]
        sids = [11 + s for s in range(n)]
        frames = [make_frame(cfg, f) for f in fidx]
        codes, st, trs = decode_many(env, frames, fidx, sids)
        worst = 0.0
        for s in range(n):
            assert st[s, 4] == 0 and st[s, 1] == cfg.n_pos, (s, st[s])
            worst = max(worst, check_trace_against_oracle(cfg, env.model, frames[s], sids[s], fidx[s], trs[s],
                                                          codes[s], int(st[s, 0]), logit_tol=2e-2))
        print(cfg.max_streams, "streams: max |dlogit|", worst)
    env.dec.close()


@pytest.mark.parametrize("n_streams,checked", [(32, (0, 13, 31)), (128, tuple(range(128)))])
def test_gemm_path_full_size(n_streams, checked):
    """MultiCodeDecoder bf16 at B = 32 and 128 streams (128 and 512 packed rows): every
    stream finishes its frame; at B = 128 every stream (three sampled ones at B = 32)
    replays exactly against the oracle."""
    cfg = MCD.replace(max_streams=n_streams)
    env = Env(cfg)
    fidx, sids = [7 + s for s in range(n_streams)], [1000 + s for s in range(n_streams)]
    frames = [make_frame(cfg, f) for f in fidx]
    codes, st, trs = decode_many(env, frames, fidx, sids)
    assert (st[:, 4] == 0).all() and (st[:, 1] == cfg.n_pos).all()
    assert ((codes >= 0) & (codes < cfg.vocab)).all()
    for s in checked:
        err = check_trace_against_oracle(cfg, env.model, frames[s], sids[s], fidx[s], trs[s], codes[s],
                                         int(st[s, 0]), logit_tol=2e-2)
        print("gemm path stream", s, "of", n_streams, "max |dlogit|", err)
    # a second frame on the same context (the graph is reused)
    codes2, st2, _ = decode_many(env, frames, [f + 1 for f in fidx], sids)
    assert (st2[:, 1] == cfg.n_pos).all()
    env.dec.close()


# ------------------------------------------------- sparse tree verification (Fig. 2) ---
def _trees():
    from oracle.tree import Tree, grow_tree
    fig2 = Tree(parent=[-1, -1, 0, 0, 1, 2, 4, 4], rank=[0, 1, 0, 1, 0, 0, 0, 1])
    big = grow_tree([[0.5, 0.3, 0.2, 0.1, 0.05], [0.4, 0.25, 0.1], [0.3, 0.2]], 31)
    # the sweep's larger sizes (Fig. 4: N = 32, 48, 64), grown for rank-decreasing statistics
    # of 8 candidates at each of 3 depths
    acc = [[0.6 / (r + 1) ** 0.5 for r in range(8)] for _ in range(3)]
    return {"chain3": Tree.chain(3), "fig2": fig2, "wide": Tree(parent=[-1, -1, -1, -1], rank=[0, 1, 2, 3]),
            "big31": big, "grown32": grow_tree(acc, 32), "grown48": grow_tree(acc, 48),
            "grown64": grow_tree(acc, 64)}


def test_grown_trees_need_two_and_three_passes():
    t = _trees()
    assert [t[k].n for k in ("big31", "grown32", "grown48", "grown64")] == [31, 32, 48, 64]
    assert max(t["grown64"].depth) == 3 and max(t["grown64"].rank) == 7


@pytest.mark.parametrize("name", ["chain3", "fig2", "wide", "big31", "grown32", "grown48", "grown64"])
def test_tree_mode_trace_parity_tiny(name):
    """TREE mode: every call's rows, logits (1e-5), walk, kept path, codes and next candidates
    against the oracle; the 31-node tree packs 32 rows per call, the 32-, 48- and 64-node
    trees run 33, 49 and 65 rows in two and three passes."""
    tree = _trees()[name]
    cfg = TINY.replace(draft_mode=3, draft_len=3, n_pos=8)
    env = Env(cfg)
    mcd.mcd_set_tree(env.dec.ctx, tree.parent, tree.rank)
    worst = 0.0
    for f in range(4):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, stream_id=1, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos, st
        worst = max(worst, check_tree_trace_against_oracle(cfg, env.model, fr, 1, f, tr, codes, int(st[0]), tree,
                                                           logit_tol=1e-5))
    print(name, "max |dlogit|", worst)
    if tree.n > 31:
        trecs = mcd.parse_tree_trace(np.asarray(tr, dtype=np.uint8), cfg.vocab)[0]
        rows = [int(r["n_rows"]) for r in trecs[1:int(st[0])]]
        assert max(rows) == 1 + tree.n, rows                  # the full tree was fed at least once
        assert all(int(r["n_passes"]) == (n + 31) // 32 for r, n in zip(trecs[1:], rows))
    env.dec.close()


def test_chain_tree_equals_greedy_drafts_on_gpu():
    cfg = TINY.replace(draft_len=3, n_pos=8)
    tree_env = Env(cfg.replace(draft_mode=3))
    greedy_env = Env(cfg.replace(draft_mode=DRAFT_GREEDY))
    for f in range(6):
        fr = make_frame(cfg, f)
        a, sa, _ = tree_env.decode(fr, f)
        b, sb, _ = greedy_env.decode(fr, f)
        assert list(a) == list(b) and int(sa[0]) == int(sb[0]), f
    tree_env.dec.close()
    greedy_env.dec.close()


@pytest.mark.parametrize("name,frames", [("fig2", (0, 1)), ("grown64", (2,))])
def test_tree_mode_full_size(name, frames):
    """The full-size model (bf16 weights, logits within 2e-2): the Fig. 2 tree and the 64-node
    tree (65 rows in three passes)."""
    tree = _trees()[name]
    cfg = MCD.replace(draft_mode=3, draft_len=3)
    env = Env(cfg)
    mcd.mcd_set_tree(env.dec.ctx, tree.parent, tree.rank)
    for f in frames:
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        err = check_tree_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]), tree, logit_tol=2e-2)
        print("tree full size max |dlogit|", err)
    env.dec.close()


def test_tree_api_rejects_malformed_trees():
    env = Env(TINY.replace(draft_mode=3, draft_len=2))
    ctx = env.dec.ctx
    for parent, rank in (([0], [0]), ([-1, -1], [0, 0]), ([-1, 0, 1], [0, 0, 0]), ([-1], [8])):
        with pytest.raises(mcd.MCDError):
            mcd.mcd_set_tree(ctx, parent, rank)
    env.dec.close()
    with pytest.raises(mcd.MCDError):
        mcd.Decoder(TINY.replace(draft_mode=3, max_streams=2))


# ------------------------------------------------- noisy-target drafts (K sweep) ------
@pytest.mark.parametrize("K,sigma", [(1, 0.5), (2, 1.0), (3, 0.25), (7, 2.0)])
def test_tiny_noisy_target_trace_parity(K, sigma):
    """Drafts from the target's own logits plus counter-based Gaussian noise (the controlled-
    acceptance workload): every verify row and every noisy draft row within 1e-5 of the
    oracle, every decision identical."""
    cfg = TINY.replace(draft_len=K, n_pos=12 if K > 3 else TINY.n_pos, draft_mode=DRAFT_NOISY_TARGET,
                       noise_sigma=sigma)
    env = Env(cfg)
    for f in range(4):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        check_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]), logit_tol=1e-5,
                                   draft_mode=cfg.draft_mode)
    env.dec.close()


def test_noise_free_target_drafts_are_all_kept_on_gpu():
    cfg = TINY.replace(draft_len=2, draft_mode=DRAFT_NOISY_TARGET, noise_sigma=0.0)
    env = Env(cfg)
    for f in range(3):
        codes, st, _ = env.decode(make_frame(cfg, f), f)
        assert int(st[0]) == accounting.chain_calls_per_frame_all_accepted(2, cfg.n_pos)
        assert int(st[3]) == int(st[2])            # accepted == drafted
        ref = decode_frame(env.model, make_frame(cfg, f), frame_idx=f)
        assert list(codes) == ref.codes
    env.dec.close()


@pytest.mark.parametrize("sigma,frames", [(1.0, 1), (0.25, 6)])
def test_mcd_noisy_target_trace_parity_full_size(sigma, frames):
    """Full-size noisy-target frames; at sigma = 0.25 most drafts are kept, so calls that
    accept two or three drafts (and the bonus draw after them) run at full size."""
    cfg = MCD.replace(draft_mode=DRAFT_NOISY_TARGET, noise_sigma=sigma)
    env = Env(cfg)
    accepted = multi = 0
    for f in range(3, 3 + frames):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        err = check_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]), logit_tol=2e-2,
                                         draft_mode=cfg.draft_mode)
        recs, _, _ = mcd.parse_trace(np.asarray(tr, dtype=np.uint8), cfg.vocab)
        n_acc = [int(recs[c]["n_acc"]) for c in range(int(st[0]))]
        accepted += sum(n_acc)
        multi += sum(1 for v in n_acc if v >= 2)
        print("mcd noisy sigma", sigma, "max |dlogit|", err)
    if sigma <= 0.25:
        assert multi >= frames, (accepted, multi)
    env.dec.close()


def test_stepwise_api_matches_decode_frame(tiny):
    cfg = tiny.cfg
    dec = tiny.dec
    fr = make_frame(cfg, 7)
    ref, st, _ = tiny.decode(fr, 7)
    cond, c0, emb = tiny.frame_inputs(fr)
    mcd.mcd_begin_frame(dec.ctx, 0, 7, cond, c0, emb)
    emitted = torch.zeros(8, dtype=torch.int32, device=DEV)
    n_em = torch.zeros(1, dtype=torch.int32, device=DEV)
    logits = torch.zeros((8, cfg.vocab), dtype=torch.float32, device=DEV)
    got = []
    for call in range(cfg.n_pos + 1):
        mcd.mcd_verify_accept(dec.ctx, emitted, n_em, logits)
        mcd.mcd_sync(dec.ctx)
        k = int(n_em.item())
        if k == 0:
            break
        got += emitted.cpu().numpy()[:k].tolist()
    assert got == list(ref)
    assert call == int(st[0])


def test_stepwise_api_runs_noisy_target_passes():
    cfg = TINY.replace(draft_len=2, draft_mode=DRAFT_NOISY_TARGET, noise_sigma=0.5)
    env = Env(cfg)
    fr = make_frame(cfg, 5)
    ref, st, _ = env.decode(fr, 5)
    cond, c0, emb = env.frame_inputs(fr)
    mcd.mcd_begin_frame(env.dec.ctx, 0, 5, cond, c0, emb)
    emitted = torch.zeros(8, dtype=torch.int32, device=DEV)
    n_em = torch.zeros(1, dtype=torch.int32, device=DEV)
    got = []
    for call in range(cfg.n_pos + 1):
        mcd.mcd_verify_accept(env.dec.ctx, emitted, n_em, None)   # a verify call + its drafting passes
        mcd.mcd_sync(env.dec.ctx)
        k = int(n_em.item())
        if k == 0:
            break
        got += emitted.cpu().numpy()[:k].tolist()
    assert got == list(ref)
    assert call == int(st[0])
    env.dec.close()


def test_draft_api_matches_oracle(tiny):
    cfg = tiny.cfg
    dec = tiny.dec
    m = tiny.model
    _begin(dec, cfg, 2, 5)
    rng = np.random.default_rng(3)
    h = rng.standard_normal(cfg.hidden).astype(np.float32)
    K = cfg.draft_len
    ids = torch.zeros(K, dtype=torch.int32, device=DEV)
    q_ids = torch.zeros((K, cfg.top_k), dtype=torch.int32, device=DEV)
    q_w = torch.zeros((K, cfg.top_k), dtype=torch.int32, device=DEV)
    z = torch.zeros((K, cfg.vocab), dtype=torch.float32, device=DEV)
    S = Sampling(cfg, 2, 5)
    for k_pos in (1, 2):
        mcd.mcd_draft(dec.ctx, k_pos, 4, t(h), ids, q_ids, q_w, z)
        mcd.mcd_sync(dec.ctx)
        n_j = min(K, cfg.n_pos - k_pos)
        zz = z.cpu().numpy()
        for j in range(1, n_j + 1):
            ref = m.draft_logits(k_pos, j, h.astype(np.float64))
            assert np.max(np.abs(zz[j - 1] - ref)) < 1e-5
            q = S.dist(zz[j - 1])
            from oracle.sampler import draw
            assert int(ids[j - 1]) == draw(q, S.u(4, k_pos + j, 2))
            assert q_ids.cpu().numpy()[j - 1].tolist() == q.ids
            assert [int(v) for v in q_w.cpu().numpy().view(np.uint32)[j - 1]] == q.W


# ------------------------------------------------- W8A16 weight streaming -------------
@pytest.mark.parametrize("variant", ["tiny", "tiny_k0", "tiny_greedy"])
def test_w8a16_trace_parity_tiny(variant):
    """int8 weights quantised per row at load (R-Q1): every call against the oracle computing
    with q * s (1e-4: the activations enter the tensor cores as bf16 hi + lo pairs)."""
    cfg = {"tiny": TINY, "tiny_k0": TINY.replace(draft_len=0),
           "tiny_greedy": TINY.replace(draft_mode=DRAFT_GREEDY)}[variant].replace(weight_dtype=2)
    env = Env(cfg)
    worst = 0.0
    for f in range(5):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        worst = max(worst, check_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]),
                                                      logit_tol=1e-4))
    print(variant, "w8a16 max |dlogit|", worst)
    env.dec.close()


def test_w8a16_heads_are_quantised_like_the_oracle():
    """mcd_draft reads the int8 LM heads and their row scales directly: its draft logits
    equal the oracle's with the same q * s heads to fp32 rounding, so every quantised weight
    of the heads (and the draft offsets' bias) matches R-Q1."""
    cfg = TINY.replace(weight_dtype=2)
    env = Env(cfg)
    _begin(env.dec, cfg, 0, 0)
    h = np.random.default_rng(8).standard_normal(cfg.hidden).astype(np.float32)
    K = cfg.draft_len
    ids = torch.zeros(K, dtype=torch.int32, device=DEV)
    z = torch.zeros((K, cfg.vocab), dtype=torch.float32, device=DEV)
    for k_pos in (1, 2):
        mcd.mcd_draft(env.dec.ctx, k_pos, 0, t(h), ids, None, None, z)
        mcd.mcd_sync(env.dec.ctx)
        zz = z.cpu().numpy()
        for j in range(1, min(K, cfg.n_pos - k_pos) + 1):
            ref = env.model.draft_logits(k_pos, j, h.astype(np.float64))
            assert np.max(np.abs(zz[j - 1] - ref)) < 2e-6
    env.dec.close()


def test_w8a16_full_size():
    cfg = MCD.replace(weight_dtype=2)
    env = Env(cfg)
    for f in (0, 1):
        fr = make_frame(cfg, f)
        codes, st, tr = env.decode(fr, f, trace=True)
        assert st[4] == 0 and st[1] == cfg.n_pos
        err = check_trace_against_oracle(cfg, env.model, fr, 0, f, tr, codes, int(st[0]), logit_tol=2e-2)
        print("w8a16 full size max |dlogit|", err)
    env.dec.close()


def test_bad_c0_fails_the_frame_without_faulting(big):
    cfg = big.cfg
    fr = make_frame(cfg, 0)
    cond = t(fr.cond)
    c0 = t(np.array([cfg.c0_vocab + 5], dtype=np.int32))
    codes = torch.zeros(cfg.n_pos, dtype=torch.int32, device=DEV)
    mcd.mcd_decode_frame(big.dec.ctx, 0, 0, cond, c0, None, codes, None)
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_sync(big.dec.ctx)
    assert e.value.status == 1
    # the context stays usable
    codes2, st, _ = big.decode(fr, 0)
    assert st[4] == 0 and st[1] == cfg.n_pos


@pytest.mark.parametrize("env_name,pinned", [("tiny", False), ("tiny", True), ("big", True)])
def test_host_buffer_api_matches_device_api(env_name, pinned, request):
    """mcd_decode_frame_host (one gathered H2D copy, one D2H copy of codes, stats and the
    error word) returns what mcd_decode_frame returns on device buffers; tiny feeds c0 as
    an embedding, the full-size model as a token."""
    env = request.getfixturevalue(env_name)
    cfg = env.cfg
    for f in range(4):
        fr = make_frame(cfg, 300 + f)
        ref_codes, ref_st, _ = env.decode(fr, 300 + f, stream_id=1)
        cond = torch.from_numpy(np.ascontiguousarray(fr.cond, dtype=np.float32))
        c0 = torch.tensor([fr.c0], dtype=torch.int32) if cfg.c0_vocab > 0 else None
        emb = torch.from_numpy(np.ascontiguousarray(fr.c0_emb, dtype=np.float32)) if cfg.c0_vocab == 0 else None
        codes = torch.full((cfg.n_pos,), -1, dtype=torch.int32)
        st = torch.zeros(8, dtype=torch.int32)
        if pinned:
            cond, codes, st = cond.pin_memory(), codes.pin_memory(), st.pin_memory()
            c0 = c0.pin_memory() if c0 is not None else None
            emb = emb.pin_memory() if emb is not None else None
        mcd.mcd_decode_frame_host(env.dec.ctx, 1, 300 + f, cond, c0, emb, codes, st)
        assert codes.numpy().tolist() == ref_codes.tolist()
        assert st.numpy().tolist() == ref_st.tolist()


def test_host_buffer_api_reports_bad_c0_and_recovers(big):
    cfg = big.cfg
    fr = make_frame(cfg, 0)
    cond = np.ascontiguousarray(fr.cond, dtype=np.float32)
    codes = np.full(cfg.n_pos, -7, dtype=np.int32)
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_decode_frame_host(big.dec.ctx, 0, 0, cond, np.array([cfg.c0_vocab + 5], dtype=np.int32), None, codes)
    assert e.value.status == 1
    assert (codes == -7).all()                     # results of a failed frame are not written
    mcd.mcd_sync(big.dec.ctx)                      # the error was cleared by the failing call
    st = np.zeros(8, dtype=np.int32)
    mcd.mcd_decode_frame_host(big.dec.ctx, 0, 0, cond, np.array([fr.c0], dtype=np.int32), None, codes, st)
    ref_codes, ref_st, _ = big.decode(fr, 0)
    assert codes.tolist() == ref_codes.tolist() and st.tolist() == ref_st.tolist()


@pytest.mark.parametrize("kind", [0, 1])
def test_bounded_wait_times_out_and_the_context_stays_usable(big, kind):
    """Failure detection without a fault: the library's bounded wait, run on a counter
    (kind 0) or an mbarrier (kind 1) that nothing signals, gives up after its limit,
    reports MCD_ERR_TIMEOUT through the status word, and the context decodes the next
    frame exactly as before."""
    cfg = big.cfg
    fr = make_frame(cfg, 11)
    ref_codes, ref_st, _ = big.decode(fr, 11)
    status, waited = mcd.mcd_test_bounded_wait(big.dec.ctx, kind, 2_000_000)
    assert status == 5, mcd.mcd_status_str(status)                 # MCD_ERR_TIMEOUT
    assert 2_000_000 <= waited < 1_000_000_000, waited
    mcd.mcd_sync(big.dec.ctx)                                       # cleared by the call
    codes, st, _ = big.decode(fr, 11)
    assert codes.tolist() == ref_codes.tolist() and st.tolist() == ref_st.tolist()
    with pytest.raises(mcd.MCDError):
        mcd._check("mcd_test_bounded_wait", mcd.load_library().mcd_test_bounded_wait(big.dec.ctx, 2, 2_000_000, None))


# ---------------------------------------------------------------- distribution -----
def test_chi_square_of_gpu_codes_against_exact_law(tiny):
    cfg = tiny.cfg
    pm = PrefixModel(tiny.model, make_frame(cfg, 0))
    ar = ar_distribution(pm, cfg.n_pos)
    _, exp_calls = spec_distribution(pm, cfg.n_pos, cfg.draft_len)
    fr = make_frame(cfg, 0)
    cond, c0, emb = tiny.frame_inputs(fr)
    n = 20000
    codes = torch.zeros((n, cfg.n_pos), dtype=torch.int32, device=DEV)
    stats = torch.zeros((n, 8), dtype=torch.int32, device=DEV)
    for i in range(n):
        mcd.mcd_decode_frame(tiny.dec.ctx, 1, 10_000 + i, cond, c0, emb, codes[i], stats[i])
    mcd.mcd_sync(tiny.dec.ctx)
    codes, stats = codes.cpu().numpy(), stats.cpu().numpy()
    assert (stats[:, 4] == 0).all()
    from scipy import stats as ss
    for cells in ((0,), (1,), (2,), (3,), (0, 1)):
        law = Counter()
        for seq, pr in ar.items():
            law[tuple(seq[c] for c in cells)] += float(pr)
        obs = Counter(tuple(row[list(cells)]) for row in codes)
        keys = sorted(law)
        e = np.array([law[k] * n for k in keys])
        o = np.array([obs.get(k, 0) for k in keys])
        assert sum(obs.values()) == o.sum() == n, cells           # nothing outside the support
        big_ = e >= 5
        o2 = np.append(o[big_], o[~big_].sum())
        e2 = np.append(e[big_], e[~big_].sum())
        if e2[-1] == 0:
            o2, e2 = o2[:-1], e2[:-1]
        p = ss.chisquare(o2, e2 * o2.sum() / e2.sum()).pvalue
        assert p > 1e-4, (cells, p)
    mean_calls = stats[:, 0].mean()
    exp_calls = float(exp_calls)
    assert abs(mean_calls - exp_calls) < 4 * stats[:, 0].std() / math.sqrt(n) + 1e-3, (mean_calls, exp_calls)


def _decode_fixed_input(env, n, stream_id, frame0):
    """n frames of one fixed frame input (frame 0's cond and c0), frame indices frame0 + i, so
    only the Philox counters differ between frames."""
    cfg = env.cfg
    cond, c0, emb = env.frame_inputs(make_frame(cfg, 0))
    codes = torch.zeros((n, cfg.n_pos), dtype=torch.int32, device=DEV)
    stats = torch.zeros((n, 8), dtype=torch.int32, device=DEV)
    for i in range(n):
        mcd.mcd_decode_frame(env.dec.ctx, stream_id, frame0 + i, cond, c0, emb, codes[i], stats[i])
    mcd.mcd_sync(env.dec.ctx)
    codes, stats = codes.cpu().numpy(), stats.cpu().numpy()
    assert (stats[:, 4] == 0).all() and (stats[:, 1] == cfg.n_pos).all()
    return codes, stats


def _chi2_goodness(obs: Counter, law: dict, n: int, min_expected=5.0):
    from scipy import stats as ss
    keys = sorted(law)
    e = np.array([law[k] * n for k in keys])
    o = np.array([obs.get(k, 0) for k in keys])
    assert o.sum() == n, "codes outside the law's support"
    big_ = e >= min_expected
    o2, e2 = np.append(o[big_], o[~big_].sum()), np.append(e[big_], e[~big_].sum())
    if e2[-1] == 0:
        o2, e2 = o2[:-1], e2[:-1]
    return ss.chisquare(o2, e2 * o2.sum() / e2.sum()).pvalue


def test_chi_square_full_size_against_exact_law_and_ar(big):
    """MCD bf16 workload (V = 2048, top-k 50, T 0.9, K = 3): 20,000 frames of one fixed
    frame input.  (1) The c1 histogram and the (c1, c2) histogram against the exact law the
    oracle gives for that input (c1 ~ p_1; c2 | c1 ~ p_2 of the row fed c1: one pass for c1
    and one row per c1 in its top-50), i.e. speculative decoding emits the target's top-k
    law (Sec. 3.2).  (2) A two-sample test of the speculative codes against 20,000 frames
    of the non-speculative decoder (K = 0, same kernels) at every position c1..c15."""
    from scipy import stats as ss
    cfg = big.cfg
    n = 20000
    spec, _ = _decode_fixed_input(big, n, 2, 50_000)
    # exact law of c1 and of (c1, c2) from the oracle's fp64 rows
    m, fr = big.model, make_frame(cfg, 0)
    kv = m.new_kv()
    m.row(kv, np.asarray(fr.cond, dtype=np.float64), 0)
    h1 = m.row(kv, m.c0_row(fr.c0, fr.c0_emb), 1)
    p1 = topk_dist(m.verify_logits(1, h1).astype(np.float32), cfg.top_k, cfg.temperature)
    law1 = {(x,): p1.prob(x) for x in p1.ids}
    law12 = {}
    for x in p1.ids:
        h2 = m.row(kv, m.code_row(1, x), 2)
        p2 = topk_dist(m.verify_logits(2, h2).astype(np.float32), cfg.top_k, cfg.temperature)
        for y in p2.ids:
            law12[(x, y)] = p1.prob(x) * p2.prob(y)
    pv1 = _chi2_goodness(Counter((int(r[0]),) for r in spec), law1, n)
    pv12 = _chi2_goodness(Counter((int(r[0]), int(r[1])) for r in spec), law12, n)
    print("full-size chi-square p: c1", pv1, "(c1, c2)", pv12)
    assert pv1 > 1e-4 and pv12 > 1e-4, (pv1, pv12)
    # speculative vs autoregressive, position by position
    ar_env = Env(cfg.replace(draft_len=0), big.w)
    try:
        ar, _ = _decode_fixed_input(ar_env, n, 3, 90_000)
    finally:
        ar_env.dec.close()
    worst = 1.0
    for t in range(cfg.n_pos):
        cs, ca = Counter(spec[:, t].tolist()), Counter(ar[:, t].tolist())
        keys = sorted(set(cs) | set(ca))
        tab = np.array([[cs.get(k, 0) for k in keys], [ca.get(k, 0) for k in keys]], dtype=np.float64)
        common = tab.sum(axis=0) >= 10
        tab = np.concatenate([tab[:, common], tab[:, ~common].sum(axis=1, keepdims=True)], axis=1)
        tab = tab[:, tab.sum(axis=0) > 0]
        p = ss.chi2_contingency(tab)[1] if tab.shape[1] > 1 else 1.0
        worst = min(worst, p)
        assert p > 1e-5, (t, p)
    print("spec vs AR two-sample chi-square: smallest p over c1..c15", worst)
