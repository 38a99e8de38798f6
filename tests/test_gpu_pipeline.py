"""GPU parity of the full frame pipeline (outer CodeDecoder + MultiCodeDecoder, Fig. 1)
against the CPU oracle; every call goes through the C ABI (include/mcd_pipeline.h).

Teacher-forced replay: each frame's GPU outputs (c0 logits, cond, c0 embedding, the inner
frame's trace and codes) are checked against the oracle run on the GPU's own earlier
codes:
  * c0 logits and cond (the post-norm hidden state) within tolerance of the oracle
    (1e-5 for the fp32 model, 2e-2 for bf16);
  * c0 identical to the oracle sampler's draw on the GPU's fp32 logits (counter of
    position 0);
  * the c0 embedding exactly row c0 of the c0 table;
  * the inner frame through tests/parity.py, fed the cond / c0 embedding the GPU produced.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2609_37007_gb300 import build as _build  # noqa: E402
from paper_2609_37007_gb300 import mcd  # noqa: E402
from paper_2609_37007_gb300.synth import (OUTER, OUTER_TINY, PIPE_INNER, TINY, WEIGHT_BF16, FrameInput,  # noqa: E402
                                          make_outer_weights, make_prompt, make_weights, outer_weights_as_f32,
                                          weights_as_f32)
from oracle.codedecoder import CodeDecoder, Pipeline as OraclePipeline, sample_c0  # noqa: E402
from oracle.model import Model  # noqa: E402
from parity import check_trace_against_oracle  # noqa: E402

DEV = torch.device("cuda:0")
_build.build()


class PipeEnv:
    def __init__(self, ocfg, icfg):
        self.ocfg, self.icfg = ocfg, icfg
        self.iw = make_weights(icfg)
        self.ow = make_outer_weights(ocfg, icfg)
        self.pl = mcd.Pipeline(ocfg, icfg, self.ow, self.iw)
        self._oracle = None

    @property
    def oracle(self):
        if self._oracle is None:
            inner = Model(self.icfg, weights_as_f32(self.icfg, self.iw))
            self._oracle = CodeDecoder(self.ocfg, outer_weights_as_f32(self.ocfg, self.ow), inner)
        return self._oracle

    def run(self, prompt, n_frames, stream_id=0, traced=None):
        """Prefill, then n_frames frames one pipeline call each.  Returns per-frame
        (codes, stats, inner trace or None) and the outer trace [n_frames, record]."""
        o, ictx = self.pl.o, self.pl.inner.ctx
        tf = mcd.mcd_outer_trace_floats(o)
        otr = torch.zeros(n_frames * tf, dtype=torch.float32, device=DEV)
        mcd.mcd_outer_set_trace(o, otr, n_frames)
        mcd.mcd_outer_prefill(o, stream_id, torch.from_numpy(np.asarray(prompt, dtype=np.int32)).to(DEV))
        W = self.icfg.n_pos + 1
        out = []
        for f in range(n_frames):
            codes = torch.full((W,), -1, dtype=torch.int32, device=DEV)
            stats = torch.zeros(8, dtype=torch.int32, device=DEV)
            keep = traced is None or f in traced
            tr = torch.zeros(mcd.mcd_trace_bytes(ictx), dtype=torch.uint8, device=DEV) if keep else None
            mcd.mcd_set_trace(ictx, tr)
            mcd.mcd_pipeline_frames(o, 1, codes, stats=stats)
            mcd.mcd_outer_sync(o)
            mcd.mcd_sync(ictx)
            out.append((codes.cpu().numpy(), stats.cpu().numpy(), tr.cpu().numpy() if keep else None))
        mcd.mcd_set_trace(ictx, None)
        mcd.mcd_outer_set_trace(o, None, 0)
        return out, otr.cpu().numpy().reshape(n_frames, tf)


def check_pipeline(env, prompt, frames, otr, tol, stream_id=0):
    ocfg, icfg = env.ocfg, env.icfg
    V0, H = ocfg.c0_vocab, ocfg.hidden
    pl = OraclePipeline(env.oracle, stream_id)
    pl.prefill(prompt)
    worst = 0.0
    prev = None
    for f, (codes, st, tr) in enumerate(frames):
        if f > 0:
            pl.step(prev)
        lg, cond, emb = otr[f, :V0], otr[f, V0:V0 + H], otr[f, V0 + H:V0 + 2 * H]
        err = max(float(np.max(np.abs(lg.astype(np.float64) - env.oracle.c0_logits(pl.h)))),
                  float(np.max(np.abs(cond.astype(np.float64) - pl.h))))
        worst = max(worst, err)
        assert err <= tol, f"frame {f}: c0 logits / hidden differ by {err}"
        c0 = sample_c0(ocfg, lg, stream_id, f)
        assert c0 == int(codes[0]), (f, c0, codes[0])
        assert np.array_equal(emb, env.oracle.w["c0_embed"][c0].astype(np.float32))
        assert int(st[4]) == 0 and int(st[1]) == icfg.n_pos
        assert all(0 <= int(c) < icfg.vocab for c in codes[1:])
        if tr is not None:
            worst = max(worst, check_trace_against_oracle(
                icfg, env.oracle.inner, FrameInput(cond=cond, c0=-1, c0_emb=emb), stream_id, f, tr, codes[1:],
                int(st[0]), logit_tol=tol))
        prev = [int(v) for v in codes]
    return worst


@pytest.fixture(scope="module")
def tiny_pipe():
    env = PipeEnv(OUTER_TINY.replace(prompt_len=45), TINY)
    yield env
    env.pl.close()


def test_tiny_pipeline_parity(tiny_pipe):
    env = tiny_pipe
    # 45 prompt rows: launches of 16, 16 and 13 rows; frames then add positions 45..50, so
    # key blocks hold cached and new keys, and some frame rows read only cached blocks
    prompt = make_prompt(env.ocfg)
    frames, otr = env.run(prompt, 6, stream_id=3)
    check_pipeline(env, prompt, frames, otr, 1e-5, stream_id=3)


def test_tiny_pipeline_repeatable_and_restartable(tiny_pipe):
    env = tiny_pipe
    prompt = make_prompt(env.ocfg, utterance=1)
    a, _ = env.run(prompt, 3)
    b, _ = env.run(prompt, 3)                     # a new prefill restarts the utterance
    assert [list(x[0]) for x in a] == [list(x[0]) for x in b]


def test_stepwise_outer_api_matches_pipeline_call(tiny_pipe):
    """mcd_outer_prefill / mcd_outer_step + mcd_outer_frame_inputs + mcd_decode_frame, driven
    by the caller, give the codes mcd_pipeline_frames gives."""
    env = tiny_pipe
    o, ictx = env.pl.o, env.pl.inner.ctx
    W, n = TINY.n_pos + 1, 5
    prompt = torch.from_numpy(make_prompt(env.ocfg, utterance=2)).to(DEV)
    ref = torch.full((n, W), -1, dtype=torch.int32, device=DEV)
    mcd.mcd_outer_prefill(o, 4, prompt)
    mcd.mcd_pipeline_frames(o, n, ref)
    got = torch.full((n, W), -1, dtype=torch.int32, device=DEV)
    lib = mcd.load_library()
    mcd.mcd_outer_prefill(o, 4, prompt, got[0, 0:1])
    for f in range(n):
        if f > 0:
            mcd.mcd_outer_step(o, got[f - 1], -1, got[f, 0:1])
        cond, emb, _, fi = mcd.mcd_outer_frame_inputs(o)
        assert fi == f
        mcd._check("mcd_decode_frame", lib.mcd_decode_frame(ictx, 4, fi, cond, None, emb, got[f, 1:].data_ptr(), None))
    mcd.mcd_outer_sync(o)
    mcd.mcd_sync(ictx)
    assert torch.equal(got, ref)


@pytest.mark.parametrize("variant", ["mha", "one_row_prompt", "ar_inner", "text_rows", "bf16"])
def test_tiny_pipeline_variants(variant):
    ocfg, icfg = OUTER_TINY, TINY
    if variant == "mha":
        ocfg = ocfg.replace(n_kv_heads=4, prompt_len=70)
    elif variant == "one_row_prompt":
        ocfg = ocfg.replace(prompt_len=1)
    elif variant == "ar_inner":
        icfg = icfg.replace(draft_len=0)
    elif variant == "bf16":
        ocfg, icfg = ocfg.replace(weight_dtype=WEIGHT_BF16, prompt_len=33), icfg.replace(weight_dtype=WEIGHT_BF16)
    tol = 2e-2 if variant == "bf16" else 1e-5
    env = PipeEnv(ocfg, icfg)
    try:
        prompt = make_prompt(ocfg)
        if variant != "text_rows":
            frames, otr = env.run(prompt, 4)
            check_pipeline(env, prompt, frames, otr, tol)
            return
        # per-frame text rows (the caption's t_i) through mcd_pipeline_frames
        o = env.pl.o
        W, V0, H = icfg.n_pos + 1, ocfg.c0_vocab, ocfg.hidden
        tf = mcd.mcd_outer_trace_floats(o)
        otr = torch.zeros(3 * tf, dtype=torch.float32, device=DEV)
        mcd.mcd_outer_set_trace(o, otr, 3)
        mcd.mcd_outer_prefill(o, 0, torch.from_numpy(prompt).to(DEV))
        codes = torch.full((3, W), -1, dtype=torch.int32, device=DEV)
        text = [-1, 17, 400]
        mcd.mcd_pipeline_frames(o, 3, codes, text_ids=text)
        mcd.mcd_outer_sync(o)
        got, tr = codes.cpu().numpy(), otr.cpu().numpy().reshape(3, tf)
        pl = OraclePipeline(env.oracle, 0)
        pl.prefill(prompt)
        for f in range(3):
            if f > 0:
                pl.step([int(v) for v in got[f - 1]], text[f])
            lg = tr[f, :V0]
            assert np.max(np.abs(lg.astype(np.float64) - env.oracle.c0_logits(pl.h))) <= 1e-5
            assert np.max(np.abs(tr[f, V0:V0 + H].astype(np.float64) - pl.h)) <= 1e-5
            assert sample_c0(ocfg, lg, 0, f) == int(got[f, 0])
    finally:
        env.pl.close()


def test_pipeline_errors_are_reported():
    env = PipeEnv(OUTER_TINY.replace(prompt_len=4, frames=2), TINY)     # KV capacity 5
    o = env.pl.o
    W = TINY.n_pos + 1
    codes = torch.full((3, W), -1, dtype=torch.int32, device=DEV)
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_pipeline_frames(o, 1, codes)                            # no prompt yet
    assert e.value.status == 2
    mcd.mcd_outer_prefill(o, 0, torch.arange(4, dtype=torch.int32, device=DEV))
    mcd.mcd_pipeline_frames(o, 2, codes)                                # frames 0 and 1 fill the cache
    mcd.mcd_outer_sync(o)
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_pipeline_frames(o, 1, codes[2:])                        # no room for frame 2
    assert e.value.status == 2
    bad = torch.tensor([1, OUTER_TINY.text_vocab + 5], dtype=torch.int32, device=DEV)
    mcd.mcd_outer_prefill(o, 0, bad)
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_outer_sync(o)                                           # the kernel refused the id
    assert e.value.status == 1
    env.pl.close()
    inner = mcd.Decoder(TINY.replace(c0_vocab=64), make_weights(TINY.replace(c0_vocab=64)))
    with pytest.raises(mcd.MCDError) as e:
        mcd.mcd_outer_create(OUTER_TINY, inner.ctx)                    # the inner model must take c0 vectors
    assert e.value.status == 1
    inner.close()


@pytest.fixture(scope="module")
def full_pipe():
    env = PipeEnv(OUTER.replace(prompt_len=600, frames=31), PIPE_INNER)
    yield env
    env.pl.close()


def test_full_size_pipeline_parity(full_pipe):
    """CodeDecoder-shaped bf16 model over a 600-token prompt and 31 frames, so that the last
    frame's row reads 630 cached positions (20 key blocks); inner frames traced at the
    first and last frames."""
    env = full_pipe
    prompt = make_prompt(env.ocfg)
    frames, otr = env.run(prompt, 31, traced={0, 1, 30})
    err = check_pipeline(env, prompt, frames, otr, 2e-2)
    assert err < 2e-2
