"""mcd_topk_softmax_static (no device allocation, static scratch) against mcd_topk_softmax
and against the oracle's top-k / temperature distributions.

Collected last on purpose: it must pass both in a fresh process, where its first call
does the one-time set-up, and after every other test has used the library.  One test runs
the entry point in a child process that never creates a context, to show that after the
set-up call further calls leave the device's free memory unchanged."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2609_37007_gb300.synth import MCD, TINY

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _rows(n, V, seed):
    import torch
    g = torch.Generator().manual_seed(seed)
    lg = torch.randn(n, V, generator=g) * 0.7
    lg[:, ::7] = lg[:, 3:4]          # ties across ids
    return lg.cuda()


@pytest.mark.parametrize("cfg,n_rows", [(TINY, 5), (MCD, 16), (MCD, 128)])
def test_static_matches_context_entry_point_twice(cfg, n_rows):
    import torch
    from paper_2609_37007_gb300 import mcd
    dec = mcd.Decoder(cfg)
    try:
        k, V = cfg.top_k, cfg.vocab
        lg = _rows(n_rows, V, 1000 + n_rows)
        ids_ref = torch.zeros((n_rows, k), dtype=torch.int32, device="cuda")
        w_ref = torch.zeros((n_rows, k), dtype=torch.int32, device="cuda")
        s_ref = torch.zeros((n_rows,), dtype=torch.int64, device="cuda")
        mcd.mcd_topk_softmax(dec.ctx, n_rows, lg, ids_ref, w_ref, s_ref)
        mcd.mcd_sync(dec.ctx)
        stream = torch.cuda.current_stream()
        for rep in range(2):                                        # two calls in a row
            ids = torch.full((n_rows, k), -7, dtype=torch.int32, device="cuda")
            w = torch.zeros((n_rows, k), dtype=torch.int32, device="cuda")
            s = torch.zeros((n_rows,), dtype=torch.int64, device="cuda")
            mcd.mcd_topk_softmax_static(n_rows, V, k, cfg.temperature, lg, ids, w, s, stream)
            torch.cuda.synchronize()
            assert torch.equal(ids, ids_ref), rep
            assert torch.equal(w, w_ref), rep
            assert torch.equal(s, s_ref), rep
        ids_h = ids.cpu().numpy()
        assert (np.diff(ids_h, axis=1) > 0).all()                   # ascending id order
        if cfg is TINY:                                             # and the oracle's law
            from oracle.sampler import topk_dist
            lg_h, w_h, s_h = lg.cpu().numpy(), w.cpu().numpy().view(np.uint32), s.cpu().numpy()
            for r in range(n_rows):
                d = topk_dist(lg_h[r], k, cfg.temperature)
                assert ids_h[r].tolist() == d.ids, r
                assert [int(v) for v in w_h[r]] == d.W, r
                assert int(s_h[r]) == d.S, r
    finally:
        dec.close()


# Child process: no mcd_ctx anywhere, every buffer allocated before the first call; the
# free device memory after the set-up call must not move over further calls of up to the
# scratch's row limit, and every row must equal the oracle's distribution.
_CHILD = r"""
import sys
sys.path.insert(0, sys.argv[1])
import numpy as np, torch
from paper_2609_37007_gb300 import mcd
from paper_2609_37007_gb300.synth import MCD
from oracle.sampler import topk_dist
V, k, T, n = MCD.vocab, MCD.top_k, MCD.temperature, mcd.STATIC_TOPK_MAX_ROWS
g = torch.Generator().manual_seed(77)
lg = (torch.randn(n, V, generator=g) * 0.7).cuda()
ids = torch.zeros((n, k), dtype=torch.int32, device="cuda")
w = torch.zeros((n, k), dtype=torch.int32, device="cuda")
s = torch.zeros((n,), dtype=torch.int64, device="cuda")
stream = torch.cuda.current_stream()
mcd.mcd_topk_softmax_static(4, V, k, T, lg, ids, w, s, stream)     # one-time set-up
torch.cuda.synchronize()
free0 = torch.cuda.mem_get_info()[0]
for rows in (n, 17, n):
    mcd.mcd_topk_softmax_static(rows, V, k, T, lg, ids, w, s, stream)
    torch.cuda.synchronize()
free1 = torch.cuda.mem_get_info()[0]
assert free1 == free0, (free0, free1)
lg_h, ids_h, w_h, s_h = lg.cpu().numpy(), ids.cpu().numpy(), w.cpu().numpy().view(np.uint32), s.cpu().numpy()
for r in range(n):
    d = topk_dist(lg_h[r], k, T)
    assert ids_h[r].tolist() == d.ids and [int(v) for v in w_h[r]] == d.W and int(s_h[r]) == d.S, r
print("NO_ALLOC_OK", free0)
"""


def test_static_allocates_nothing_without_a_context():
    r = subprocess.run([sys.executable, "-c", _CHILD, ROOT], capture_output=True, text=True, timeout=600)
    assert r.returncode == 0 and "NO_ALLOC_OK" in r.stdout, r.stdout[-2000:] + r.stderr[-2000:]


def test_static_rejects_sizes_beyond_its_scratch():
    import torch
    from paper_2609_37007_gb300 import mcd
    V, k = MCD.vocab, MCD.top_k
    n = mcd.load_library().mcd_topk_softmax_static  # raw status, no exception
    lg = _rows(4, V, 5)
    ids = torch.zeros((4, k), dtype=torch.int32, device="cuda")
    st = n(mcd.STATIC_TOPK_MAX_ROWS + 1, V, k, 0.9, lg.data_ptr(), ids.data_ptr(), None, None, None)
    assert mcd.STATUS_NAMES[st] == "MCD_ERR_UNSUPPORTED"
    st = n(4, V, 129, 0.9, lg.data_ptr(), ids.data_ptr(), None, None, None)
    assert mcd.STATUS_NAMES[st] == "MCD_ERR_UNSUPPORTED"
    st = n(4, V + 8, k, 0.9, lg.data_ptr(), ids.data_ptr(), None, None, None)
    assert mcd.STATUS_NAMES[st] == "MCD_ERR_INVALID_ARG"
    st = n(4, V, k, 0.0, lg.data_ptr(), ids.data_ptr(), None, None, None)
    assert mcd.STATUS_NAMES[st] == "MCD_ERR_INVALID_ARG"
    assert n(0, V, k, 0.9, lg.data_ptr(), ids.data_ptr(), None, None, None) == 0
    torch.cuda.synchronize()
