"""mcd_topk_softmax_static (no device allocation, static scratch) against mcd_topk_softmax.

Collected last on purpose: it must pass both in a fresh process, where its first call
does the one-time set-up, and after every other test has used the library."""
import numpy as np
import pytest

from paper_2609_37007_gb300.synth import MCD, TINY

pytestmark = pytest.mark.gpu


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
    finally:
        dec.close()


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
