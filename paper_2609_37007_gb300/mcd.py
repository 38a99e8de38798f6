"""Thin ctypes binding of libmcd.so (include/mcd.h); argument marshalling only.

Every function has the name of the C entry point it wraps.  Device buffers are torch CUDA
tensors (their data_ptr() is passed through); weights are numpy arrays.  Nothing here
computes any part of the decoding path, and there is no fallback: if the library is
missing, loading it raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, Optional, Tuple

import numpy as np

from .synth import MCDConfig, OuterConfig

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmcd.so")
_lib: Optional[ctypes.CDLL] = None

MCD_OK = 0
STATUS_NAMES = {0: "MCD_OK", 1: "MCD_ERR_INVALID_ARG", 2: "MCD_ERR_STATE", 3: "MCD_ERR_CUDA",
                4: "MCD_ERR_OOM", 5: "MCD_ERR_TIMEOUT", 6: "MCD_ERR_WEIGHTS", 7: "MCD_ERR_UNSUPPORTED"}

MAX_CALLS = 16
MAX_ROWS = 8
STATIC_TOPK_MAX_ROWS = 128     # MCD_STATIC_TOPK_MAX_ROWS


class McdConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("n_pos", ctypes.c_int32), ("vocab", ctypes.c_int32), ("c0_vocab", ctypes.c_int32),
                ("rms_eps", ctypes.c_float), ("rope_base", ctypes.c_float),
                ("qk_norm", ctypes.c_int32), ("weight_dtype", ctypes.c_int32),
                ("draft_len", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("draft_mode", ctypes.c_int32),
                ("noise_sigma", ctypes.c_float), ("seed", ctypes.c_uint64), ("max_streams", ctypes.c_int32)]


class McdOuterConfig(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("c0_vocab", ctypes.c_int32), ("text_vocab", ctypes.c_int32),
                ("max_tokens", ctypes.c_int32), ("rms_eps", ctypes.c_float),
                ("rope_base", ctypes.c_float), ("qk_norm", ctypes.c_int32),
                ("weight_dtype", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("temperature", ctypes.c_float), ("seed", ctypes.c_uint64)]


CALL_TRACE_DTYPE = np.dtype([("a", "<i4"), ("n_rows", "<i4"), ("pos0", "<i4"), ("n_drafts", "<i4"),
                             ("input_ids", "<i4", 8), ("drafts", "<i4", 8), ("n_acc", "<i4"),
                             ("n_emit", "<i4"), ("emitted", "<i4", 8), ("n_next", "<i4"),
                             ("next_drafts", "<i4", 8), ("draft_row", "<i4"), ("reserved", "<i4", 24)])
assert CALL_TRACE_DTYPE.itemsize == 256

MAX_TREE_NODES = 64            # MCD_MAX_TREE_NODES
MAX_TREE_ROWS = 65             # MCD_MAX_TREE_ROWS
TREE_TRACE_DTYPE = np.dtype([("n_rows", "<i4"), ("row_node", "<i4", MAX_TREE_ROWS),
                             ("row_id", "<i4", MAX_TREE_ROWS), ("path_len", "<i4"), ("path", "<i4", 8),
                             ("draft_row", "<i4"), ("n_next", "<i4"), ("next_cand", "<i4", (8, 8)),
                             ("n_passes", "<i4"), ("reserved", "<i4", 17)])
assert TREE_TRACE_DTYPE.itemsize == 896


class MCDError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        super().__init__(f"{fn} failed: {STATUS_NAMES.get(status, status)}")


def library_path() -> str:
    return _LIB_PATH


def load_library() -> ctypes.CDLL:
    """Load the in-tree libmcd.so (built by __graft_entry__.build()); raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"{_LIB_PATH} is missing: build it with __graft_entry__.build()")
    lib = ctypes.CDLL(_LIB_PATH)
    P, I32, I64, U32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    sig = {
        "mcd_create": (I32, [ctypes.POINTER(McdConfig), P, ctypes.POINTER(P)]),
        "mcd_load_weights": (I32, [P, I32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(P),
                                   ctypes.POINTER(I64)]),
        "mcd_decode_frame": (I32, [P, U32, U32, P, P, P, P, P]),
        "mcd_decode_frame_host": (I32, [P, U32, U32, P, P, P, P, P]),
        "mcd_decode_frames": (I32, [P, I32, P, P, P, P, P, P, P]),
        "mcd_begin_frame": (I32, [P, U32, U32, P, P, P]),
        "mcd_verify_accept": (I32, [P, P, P, P]),
        "mcd_draft": (I32, [P, I32, I32, P, P, P, P, P]),
        "mcd_accept_from_logits": (I32, [P, I32, I32, I32, P, P, P, P, P]),
        "mcd_topk_softmax": (I32, [P, I32, P, P, P, P]),
        "mcd_topk_softmax_static": (I32, [I32, I32, I32, ctypes.c_float, P, P, P, P, P]),
        "mcd_trace_bytes": (I64, [P]),
        "mcd_set_trace": (I32, [P, P]),
        "mcd_set_timeline": (I32, [P, P]),
        "mcd_sync": (I32, [P]),
        "mcd_test_bounded_wait": (I32, [P, I32, ctypes.c_uint64, P]),
        "mcd_call_weight_bytes": (I64, [P, I32]),
        "mcd_num_ctas": (I32, [P]),
        "mcd_destroy": (None, [P]),
        "mcd_status_str": (ctypes.c_char_p, [I32]),
        "mcd_set_tree": (I32, [P, I32, P, P]),
        "mcd_outer_create": (I32, [ctypes.POINTER(McdOuterConfig), P, ctypes.POINTER(P)]),
        "mcd_outer_destroy": (None, [P]),
        "mcd_outer_load_weights": (I32, [P, I32, ctypes.POINTER(ctypes.c_char_p), ctypes.POINTER(P),
                                         ctypes.POINTER(I64)]),
        "mcd_outer_prefill": (I32, [P, U32, I32, P, P]),
        "mcd_outer_step": (I32, [P, P, I32, P]),
        "mcd_outer_frame_inputs": (I32, [P, ctypes.POINTER(P), ctypes.POINTER(P), ctypes.POINTER(P),
                                         ctypes.POINTER(U32)]),
        "mcd_pipeline_frames": (I32, [P, I32, P, P, P]),
        "mcd_outer_trace_floats": (I64, [P]),
        "mcd_outer_set_trace": (I32, [P, P, I32]),
        "mcd_outer_sync": (I32, [P]),
        "mcd_outer_step_weight_bytes": (I64, [P]),
        "mcd_tc_gemm": (I32, [I32, I32, I32, I32, P, P, P, P]),
        "mcd_tc_tile": (I32, [I32, I32, I32, P, P, P]),
        "mcd_tc_gemm_tiled": (I32, [I32, I32, I32, I32, P, P, P, P, P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _lib = lib
    return lib


def _check(fn: str, status: int):
    if status != MCD_OK:
        raise MCDError(fn, status)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("device buffers must be CUDA tensors")
    return t.data_ptr()


def _hptr(a) -> Optional[int]:
    """Host buffer address: a C-contiguous numpy array or CPU torch tensor."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags["C_CONTIGUOUS"]:
            raise ValueError("host buffers must be C-contiguous")
        return a.ctypes.data
    if a.is_cuda or not a.is_contiguous():
        raise ValueError("host buffers must be contiguous CPU tensors")
    return a.data_ptr()


def config_struct(cfg: MCDConfig) -> McdConfig:
    return McdConfig(cfg.n_layers, cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn,
                     cfg.n_pos, cfg.vocab, cfg.c0_vocab, cfg.rms_eps, cfg.rope_base, cfg.qk_norm,
                     cfg.weight_dtype, cfg.draft_len, cfg.top_k, cfg.temperature, cfg.draft_mode,
                     cfg.noise_sigma, cfg.sample_seed, cfg.max_streams)


# ---- one wrapper per entry point ------------------------------------------------------
def mcd_create(cfg: MCDConfig, stream=None) -> ctypes.c_void_p:
    lib = load_library()
    c = config_struct(cfg)
    out = ctypes.c_void_p()
    s = ctypes.c_void_p(stream.cuda_stream if stream is not None else None)
    _check("mcd_create", lib.mcd_create(ctypes.byref(c), s, ctypes.byref(out)))
    return out


def _weight_args(weights: Dict[str, np.ndarray]):
    names = list(weights)
    arrs = [np.ascontiguousarray(weights[k]) for k in names]
    n = len(names)
    c_names = (ctypes.c_char_p * n)(*[k.encode() for k in names])
    c_ptrs = (ctypes.c_void_p * n)(*[a.ctypes.data for a in arrs])
    c_sz = (ctypes.c_int64 * n)(*[a.nbytes for a in arrs])
    return n, c_names, c_ptrs, c_sz, arrs


def mcd_load_weights(ctx, weights: Dict[str, np.ndarray]):
    n, c_names, c_ptrs, c_sz, _keep = _weight_args(weights)
    _check("mcd_load_weights", load_library().mcd_load_weights(ctx, n, c_names, c_ptrs, c_sz))


def mcd_decode_frame(ctx, stream_id: int, frame_idx: int, cond, c0, c0_emb, codes_out, stats=None):
    _check("mcd_decode_frame", load_library().mcd_decode_frame(
        ctx, stream_id, frame_idx, _ptr(cond), _ptr(c0), _ptr(c0_emb), _ptr(codes_out), _ptr(stats)))


def mcd_decode_frames(ctx, stream_ids, frame_idx, cond, c0, c0_emb, codes_out, stats=None):
    """Several streams' frames in one launch; stream_ids / frame_idx are host integer lists."""
    n = len(stream_ids)
    sid = (ctypes.c_uint32 * n)(*[int(v) for v in stream_ids])
    fid = (ctypes.c_uint32 * n)(*[int(v) for v in frame_idx])
    _check("mcd_decode_frames", load_library().mcd_decode_frames(
        ctx, n, sid, fid, _ptr(cond), _ptr(c0), _ptr(c0_emb), _ptr(codes_out), _ptr(stats)))


def mcd_decode_frame_host(ctx, stream_id: int, frame_idx: int, cond, c0, c0_emb, codes_out, stats=None):
    """Host buffers (numpy arrays or CPU tensors, pinned or pageable); returns when done."""
    _check("mcd_decode_frame_host", load_library().mcd_decode_frame_host(
        ctx, stream_id, frame_idx, _hptr(cond), _hptr(c0), _hptr(c0_emb), _hptr(codes_out), _hptr(stats)))


def mcd_begin_frame(ctx, stream_id: int, frame_idx: int, cond, c0, c0_emb):
    _check("mcd_begin_frame", load_library().mcd_begin_frame(
        ctx, stream_id, frame_idx, _ptr(cond), _ptr(c0), _ptr(c0_emb)))


def mcd_verify_accept(ctx, emitted, n_emitted, logits_out=None):
    _check("mcd_verify_accept", load_library().mcd_verify_accept(
        ctx, _ptr(emitted), _ptr(n_emitted), _ptr(logits_out)))


def mcd_draft(ctx, pos_k: int, call_idx: int, h_k, draft_ids, q_ids=None, q_weights=None, z_out=None):
    _check("mcd_draft", load_library().mcd_draft(
        ctx, pos_k, call_idx, _ptr(h_k), _ptr(draft_ids), _ptr(q_ids), _ptr(q_weights), _ptr(z_out)))


def mcd_accept_from_logits(ctx, a: int, n_drafts: int, call_idx: int, p_logits, q_logits, draft_ids,
                           emitted, out2):
    _check("mcd_accept_from_logits", load_library().mcd_accept_from_logits(
        ctx, a, n_drafts, call_idx, _ptr(p_logits), _ptr(q_logits), _ptr(draft_ids), _ptr(emitted),
        _ptr(out2)))


def mcd_topk_softmax(ctx, n_rows: int, logits, ids, weights=None, sums=None):
    _check("mcd_topk_softmax", load_library().mcd_topk_softmax(ctx, n_rows, _ptr(logits), _ptr(ids),
                                                                _ptr(weights), _ptr(sums)))


def mcd_topk_softmax_static(n_rows: int, vocab: int, top_k: int, temperature: float, logits, ids,
                            weights=None, sums=None, stream=None):
    _check("mcd_topk_softmax_static", load_library().mcd_topk_softmax_static(
        n_rows, vocab, top_k, temperature, _ptr(logits), _ptr(ids), _ptr(weights), _ptr(sums),
        ctypes.c_void_p(stream.cuda_stream if stream is not None else None)))


def mcd_trace_bytes(ctx) -> int:
    return int(load_library().mcd_trace_bytes(ctx))


def mcd_set_trace(ctx, trace):
    _check("mcd_set_trace", load_library().mcd_set_trace(ctx, _ptr(trace)))


def mcd_set_timeline(ctx, timeline):
    _check("mcd_set_timeline", load_library().mcd_set_timeline(ctx, _ptr(timeline)))


def mcd_sync(ctx):
    _check("mcd_sync", load_library().mcd_sync(ctx))


def mcd_test_bounded_wait(ctx, kind: int, wait_ns: int) -> Tuple[int, int]:
    """(status, device-measured wait in ns) of one bounded wait on something nothing
    signals; MCD_ERR_TIMEOUT is the expected status."""
    waited = ctypes.c_uint64(0)
    st = int(load_library().mcd_test_bounded_wait(ctx, kind, wait_ns, ctypes.addressof(waited)))
    return st, int(waited.value)


def mcd_call_weight_bytes(ctx, n_heads: int) -> int:
    return int(load_library().mcd_call_weight_bytes(ctx, n_heads))


def mcd_num_ctas(ctx) -> int:
    return int(load_library().mcd_num_ctas(ctx))


def mcd_destroy(ctx):
    load_library().mcd_destroy(ctx)


def mcd_tc_gemm(M: int, N: int, K: int, bn: int, A, B, Y, stream=None):
    """Y[n][m] = sum_k A[m][k] B[n][k] on the tensor cores (tcgen05): A bf16 [M, K], B bf16
    [N, K], Y fp32 [N, M], all device tensors (synchronises the stream)."""
    _check("mcd_tc_gemm", load_library().mcd_tc_gemm(M, N, K, bn, _ptr(A), _ptr(B), _ptr(Y),
                                                     ctypes.c_void_p(stream.cuda_stream if stream is not None else None)))


def mcd_tc_tile(R: int, K: int, src, dst, stream=None, ld=None):
    """Re-lay device bf16 src [R][K] (row stride ld, default K) into the swizzled tile layout
    of mcd_tc_gemm_tiled in dst (device, R * K * 2 bytes); asynchronous on the stream."""
    _check("mcd_tc_tile", load_library().mcd_tc_tile(R, K, K if ld is None else ld, _ptr(src), _ptr(dst),
                                                     ctypes.c_void_p(stream.cuda_stream if stream is not None else None)))


def mcd_tc_gemm_tiled(M: int, N: int, K: int, bn: int, A_tiled, B_tiled, Y, err, stream=None):
    """Y[n][m] = sum_k A[m][k] B[n][k] from tiled operands (mcd_tc_tile); err: device int32,
    zeroed by the caller.  Asynchronous: launches the product on the stream and returns."""
    _check("mcd_tc_gemm_tiled", load_library().mcd_tc_gemm_tiled(
        M, N, K, bn, _ptr(A_tiled), _ptr(B_tiled), _ptr(Y), _ptr(err),
        ctypes.c_void_p(stream.cuda_stream if stream is not None else None)))


def mcd_status_str(status: int) -> str:
    return load_library().mcd_status_str(status).decode()


def parse_trace(buf: np.ndarray, vocab: int):
    """Split a trace buffer (uint8, mcd_trace_bytes long) into (records, verify, draft)."""
    rec_bytes = CALL_TRACE_DTYPE.itemsize * MAX_CALLS
    recs = buf[:rec_bytes].view(CALL_TRACE_DTYPE)
    logits = buf[rec_bytes:].view(np.float32)
    n = MAX_CALLS * MAX_ROWS * vocab
    return recs, logits[:n].reshape(MAX_CALLS, MAX_ROWS, vocab), logits[n:2 * n].reshape(
        MAX_CALLS, MAX_ROWS, vocab)


def mcd_set_tree(ctx, parent, rank):
    """Sparse tree of TREE mode: parent[i] (-1: child of the call's first row), rank[i]."""
    n = len(parent)
    pa = (ctypes.c_int32 * n)(*[int(v) for v in parent])
    rk = (ctypes.c_int32 * n)(*[int(v) for v in rank])
    _check("mcd_set_tree", load_library().mcd_set_tree(ctx, n, pa, rk))


def parse_tree_trace(buf: np.ndarray, vocab: int):
    """TREE mode: (tree records [16], verify logits of every row [16 calls][65 rows][vocab])."""
    start = CALL_TRACE_DTYPE.itemsize * MAX_CALLS + 2 * MAX_CALLS * MAX_ROWS * vocab * 4
    n = TREE_TRACE_DTYPE.itemsize * MAX_CALLS
    recs = buf[start:start + n].view(TREE_TRACE_DTYPE)
    nv = MAX_CALLS * MAX_TREE_ROWS * vocab
    vall = buf[start + n:start + n + nv * 4].view(np.float32).reshape(MAX_CALLS, MAX_TREE_ROWS, vocab)
    return recs, vall


class Decoder:
    """Owns one context: weights, per-frame state and the stream it runs on."""

    def __init__(self, cfg: MCDConfig, weights: Optional[Dict[str, np.ndarray]] = None, stream=None):
        import torch
        self.cfg = cfg
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.ctx = mcd_create(cfg, self.stream)
        if weights is not None:
            mcd_load_weights(self.ctx, weights)

    def close(self):
        if self.ctx:
            mcd_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ---- outer CodeDecoder and the frame pipeline (include/mcd_pipeline.h) ------------------
def outer_config_struct(cfg: OuterConfig) -> McdOuterConfig:
    return McdOuterConfig(cfg.n_layers, cfg.hidden, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.ffn,
                          cfg.c0_vocab, cfg.text_vocab, cfg.max_tokens, cfg.rms_eps, cfg.rope_base,
                          cfg.qk_norm, cfg.weight_dtype, cfg.top_k, cfg.temperature, cfg.sample_seed)


def mcd_outer_create(cfg: OuterConfig, inner_ctx) -> ctypes.c_void_p:
    c = outer_config_struct(cfg)
    out = ctypes.c_void_p()
    _check("mcd_outer_create", load_library().mcd_outer_create(ctypes.byref(c), inner_ctx, ctypes.byref(out)))
    return out


def mcd_outer_destroy(o):
    load_library().mcd_outer_destroy(o)


def mcd_outer_load_weights(o, weights: Dict[str, np.ndarray]):
    n, c_names, c_ptrs, c_sz, _keep = _weight_args(weights)
    _check("mcd_outer_load_weights", load_library().mcd_outer_load_weights(o, n, c_names, c_ptrs, c_sz))


def mcd_outer_prefill(o, stream_id: int, text_ids, c0_out=None):
    _check("mcd_outer_prefill", load_library().mcd_outer_prefill(o, stream_id, int(text_ids.numel()),
                                                                  _ptr(text_ids), _ptr(c0_out)))


def mcd_outer_step(o, prev_codes, text_id: int = -1, c0_out=None):
    _check("mcd_outer_step", load_library().mcd_outer_step(o, _ptr(prev_codes), int(text_id), _ptr(c0_out)))


def mcd_outer_frame_inputs(o):
    """Device addresses (cond, c0_emb, c0) and the frame index of the current frame."""
    cond, emb, c0 = ctypes.c_void_p(), ctypes.c_void_p(), ctypes.c_void_p()
    fi = ctypes.c_uint32()
    _check("mcd_outer_frame_inputs", load_library().mcd_outer_frame_inputs(
        o, ctypes.byref(cond), ctypes.byref(emb), ctypes.byref(c0), ctypes.byref(fi)))
    return cond.value, emb.value, c0.value, fi.value


def mcd_pipeline_frames(o, n_frames: int, codes_out, text_ids=None, stats=None):
    tid = None
    if text_ids is not None:
        tid = (ctypes.c_int32 * n_frames)(*[int(v) for v in text_ids])
    _check("mcd_pipeline_frames", load_library().mcd_pipeline_frames(o, n_frames, tid, _ptr(codes_out),
                                                                      _ptr(stats)))


def mcd_outer_trace_floats(o) -> int:
    return int(load_library().mcd_outer_trace_floats(o))


def mcd_outer_set_trace(o, trace, n_frames: int):
    _check("mcd_outer_set_trace", load_library().mcd_outer_set_trace(o, _ptr(trace), n_frames))


def mcd_outer_sync(o):
    _check("mcd_outer_sync", load_library().mcd_outer_sync(o))


def mcd_outer_step_weight_bytes(o) -> int:
    return int(load_library().mcd_outer_step_weight_bytes(o))


class Pipeline:
    """An inner Decoder plus the outer CodeDecoder on top of it (one utterance at a time)."""

    def __init__(self, outer_cfg: OuterConfig, inner_cfg: MCDConfig,
                 outer_weights: Optional[Dict[str, np.ndarray]] = None,
                 inner_weights: Optional[Dict[str, np.ndarray]] = None, stream=None):
        self.inner = Decoder(inner_cfg, inner_weights, stream)
        self.cfg = outer_cfg
        self.o = mcd_outer_create(outer_cfg, self.inner.ctx)
        if outer_weights is not None:
            mcd_outer_load_weights(self.o, outer_weights)

    def close(self):
        if self.o:
            mcd_outer_destroy(self.o)
            self.o = None
        self.inner.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
