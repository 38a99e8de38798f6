/*
 * mcd.h -- C ABI of the GB300 MultiCodeDecoder speculative-decoding library (libmcd.so).
 *
 * Operation (arXiv 2609.37007): per 80 ms audio frame the MultiCodeDecoder (MCD) emits
 * the 15 residual RVQ codes c1..c15 after the outer model's c0 (Sec. 1, Fig. 1).  This
 * library runs that inner loop with RVQ-position-aware speculative decoding
 * (Sec. 2.2, Fig. 3): each model call feeds the last emitted code plus K drafted codes,
 * verifies the drafts with the lossless acceptance rule min(1, p/q) with residual
 * resampling under the deployed top-k / temperature sampling (Abstract, Sec. 3.2), and
 * drafts the next K codes from LM head k+j applied to h_k + b_j, where h_k is the
 * hidden state that emitted the last code and b_1..b_K are the per-lookahead offsets.
 *
 * Conventions
 *   - Every call returns an mcd_status; nothing aborts or throws across the ABI.
 *   - "dev" pointers are CUDA device pointers owned by the caller, valid until the work
 *     queued on the context's stream has finished.  "host" pointers are read before the
 *     call returns.  The context owns its weights, KV cache, scratch and counters.
 *   - Calls that launch work are asynchronous on the stream given to mcd_create unless
 *     stated otherwise.  Device-side failures (a bounded wait that ran out) are recorded
 *     in the context and reported by mcd_sync() and by the `status` field of
 *     mcd_frame_stats.
 *   - There is no CPU fallback: without a usable CUDA device mcd_create fails.
 *   - A context is not thread-safe; use one context per host thread.
 *
 * Random numbers: Philox4x32-10 (Salmon et al., SC'11) with key = (seed lo, seed hi) and
 * counter = (stream id, frame index, (call index << 8) | position, purpose); purpose
 * 0 = target / residual / bonus sample, 1 = accept test, 2 = draft sample,
 * 3 + v/2 = Gaussian pair for vocabulary entries (v, v+1) of a noisy draft row.
 * A decision uses U = (w0 >> 5) * 2^26 + (w1 >> 6) from words 0 and 1 (u = U / 2^53).
 *
 * Distributions: the top-k set of a logits row (ranked by fp32 logit desc, then id asc,
 * and listed in ascending id order, the order draws walk) with integer weights
 * W_i = floor(2^24 * exp32(z_i - z_max)), z = fp32 logit / fp32 T, where
 * exp32 is an fp32 exponential (Cody-Waite range reduction, degree-7 Taylor polynomial);
 * p(x) = W_x / S, S = sum W.  Draws, accept tests (u < p(d)/q(d)) and residual draws
 * (normalised max(0, p - q)) are exact integer comparisons.
 */
#ifndef MCD_H
#define MCD_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct mcd_ctx mcd_ctx;

typedef enum {
  MCD_OK = 0,
  MCD_ERR_INVALID_ARG = 1,   /* bad pointer, size or configuration value               */
  MCD_ERR_STATE = 2,         /* call out of order (e.g. decode before weights)         */
  MCD_ERR_CUDA = 3,          /* a CUDA runtime call failed; context must be destroyed  */
  MCD_ERR_OOM = 4,           /* device allocation failed                               */
  MCD_ERR_TIMEOUT = 5,       /* a bounded device-side wait ran out                     */
  MCD_ERR_WEIGHTS = 6,       /* missing, duplicate or wrongly sized weight tensor      */
  MCD_ERR_UNSUPPORTED = 7    /* shape outside the kernels' limits                      */
} mcd_status;

/* MCD_WEIGHT_INT8 (W8A16, Sec. 3.3): weights are passed in bf16 like MCD_WEIGHT_BF16 and
 * the library quantises every streamed matrix (Wq, Wk, Wv, Wo, Wg, Wu, Wd, LM heads) per
 * output row at load: s = fp32(max |w| / 127), q = clamp(rint(fp32(w / s)), -127, 127),
 * computing with q * s; embedding tables stay bf16.  Single-stream and up to 32 packed rows. */
enum { MCD_WEIGHT_F32 = 0, MCD_WEIGHT_BF16 = 1, MCD_WEIGHT_INT8 = 2 };
enum { MCD_DRAFT_SAMPLE = 0, MCD_DRAFT_GREEDY = 1, MCD_DRAFT_NOISY_TARGET = 2, MCD_DRAFT_TREE = 3 };

/* Model and sampling configuration.  Limits: hidden, ffn multiples of 128; head_dim 64
 * or 128; n_q_heads multiple of n_kv_heads; vocab multiple of 16 and <= 4096;
 * n_pos <= 15; draft_len (K) <= 7; top_k in 1..128 and <= vocab; c0_vocab <= 4096. */
typedef struct {
  int32_t n_layers, hidden, n_q_heads, n_kv_heads, head_dim, ffn;
  int32_t n_pos;        /* residual positions c1..c_{n_pos} (15 in the paper)           */
  int32_t vocab;        /* codebook size of c1..c_{n_pos}                               */
  int32_t c0_vocab;     /* rows of table 0; 0 = frames pass a c0 embedding vector       */
  float rms_eps, rope_base;
  int32_t qk_norm;      /* per-head RMSNorm of q and k before RoPE                      */
  int32_t weight_dtype; /* MCD_WEIGHT_F32, MCD_WEIGHT_BF16 or MCD_WEIGHT_INT8             */
  int32_t draft_len;    /* K; 0 = plain autoregressive decoding                         */
  int32_t top_k;
  float temperature;
  int32_t draft_mode;   /* MCD_DRAFT_*: SAMPLE = position-aware offset drafter (Sec. 2.2),
                         * GREEDY = its argmax, NOISY_TARGET = controlled-acceptance drafts:
                         * q for position s is the target's own fp32 logits of s given the
                         * drafted prefix (one extra one-row pass per draft, run inside the
                         * same frame launch) plus noise_sigma * N(0,1) per entry,
                         * TREE = sparse tree of top-m candidates per drafted position
                         * (mcd_set_tree; Sec. 2.2 and Fig. 2), verified in one call       */
  float noise_sigma;    /* MCD_DRAFT_NOISY_TARGET only (>= 0)                            */
  uint64_t seed;        /* Philox key                                                    */
  int32_t max_streams;  /* streams one mcd_decode_frames call may decode together (1..128).
                         * Up to 8 streams and 32 packed rows (streams x max(K + 1, 2)) a
                         * frame is one persistent-kernel launch; beyond that calls run on
                         * the batched GEMM path (bf16 weights, <= 512 packed rows, one
                         * CUDA graph launch per frame), which also takes launches of 5 or
                         * more streams when the shapes allow its tensor-core products
                         * (bf16; q / kv / ffn widths multiples of 128).  NOISY_TARGET and
                         * TREE need 1                                                     */
} mcd_config;

/* Per-frame counters written by the device (device memory, caller-owned). */
typedef struct {
  int32_t calls;     /* model calls (rounds) spent on the frame                */
  int32_t codes;     /* codes emitted (n_pos on success)                        */
  int32_t drafted;   /* drafts tested                                           */
  int32_t accepted;  /* drafts kept                                             */
  int32_t status;    /* 0, or an mcd_status value set by a failed device wait   */
  int32_t heads_read;/* LM heads streamed, summed over the calls (byte accounting) */
  int32_t kv_rows;   /* sum over calls of (first row position + rows): KV touched   */
  int32_t rows_fed;  /* sum over calls of rows fed                                  */
} mcd_frame_stats;

/* Per-call record written when tracing is on (mcd_set_trace).  One record per verify
 * call, in call order; logits of record r live in the trace buffer after all records (see
 * mcd_trace_bytes for the layout).  With NOISY_TARGET drafts the draft rows of record r are
 * the noisy rows its drafts were drawn from. */
typedef struct {
  int32_t a;              /* codes emitted before this call                           */
  int32_t n_rows;         /* rows fed                                                 */
  int32_t pos0;           /* sequence position of the first row                       */
  int32_t n_drafts;       /* drafts tested                                            */
  int32_t input_ids[8];   /* code fed at each row (-1: conditioning / c0 vector)      */
  int32_t drafts[8];      /* drafts tested (positions a+1..)                          */
  int32_t n_acc;          /* drafts kept                                              */
  int32_t n_emit;         /* codes emitted                                            */
  int32_t emitted[8];
  int32_t n_next;         /* drafts made for the next call                            */
  int32_t next_drafts[8];
  int32_t draft_row;      /* row whose hidden state drafted them (= n_acc)            */
  int32_t reserved[24];
} mcd_call_trace;

/* Create a context on the current CUDA device for one MultiCodeDecoder (the 5-layer
 * inner model of Sec. 1 and Fig. 1 that emits c1..c15 after c0, with one embedding table
 * and one LM head per residual position, Sec. 2.1) and its sampling configuration.
 * `cfg` (host) is copied.  `cuda_stream` is a cudaStream_t (NULL = legacy default stream)
 * used by every later call.  Allocates device buffers and sets kernel attributes.  On
 * failure *out is NULL. */
mcd_status mcd_create(const mcd_config* cfg, void* cuda_stream, mcd_ctx** out);

/* Load all weights of the model of Sec. 1 / Fig. 1 (the backbone, the per-position tables
 * and LM heads of Sec. 2.1, and the offsets b_1..b_K of Sec. 2.2 "RVQ position aware
 * offsets", Fig. 3).  `names`, `host_ptrs`, `nbytes`: n host arrays describing named
 * tensors in the dtype of cfg.weight_dtype (bf16 as raw 16-bit patterns), row-major,
 * matrices [out, in].  Required names (l = layer, i = table, P = position, j = offset):
 *   layers.l.{attn_norm[H], wq[Hq*D,H], wk[Hkv*D,H], wv[Hkv*D,H], q_norm[D], k_norm[D]
 *            (qk_norm only), wo[H,Hq*D], ffn_norm[H], wg[F,H], wu[F,H], wd[H,F]},
 *   final_norm[H], embed.0[c0_vocab,H] (c0_vocab > 0), embed.i[V,H] (i = 1..n_pos-1),
 *   head.P[V,H] (P = 1..n_pos), offset.j[H] (j = 1..max(K,1)).
 * The library copies and re-tiles them (the caller keeps ownership) and synchronises
 * the stream before returning.  Extra names are ignored. */
mcd_status mcd_load_weights(mcd_ctx* ctx, int32_t n, const char* const* names,
                            const void* const* host_ptrs, const int64_t* nbytes);

/* Decode one frame: emit c1..c_{n_pos} into codes_out (dev int32 [n_pos]) -- the per-frame
 * inner loop of Sec. 1 / Fig. 1, run with the draft-and-verify calls of Sec. 2.2 / Fig. 3
 * until every residual code of the frame is emitted.
 *   cond   dev float [hidden], 16-byte aligned: the outer model's hidden state
 *          (sequence position 0).
 *   c0     dev int32 [1]: the frame's c0 id (c0_vocab > 0), else NULL; an id outside
 *          [0, c0_vocab) fails the frame with MCD_ERR_INVALID_ARG (reported by mcd_sync).
 *   c0_emb dev float [hidden], 16-byte aligned: c0 embedding (c0_vocab == 0), else NULL.
 *   stats  dev mcd_frame_stats, optional (NULL).
 * One cooperative persistent-kernel launch runs every call of the frame on device. */
mcd_status mcd_decode_frame(mcd_ctx* ctx, uint32_t stream_id, uint32_t frame_idx,
                            const float* cond, const int32_t* c0, const float* c0_emb,
                            int32_t* codes_out, mcd_frame_stats* stats);

/* Batched streams: decode one frame for each of n_streams (1..max_streams) independent
 * streams in one launch.  The streams advance in lock step, one call at a time; every
 * call packs the rows of every stream whose frame is not complete into one operand
 * (re-packed each call, since streams accept different numbers of drafts), streams the
 * backbone once and the union of the LM heads the streams need, and runs each stream's
 * acceptance on its own CTA.  Stream s uses the Philox counters of (stream_ids[s],
 * frame_idx[s]) and its own KV cache, so its codes are those a single-stream
 * mcd_decode_frame would emit from the same logits.
 *   stream_ids, frame_idx  host uint32 [n_streams]
 *   cond      dev float [n_streams, hidden] (16-byte aligned rows)
 *   c0        dev int32 [n_streams] (c0_vocab > 0) or c0_emb dev float [n_streams, hidden]
 *   codes_out dev int32 [n_streams, n_pos]; stats dev mcd_frame_stats [n_streams], optional.
 * Tracing (mcd_set_trace) records every stream: stream s's block starts at byte
 * s * mcd_trace_bytes() / max_streams. */
mcd_status mcd_decode_frames(mcd_ctx* ctx, int32_t n_streams, const uint32_t* stream_ids,
                             const uint32_t* frame_idx, const float* cond, const int32_t* c0,
                             const float* c0_emb, int32_t* codes_out, mcd_frame_stats* stats);

/* mcd_decode_frame on host buffers: cond (host float [hidden]), c0 (host int32 [1]) or
 * c0_emb (host float [hidden]) are gathered into the context's pinned host mirror and
 * copied to its device staging area in one transfer, the frame is decoded, and codes,
 * stats and the device error word come back in one transfer; the call waits for the
 * stream once, then fills codes_out (host int32 [n_pos]) and stats (host, optional).
 * Bytes moved per frame: hidden*4 + 16 in (hidden*8 + 16 with c0_emb), 112 out.
 * Any host memory works, pinned or pageable.  Returns the first device-side failure like
 * mcd_sync (clearing it); codes_out and stats are then left unwritten.  The per-frame
 * entry point of a host-driven TTS loop. */
mcd_status mcd_decode_frame_host(mcd_ctx* ctx, uint32_t stream_id, uint32_t frame_idx,
                                 const float* cond, const int32_t* c0, const float* c0_emb,
                                 int32_t* codes_out, mcd_frame_stats* stats);

/* Stepwise use of the same kernels: one verify call of Sec. 2.2 / Fig. 3 at a time
 * (LMH_k reads h_k and emits the verified code, LMH_{k+j} reads h_k + b_j and drafts;
 * acceptance min(1, p/q) with residual resampling, Sec. 3.2).  mcd_begin_frame resets the
 * per-frame state (Sec. 1: every frame starts at c1 after c0) and
 * selects the (stream id, frame index) of the Philox counters; it needs no weights, so
 * the sampler hooks below can run on a context without them;
 * mcd_verify_accept runs exactly one verify call (the first call feeds cond and c0) and,
 * with NOISY_TARGET drafts, the one-row passes that draft for the next call,
 * writing the codes it emitted to emitted (dev int32 [K+1]) and their count to
 * n_emitted (dev int32 [1]); a call after the frame is complete emits 0 codes.
 * logits_out (dev float [K+1, vocab], optional) receives the verify logits of the
 * call's rows that read an LM head. */
mcd_status mcd_begin_frame(mcd_ctx* ctx, uint32_t stream_id, uint32_t frame_idx,
                           const float* cond, const int32_t* c0, const float* c0_emb);
mcd_status mcd_verify_accept(mcd_ctx* ctx, int32_t* emitted, int32_t* n_emitted,
                             float* logits_out);

/* Position-aware drafting on its own (Sec. 2.2, Fig. 3): for j = 1..min(K, n_pos-k)
 * z_j = LMH_{k+j}(h_k + b_j); q_j = top-k/temperature softmax of z_j; d_j ~ q_j with the
 * draft-purpose uniform of (call_idx, k+j) under the frame set by mcd_begin_frame.
 *   h_k      dev float [hidden], the post-norm hidden state read by LM head k (1 <= k < n_pos)
 *   draft_ids dev int32 [K]; q_ids dev int32 [K, top_k] and q_weights dev uint32
 *   [K, top_k] (optional): the draft distributions; z_out dev float [K, vocab], optional.
 *   Unused rows are left untouched. */
mcd_status mcd_draft(mcd_ctx* ctx, int32_t pos_k, int32_t call_idx, const float* h_k,
                     int32_t* draft_ids, int32_t* q_ids, uint32_t* q_weights, float* z_out);

/* Sampler on given fp32 logits: the acceptance rule of Sec. 2.2 and Sec. 3.2 (accept d
 * with probability min(1, p(d)/q(d)), else resample from normalised max(0, p - q); the
 * bonus code from p when every draft is kept), as a parity hook.  p_logits dev
 * float [n_drafts+1, vocab] are the verify rows of positions a+1..a+1+n_drafts (the last
 * row is only read when a bonus position exists), q_logits dev float [n_drafts, vocab]
 * the draft rows, draft_ids dev int32 [n_drafts].  Uniforms use (call_idx, position)
 * under the frame set by mcd_begin_frame.  Writes emitted (dev int32 [n_drafts+1]) and
 * out2 (dev int32 [2]) = {n_acc, n_emit}.  Uses cfg.top_k, temperature, draft_mode
 * (SAMPLE or GREEDY). */
mcd_status mcd_accept_from_logits(mcd_ctx* ctx, int32_t a, int32_t n_drafts, int32_t call_idx,
                                  const float* p_logits, const float* q_logits,
                                  const int32_t* draft_ids, int32_t* emitted, int32_t* out2);

/* Top-k / temperature distributions (Abstract and Sec. 3.1: the deployed top-k sampling)
 * of n_rows fp32 logits rows (dev float [n_rows, vocab], n_rows <= 128): ids (dev int32
 * [n_rows, top_k]) in ascending id order (the sampling order), weights (dev uint32
 * [n_rows, top_k]) and sums (dev uint64 [n_rows]); any output may be NULL.  With
 * draft_mode GREEDY the rows are still full top-k distributions (greedy applies to
 * drafts only). */
mcd_status mcd_topk_softmax(mcd_ctx* ctx, int32_t n_rows, const float* logits,
                            int32_t* ids, uint32_t* weights, uint64_t* sums);

/* No-allocation variant of mcd_topk_softmax (the paper has no counterpart: it is a
 * deployment convenience).  Some callers cannot allocate device memory when they need a
 * distribution: a host that hands all device memory to its own pool up front, or a
 * real-time audio thread that must not enter the CUDA allocator, which can block on
 * locks shared with other threads.  This call needs no mcd_ctx (creating one allocates)
 * and allocates nothing: its per-row scratch is a fixed array of
 * MCD_STATIC_TOPK_MAX_ROWS records in the library's own device memory, so it takes at
 * most that many rows per call.
 *   logits   dev float [n_rows, vocab], 16-byte aligned; vocab a multiple of 16, <= 4096
 *   ids      dev int32 [n_rows, top_k], ascending id order; weights dev uint32
 *            [n_rows, top_k]; sums dev uint64 [n_rows]; any output may be NULL
 *   top_k in 1..min(128, vocab); temperature > 0; cuda_stream a cudaStream_t (NULL = legacy
 *   default stream).  Results are the ones mcd_topk_softmax gives for the same rows.
 * Errors: MCD_ERR_INVALID_ARG for a bad pointer, alignment, vocab (< 16 or not a multiple
 * of 16), top_k < 1 or top_k > vocab, or temperature; MCD_ERR_UNSUPPORTED for
 * n_rows > MCD_STATIC_TOPK_MAX_ROWS (nothing is launched), top_k > 128 or vocab > 4096
 * (the limits mcd_create reports the same way); MCD_ERR_CUDA if the set-up or the launch
 * fails.
 * The first call on each device (made with that device current) does a one-time set-up
 * that looks up the scratch's device address; make it before any stream capture begins.
 * Later calls take no lock.  After cudaDeviceReset the cached address is stale: do not
 * call this entry point on that device again in the same process.
 * Nothing in the scratch needs to start at zero.  The scratch is shared by every call on
 * a device: calls whose work can overlap (other streams, other host threads) race on it,
 * so serialise them, e.g. on one stream. */
#define MCD_STATIC_TOPK_MAX_ROWS 128
mcd_status mcd_topk_softmax_static(int32_t n_rows, int32_t vocab, int32_t top_k, float temperature,
                                   const float* logits, int32_t* ids, uint32_t* weights,
                                   uint64_t* sums, void* cuda_stream);

/* Tracing for parity tests: while `trace` (dev, mcd_trace_bytes() bytes) is set, frame
 * decoding writes one mcd_call_trace per call followed, after 16 records, by float
 * logits [16 calls][8 rows][vocab] (verify rows) and [16 calls][8 drafts][vocab] (the
 * draft rows used).  In TREE mode the block continues with 16 mcd_tree_trace records and
 * the verify logits of every row, [16 calls][MCD_MAX_TREE_ROWS rows][vocab].  NULL turns tracing off. */
int64_t mcd_trace_bytes(const mcd_ctx* ctx);
mcd_status mcd_set_trace(mcd_ctx* ctx, void* trace);

/* Per-call record of TREE mode (after the mcd_call_trace records; see mcd_set_trace). */
#define MCD_MAX_TREE_NODES 64
#define MCD_MAX_TREE_ROWS 65   /* rows of one tree call: the last emitted code + the nodes */
typedef struct {
  int32_t n_rows;         /* rows fed: row 0 = the last emitted code, then tree nodes     */
  int32_t row_node[MCD_MAX_TREE_ROWS];  /* tree node of each row (-1: row 0)              */
  int32_t row_id[MCD_MAX_TREE_ROWS];    /* code fed at each row                           */
  int32_t path_len;       /* nodes kept                                                   */
  int32_t path[8];        /* kept nodes, root first                                       */
  int32_t draft_row;      /* row whose draft logits gave the next call's candidates       */
  int32_t n_next;         /* candidate depths of the next call                            */
  int32_t next_cand[8][8];/* [depth - 1][rank] candidate ids of the next call             */
  int32_t n_passes;       /* weight passes of the call: ceil(n_rows / 32)                 */
  int32_t reserved[17];
} mcd_tree_trace;

/* Sparse tree of TREE mode (Sec. 2.2 "Tree attention ...", Fig. 2; sizes N = 16..64 as in
 * the tree sweep of Sec. 3.4, Fig. 4): n_nodes <= 64 (MCD_MAX_TREE_NODES) nodes
 * in breadth-first order (host arrays); node i has parent[i] (-1: a child of the call's
 * first row, else an earlier node) and rank[i] < 8 (distinct among siblings), depth =
 * parent's depth + 1 <= draft_len.  A node of depth d proposes the id of rank rank[i] in
 * the draft logits of depth d (fp32 logit descending, id ascending) of the row whose LM
 * head emitted the call's last code; rows attend to the committed prefix, the call's
 * first row, their ancestors and themselves.  Verification walks from the first row: the
 * children of a node are tested in rank order, test i keeping its candidate x with
 * probability p'(x), p' being the node's distribution without the candidates already
 * rejected there (uniform of counter (call, code position, purpose 1 for i = 0, else
 * 0x10000 + i)); when none is kept, or the node has no children, a code is drawn from p'
 * with purpose 0.  The kept nodes' keys and values become the committed cache.  A call
 * of more than 32 rows runs as passes of up to 32 rows through the whole model (rows
 * 32 t .. 32 t + 31 in pass t; later rows attend to earlier ones through the cache); the
 * acceptance step follows the last pass.  Until
 * set, the tree is the chain of draft_len rank-0 nodes.  Errors: MCD_ERR_INVALID_ARG
 * (malformed tree), MCD_ERR_STATE (context not in TREE mode). */
mcd_status mcd_set_tree(mcd_ctx* ctx, int32_t n_nodes, const int32_t* parent, const int32_t* rank);

/* Profiling hook: while `timeline` (dev, uint64 [16 calls][128], zeroed by the caller)
 * is set, frame decoding writes %globaltimer stamps (ns) per call: slot 0 call start;
 * 1 top-k inputs ready; 2 / 3 top-k done by CTA 0 / by the last CTA; 4..7 acceptance
 * start, records staged, decided, end.  Stage s (s = 4l + k for step k of layer l:
 * 0 QKV, 1 attention + Wo, 2 gate/up, 3 down; s = 4L heads) uses slots 8+4s..: +0 inputs
 * ready and +1 first weight unit in shared memory (CTA 0), +2 last epilogue done and +3
 * completion signalled (maximum over CTAs).  NULL turns it off. */
mcd_status mcd_set_timeline(mcd_ctx* ctx, uint64_t* timeline);

/* Wait for the context's stream; returns the first device-side failure, if any. */
mcd_status mcd_sync(mcd_ctx* ctx);

/* Failure-detection hook: runs, in a one-CTA kernel on the context's stream, the bounded
 * wait that every kernel of the library uses on something nothing will ever signal, and
 * reports the outcome.  kind 0 waits on a device counter that is never incremented (the
 * grid-level arrival counters' wait); kind 1 waits on a shared-memory mbarrier that never
 * completes (the weight ring's wait).  The wait gives up after wait_ns (1 us .. 10 s),
 * records MCD_ERR_TIMEOUT in the context like any device-side timeout, and the call waits
 * for the stream and returns that status (clearing it, like mcd_sync), so MCD_ERR_TIMEOUT
 * is the expected result; the context stays usable.  waited_ns (host, optional) receives
 * the device-measured (%globaltimer) duration of the wait.  Errors: MCD_ERR_INVALID_ARG
 * (kind or wait_ns out of range), MCD_ERR_STATE (a device-side failure was pending). */
mcd_status mcd_test_bounded_wait(mcd_ctx* ctx, int32_t kind, uint64_t wait_ns, uint64_t* waited_ns);

/* Bytes of weights one verify call streams for a call that reads `n_heads` LM heads
 * (backbone + heads), the algorithmic traffic used for roofline accounting. */
int64_t mcd_call_weight_bytes(const mcd_ctx* ctx, int32_t n_heads);

/* Number of persistent CTAs (one per SM) the frame kernel launches. */
int32_t mcd_num_ctas(const mcd_ctx* ctx);

void mcd_destroy(mcd_ctx* ctx);
const char* mcd_status_str(mcd_status s);

#ifdef __cplusplus
}
#endif
#endif /* MCD_H */
