/* libmcd: the outer CodeDecoder and the full frame pipeline (arXiv 2609.37007).
 *
 * The paper's generation loop (Sec. 1 and Fig. 1 with its caption): per 80 ms frame a
 * 28-layer CodeDecoder is called once and emits the seed code c0; the MultiCodeDecoder
 * then emits c1..c15 (mcd.h); the next frame's CodeDecoder input is the sum of the text
 * token's embedding and the embeddings of the 16 codes of the frame before.
 *
 * Readings of what the paper leaves open, shared with the CPU oracle:
 *   - the CodeDecoder block is the MultiCodeDecoder's block (mcd.h), positions are absolute
 *     over the utterance: the text prompt fills positions 0..T-1, frame f >= 1 adds one row
 *     at position T - 1 + f;
 *   - frame 0's c0 and MultiCodeDecoder input come from the last prompt row;
 *   - the input row of frame f >= 1 is t_f + E_c0(c0) + E_1(c1) + ... + E_P(c_P) of frame
 *     f - 1 (fp32 sum in that order), E_1..E_{P-1} being the MultiCodeDecoder's own code
 *     tables and E_P the outer model's `code_embed.P`; t_f is zero unless a text id is given;
 *   - the KV cache holds K (after QK-norm and RoPE) and V in the weight dtype (bf16 values
 *     rounded to nearest even), and every read of a position sees the stored value;
 *   - c0 ~ top-k / temperature of the c0 logits W_c0 h, drawn with the 53-bit uniform of the
 *     Philox counter (stream, frame, round 0, position 0, purpose 0) under `seed`
 *     (position 0 is never used by a MultiCodeDecoder decision);
 *   - the MultiCodeDecoder receives cond = h (fp32, the CodeDecoder's post-final-norm
 *     hidden state) and the c0 embedding E_c0(c0) as an fp32 vector: its context must have
 *     c0_vocab = 0.
 *
 * Conventions are those of mcd.h: every call returns a status, device pointers must be
 * valid on the inner context's stream, calls are asynchronous on that stream, a failed
 * device-side check is reported by mcd_outer_sync.
 */
#ifndef MCD_PIPELINE_H
#define MCD_PIPELINE_H

#include "mcd.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct mcd_outer mcd_outer;

typedef struct {
  int32_t n_layers;      /* 28 for the CodeDecoder */
  int32_t hidden;        /* must equal the inner model's hidden size */
  int32_t n_q_heads;
  int32_t n_kv_heads;    /* n_q_heads / n_kv_heads <= 8 */
  int32_t head_dim;      /* 64 or 128 */
  int32_t ffn;
  int32_t c0_vocab;      /* rows of the c0 table and of the c0 head: 16..4096, a multiple of 16 */
  int32_t text_vocab;    /* rows of the text-token table */
  int32_t max_tokens;    /* KV capacity = prompt tokens + frames - 1, at most 1024 */
  float rms_eps;
  float rope_base;
  int32_t qk_norm;
  int32_t weight_dtype;  /* MCD_WEIGHT_F32 / MCD_WEIGHT_BF16, equal to the inner model's */
  int32_t top_k;         /* c0 sampling: top-k (<= 128) */
  float temperature;
  uint64_t seed;         /* Philox key of the c0 draws */
} mcd_outer_config;

/* Create the outer model on top of an inner (MultiCodeDecoder) context.  The outer
 * context uses the inner context's stream and device, reads its code tables 1..P-1 in the
 * frame sum, and must be destroyed before it.  Errors: MCD_ERR_INVALID_ARG (null pointer,
 * dtype differing from the inner model's, inner context with a c0 table),
 * MCD_ERR_UNSUPPORTED (shape outside the kernels' limits), MCD_ERR_OOM, MCD_ERR_CUDA. */
mcd_status mcd_outer_create(const mcd_outer_config* cfg, mcd_ctx* inner, mcd_outer** out);
void mcd_outer_destroy(mcd_outer* o);

/* Copy the outer weights from host memory (the caller keeps ownership; row-major [out, in]
 * matrices in the weight dtype: bf16 as uint16 bit patterns).  Names: for each layer l
 * "layers.l.{attn_norm,wq,wk,wv,q_norm,k_norm,wo,ffn_norm,wg,wu,wd}" as in mcd.h (q_norm /
 * k_norm only with qk_norm), "final_norm" [H], "c0_head" [c0_vocab, H], "c0_embed"
 * [c0_vocab, H], "text_embed" [text_vocab, H] and "code_embed.P" [inner vocab, H] (P = the
 * inner model's n_pos).  Synchronous.  MCD_ERR_WEIGHTS if a tensor is missing, repeated or
 * of the wrong size (nothing is copied then). */
mcd_status mcd_outer_load_weights(mcd_outer* o, int32_t n, const char* const* names, const void* const* host_ptrs,
                                  const int64_t* nbytes);

/* Start an utterance of stream `stream_id`: reset the KV cache and run the prompt rows
 * text_ids[0..n_tokens) (device int32) at positions 0..n_tokens-1 (bf16 shapes that the
 * tensor-core block products take: all rows but the last as one batch; otherwise up to 16
 * rows per launch); the last row gives frame 0's c0 and inner inputs (c0_out, device int32,
 * optional, also receives c0).  Errors: MCD_ERR_INVALID_ARG, MCD_ERR_STATE (weights not
 * loaded), MCD_ERR_UNSUPPORTED (n_tokens > max_tokens); an id outside the text table is
 * reported by mcd_outer_sync as MCD_ERR_INVALID_ARG. */
mcd_status mcd_outer_prefill(mcd_outer* o, uint32_t stream_id, int32_t n_tokens, const int32_t* text_ids,
                             int32_t* c0_out);

/* One CodeDecoder row for the next frame: input = the sum above over prev_codes (device
 * int32 [n_pos + 1]: c0..c_P of the previous frame) and text row text_id (-1: none).
 * Produces the frame's c0 and inner inputs (mcd_outer_frame_inputs); c0_out (device
 * int32, optional) also receives c0.  MCD_ERR_STATE before a prefill or when the KV cache
 * is full. */
mcd_status mcd_outer_step(mcd_outer* o, const int32_t* prev_codes, int32_t text_id, int32_t* c0_out);

/* Device pointers to the current frame's inner inputs (cond [H] fp32, c0 embedding [H]
 * fp32, c0 [1] int32) and its frame index; valid until the next prefill / step. */
mcd_status mcd_outer_frame_inputs(const mcd_outer* o, const float** cond, const float** c0_emb, const int32_t** c0,
                                  uint32_t* frame_idx);

/* Decode n_frames frames of the utterance: for each, the CodeDecoder row (except for a
 * frame whose c0 the prefill or a step already produced), then the inner model's frame
 * (mcd_decode_frame with the frame index as its Philox frame).  codes_out: device int32
 * [n_frames][n_pos + 1], row f = c0, c1..c_P of the f-th frame decoded; text_ids: host
 * int32 [n_frames] text row per frame or NULL (none); stats: device mcd_frame_stats
 * [n_frames] of the inner frames, or NULL.  No host synchronisation.  MCD_ERR_STATE before
 * a prefill, or once the KV cache is full. */
mcd_status mcd_pipeline_frames(mcd_outer* o, int32_t n_frames, const int32_t* text_ids, int32_t* codes_out,
                               mcd_frame_stats* stats);

/* Optional per-frame record for parity checks: trace (device fp32, n_frames records of
 * mcd_outer_trace_floats floats each) receives, for frame f < n_frames, the c0 logits
 * [c0_vocab], cond [H] and the c0 embedding [H].  NULL / 0 turns it off. */
int64_t mcd_outer_trace_floats(const mcd_outer* o);
mcd_status mcd_outer_set_trace(mcd_outer* o, float* trace, int32_t n_frames);

/* Wait for the stream; returns the first device-side error of the outer launches. */
mcd_status mcd_outer_sync(mcd_outer* o);

/* Weight bytes one CodeDecoder row streams: the backbone plus the c0 head. */
int64_t mcd_outer_step_weight_bytes(const mcd_outer* o);

#ifdef __cplusplus
}
#endif

#endif /* MCD_PIPELINE_H */
