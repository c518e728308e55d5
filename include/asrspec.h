/*
 * asrspec.h - C ABI of the GB300 (sm_103a) draft-verify step for single-model
 * speculative ASR decoding ("Alignment Drift in Single-Model Speculative
 * Decoding for ASR: Mechanism, Correction, and Cost").
 *
 * The step (Sec. 3, "Speculative Loop"): a draft proposes up to K tokens per
 * utterance; the frozen target scores the pending token and the K drafts in
 * one decoder pass, accepts the longest prefix that matches its own greedy
 * output and adds its next prediction (the "bonus" token, so a round advances
 * 1 + L tokens, App. "Correction and Cost", cost derivation).  Accepted tokens
 * and their cached states feed the next round (App. "Decoding and
 * Intervention Protocol", real cached loop).  The runtime correction re-anchors
 * the next draft round at the peak of the target's head-averaged audio
 * attention at one decoder layer, recomputed from the existing key cache
 * without another target pass (Sec. 5 "Verification-Attention Correction",
 * App. "Runtime anchor construction").
 *
 * Model: a Whisper-style pre-LN decoder (Sec. 3 "Models and Protocol"):
 * learned positional table, per layer LN -> causal self-attention (biases on
 * q, v and the output; none on k) -> LN -> cross-attention to the encoder
 * states -> LN -> MLP (erf GELU), final LN, LM head tied to the token
 * embedding.  Head dimension 64.  LayerNorm eps 1e-5.
 *
 * Conventions
 *  - All calls are asynchronous on the handle's CUDA stream unless host I/O
 *    is enabled (asr_spec_set_host_io), in which case every call that takes
 *    or returns arrays synchronises before it returns.
 *  - Array arguments are device pointers by default; with host I/O enabled
 *    they are host pointers (pinned or pageable) and the library copies them.
 *  - The handle owns every device buffer it allocates (weights, caches,
 *    activations).  The caller owns every argument buffer.
 *  - Return value: ASR_OK (0) or a negative ASR_E_* code; the message is in
 *    asr_spec_last_error.  Conditions that depend on device data (a token id
 *    out of range, lens out of range, context capacity) are found by the
 *    kernels, which then skip the step without changing any state and set the
 *    device status word, read by asr_spec_status.  No kernel traps.
 *  - Arithmetic: bf16 models keep weights, K/V caches and GEMM inputs in
 *    bf16 and accumulate, normalise and run the residual stream in fp32;
 *    fp32 models run everything in fp32 (no TF32).
 */
#ifndef ASRSPEC_H_
#define ASRSPEC_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ASR_OK 0
#define ASR_E_INVAL (-1)     /* bad argument: dims, k > max_draft, B > max_batch, null pointer */
#define ASR_E_STATE (-2)     /* call out of order: prefill before encode_cache, verify before prefill */
#define ASR_E_CAPACITY (-3)  /* t_max > max_enc, P0 > max_pos */
#define ASR_E_OOM (-4)       /* device allocation failed */
#define ASR_E_CUDA (-5)      /* a CUDA runtime call failed */
#define ASR_E_DEVICE (-6)    /* the device status word is set (see asr_spec_status) */

/* Device status bits returned by asr_spec_status. */
#define ASR_ST_BAD_TOKEN 1      /* a draft, prompt or rollback token outside [0, vocab) */
#define ASR_ST_BAD_LENS 2       /* lens[b] outside [-1, k] */
#define ASR_ST_CAPACITY 4       /* kv_len[b] + lens[b] + 1 > max_pos, or enc_len out of range */
#define ASR_ST_WAIT_TIMEOUT 8   /* a bounded pipeline wait gave up; results of that call are invalid */
#define ASR_ST_NOT_READY 16     /* an utterance slot without an encoder cache or prefill */
#define ASR_ST_BAD_TREE 32      /* tree verify: a node's parent outside [0, node) */
#define ASR_ST_BOUNDS 64        /* bounds-check mode (environment ASRSPEC_CHECK=1 at create): a kernel
                                   found an index derived from device data out of range and skipped
                                   that access; results of that call are invalid */

typedef struct asr_spec* asr_spec_handle;

typedef struct {
  int32_t n_layers;     /* decoder layers L */
  int32_t d_model;      /* d, a multiple of 64 */
  int32_t n_heads;      /* H = d / 64 */
  int32_t d_ffn;        /* MLP width, a multiple of 64 */
  int32_t vocab;        /* V */
  int32_t max_pos;      /* rows of the positional table = decoder context, e.g. 448 */
  int32_t max_batch;    /* utterance slots B_max */
  int32_t max_draft;    /* largest draft length k accepted by asr_spec_verify */
  int32_t max_enc;      /* encoder frames per utterance, e.g. 1500 */
  int32_t dtype;        /* 0 = fp32, 1 = bf16 */
  int32_t anchor_layer; /* 0-based layer read by the re-anchoring readout; -1 = floor(3 L / 4) */
} asr_model_dims;

/* Host fp32 weights, one flat blob in this order (matrices [out][in], row-major):
 *   tok_emb [V][d], pos_emb [max_pos][d],
 *   per layer: ln1_g[d] ln1_b[d] wq[d][d] bq[d] wk[d][d] wv[d][d] bv[d] wo[d][d] bo[d]
 *              ln2_g ln2_b wcq[d][d] bcq[d] wck[d][d] wcv[d][d] bcv[d] wco[d][d] bco[d]
 *              ln3_g ln3_b w1[F][d] b1[F] w2[d][F] b2[d]
 *   lnf_g[d], lnf_b[d].
 * bf16 models round each value to bf16 (nearest, ties to even) on upload. */
typedef struct {
  const float* blob;
  size_t n_floats;
} asr_weights;

/* Create a handle: validate dims, allocate device weights, caches and
 * work buffers, upload the weights.  stream: a cudaStream_t on which every
 * later call is ordered; NULL makes the handle create its own blocking stream,
 * which is ordered with work on the legacy default stream.  Synchronous.
 * Errors: ASR_E_INVAL (dims), ASR_E_OOM, ASR_E_CUDA. */
int asr_spec_create(const asr_model_dims* dims, const asr_weights* weights, void* stream,
                    asr_spec_handle* out);

/* Select host (1) or device (0, default) pointers for array arguments. */
int asr_spec_set_host_io(asr_spec_handle h, int host_io);

/* Build the cross-attention K/V cache of every layer for B utterances, once per
 * utterance (the encoded audio is reused by every verification step, Sec. 1 and
 * App. "Runtime anchor construction"): Kx_l = E Wck_l^T, Vx_l = E Wcv_l^T + bcv_l.
 *   enc_states: [B][t_max][d] in the model dtype (fp32 or bf16); always a device
 *               pointer; frames t >= enc_lens[b] are ignored.
 *   enc_lens:   [B] int32, 1 <= enc_lens[b] <= t_max.
 * Occupies slots 0..B-1 and clears their decoder state (call asr_spec_prefill next).
 * Errors: ASR_E_INVAL (B, pointers), ASR_E_CAPACITY (t_max > max_enc). */
int asr_spec_encode_cache(asr_spec_handle h, int32_t B, const void* enc_states, int32_t t_max,
                          const int32_t* enc_lens);

/* Cache a prompt of P0 tokens per utterance: K/V of prompt[b][0..P0-2] at
 * positions 0..P0-2; prompt[b][P0-1] becomes the pending token, scored by the
 * next verify at position P0-1.  prompt: [B][P0] int32.
 * Errors: ASR_E_STATE (no encoder cache), ASR_E_CAPACITY (P0 > max_pos). */
int asr_spec_prefill(asr_spec_handle h, const int32_t* prompt, int32_t P0);

/* One verification round (Sec. 3 "Speculative Loop").
 *   draft [B][k] int32: proposed tokens; entries past lens[b] are ignored.
 *   lens  [B] int32: valid drafts 0..k, or -1 for an utterance that sits out.
 * Row i of utterance b is the pending token (i = 0) or draft i, at position
 * kv_len[b] + i; it attends to the committed cache and to rows 0..i of its own
 * block.  With g_i the argmax of row i (lowest id on ties):
 *   accepted[b] = n = the largest n <= lens[b] with draft[b][j-1] == g_{j-1} for all j <= n
 *   bonus[b]    = g_n;  the new kv_len[b] = old kv_len[b] + 1 + n; pending = bonus
 *   anchor[b]   = argmax over frames j < enc_len[b] of the head mean of the
 *                 per-head softmax attention of row n at the anchor layer
 *                 (lowest frame on ties).
 * Sitting-out utterances return accepted 0, bonus -1, anchor -1, kv_len unchanged.
 * Outputs are [B] int32 each.
 * Errors: ASR_E_INVAL (k outside [0, max_draft]), ASR_E_STATE (no prefill).
 * Data errors (token id, lens, capacity) skip the whole step and set the
 * status word. */
int asr_spec_verify(asr_spec_handle h, const int32_t* draft, const int32_t* lens, int32_t k,
                    int32_t* accepted, int32_t* bonus, int32_t* kv_len, int32_t* anchor);

/* One verification round over a candidate tree per utterance (the tree
 * decoder control of App. "Alternative draft and verification changes": the
 * target verifies every node in one pass under a tree attention mask).
 *   tokens [B][n] int32: token of node i + 1 (node 0 is the pending token);
 *   parent [B][n] int32: parent of node i + 1, in [0, i] (topological order);
 *   lens   [B] int32: nodes used 0..n, or -1 for an utterance that sits out.
 * Node i is scored at position kv_len[b] + depth(i) and attends to the
 * committed cache and to its ancestors (itself included); its K/V go to cache
 * slot kv_len[b] + i.  With g_i the argmax of node i, the accepted path starts
 * at the root and moves to the first child (lowest node index) whose token is
 * g of the current node, while there is one:
 *   accepted[b] = its length n; bonus[b] = g of its last node;
 *   path[b][j]  = the node at depth j + 1 (j < n), -1 past it ([B][n] int32);
 *   the path's K/V move to positions kv_len[b] + 1 .. + n (the committed cache
 *   is then what the linear verify of that path would leave); kv_len, pending
 *   and the anchor (read at the path's last node) as asr_spec_verify.
 * A one-branch tree (parent[b][i] = i) is the linear verify.  n <= 31.
 * Errors: ASR_E_INVAL (n outside [0, min(max_draft, 31)], fp32 model),
 * ASR_E_STATE (no prefill).  Data errors (token id, a parent outside
 * [0, node), lens, capacity kv_len + lens + 1 > max_pos) skip the whole step and
 * set the status word (ASR_ST_BAD_TREE for a parent). */
int asr_spec_verify_tree(asr_spec_handle h, const int32_t* tokens, const int32_t* parent, const int32_t* lens,
                         int32_t n, int32_t* accepted, int32_t* bonus, int32_t* kv_len, int32_t* anchor,
                         int32_t* path);

/* ---- The draft (App. "Draft architecture"; Sec. 3 "Speculative Loop") ----
 *
 * A one-block draft beside the target: its input at position p is
 *   w_in [f_1; f_2; f_3; f_4] + b_in + tok_emb[token] + pos_emb[p],
 * f_i the target's residual stream after layer max(0, i L / 4 - 1) at the row
 * that scored the token (position p - 1; zeros at p = 0); then one pre-LN
 * causal block (self-attention over the draft's own cache, cross-attention to
 * the encoder states through its own K/V projections, feed-forward of width
 * 2 d with erf GELU), its own final LayerNorm and the target's tied LM head.
 * Continuation proposals have no target row: the draft's own block output at
 * p - 1 stands in for all four representations. */

/* Window kinds of the draft's audio cross-attention (App. "Attention
 * conditions", "Window geometry"): frames [c - 20, c + 20] clipped to
 * [0, T) around centre c = the last verification's anchor (deployed
 * correction, Sec. 5), the anchor + 25 frames clipped to T - 1 (shifted
 * control), a caller-given centre (random control), or every frame. */
#define ASR_DRAFT_WIN_ANCHOR 0
#define ASR_DRAFT_WIN_SHIFTED 1
#define ASR_DRAFT_WIN_RANDOM 2
#define ASR_DRAFT_WIN_NONE 3

/* Attach a draft to a bf16 handle, before asr_spec_encode_cache.
 *   draft: host fp32 blob of 16 d^2 + 18 d floats, in this order (row-major,
 *   [out][in]): w_in [d][4 d], b_in [d], ln1_g, ln1_b [d], wq [d][d], bq,
 *   wk [d][d], wv [d][d], bv, wo [d][d], bo, ln2_g, ln2_b, wcq [d][d], bcq,
 *   wck [d][d], wcv [d][d], bcv, wco [d][d], bco, ln3_g, ln3_b, w1 [2 d][d],
 *   b1 [2 d], w2 [d][2 d], b2, lnf_g, lnf_b.  Copied; the caller keeps it.
 * encode_cache then also builds the draft's cross K/V, prefill its cache of
 * the prompt rows.  Synchronous.  Errors: ASR_E_INVAL (fp32 model, blob size,
 * max_batch > 256, max_pos or max_enc > 16384), ASR_E_STATE (a draft already
 * attached, or encode_cache already ran), ASR_E_OOM, ASR_E_CUDA. */
int asr_spec_draft_create(asr_spec_handle h, const asr_weights* draft);

/* One drafting round, entirely on the device.  Per utterance b with
 * committed length P = kv_len[b] and N = total_len[b]:
 *   lens_out[b] = -1 when P + 1 >= N (it holds its transcript), else the
 *   proposals made, min(k, N - P - 2);
 * the draft first re-processes the positions the last (linear) verification
 * committed, from that verification's rows (catch-up, every frame), then
 * scores the pending token at P (restart) and its own proposals at P + 1, ...
 * (continuations), each with the round's audio window; proposal j is the
 * argmax of the pass that scored position P + j - 1.
 *   window: ASR_DRAFT_WIN_*; centers [B] int32 (ASR_DRAFT_WIN_RANDOM only,
 *           frames in [0, enc_len[b])); before the first verification the
 *           anchor is frame 0.
 *   total_len [B] int32; draft_out [B][k] int32 (entries past lens_out[b]
 *   are unspecified); lens_out [B] int32 -- both fit asr_spec_verify (tokens,
 *   lens, k) as they are.
 * Errors: ASR_E_INVAL (k outside [0, max_draft], window kind, null pointer),
 * ASR_E_STATE (no draft, or no prefill). */
int asr_spec_draft_propose(asr_spec_handle h, int32_t k, int32_t window, const int32_t* centers,
                           const int32_t* total_len, int32_t* draft_out, int32_t* lens_out);

/* Confidence threshold of the draft's proposals (App. "Draft length and
 * confidence threshold": the block length varies per utterance): with
 * threshold > 0 a round stops proposing for an utterance at the first
 * position whose argmax probability under the draft (softmax of its
 * logits) is below the threshold; that position is scored but not proposed.
 * 0 (the default) turns it off.  Applies to later asr_spec_draft_propose
 * calls; with it on, the LM head writes the pass's logits and a second
 * kernel takes the argmax and its probability.
 * Errors: ASR_E_INVAL (threshold outside [0, 1]), ASR_E_STATE (no draft), ASR_E_OOM. */
int asr_spec_draft_set_threshold(asr_spec_handle h, float threshold);

/* The restart flags of the last verify (Sec. 3: after a rejected draft the
 * next round restarts drafting from the verified position, else it
 * continues): restart[b] = 1 when accepted[b] < lens[b] (linear verify) or
 * when the accepted path's last node has children (tree verify), 0 when every
 * offered draft was accepted and for utterances that sat out.  [B] int32,
 * stream-ordered after the verify call.  Errors: ASR_E_STATE (no prefill). */
int asr_spec_restart(asr_spec_handle h, int32_t* restart);

/* Test support: the head-mean attention profile behind the last verify's
 * anchors (Sec. 5 "Verification-Attention Correction": the mean over heads of
 * the per-head softmax attention of the anchor row at the anchor layer).
 * out: [B][max_enc] fp32; entries at frames >= enc_len[b], and every entry of
 * an utterance that sat out, are stale. */
int asr_spec_debug_anchor_profile(asr_spec_handle h, float* out);

/* Roll the committed cache back (App. "Decoding and Intervention Protocol":
 * the cached states of accepted tokens are what the next round reuses):
 * kv_len[b] <- new_len[b] (which must not exceed the current kv_len[b]) and
 * pending[b] <- new_pending[b].  Cache rows at and beyond new_len are dead.
 * new_len[b] = -1 leaves utterance b unchanged.  Both [B] int32.
 * Invalid values set the status word and change nothing. */
int asr_spec_rollback(asr_spec_handle h, const int32_t* new_len, const int32_t* new_pending);

/* Read the committed lengths and pending tokens: [B] int32 each. */
int asr_spec_state(asr_spec_handle h, int32_t* kv_len, int32_t* pending);

/* Test support: the LM-head logits of every row scored by the last verify,
 * recomputed from its final-LN rows with the same tensor-core arithmetic as the
 * fused argmax.  out: [R][V] fp32 with R = the number of rows of that call
 * (sum over active b of lens[b] + 1, in utterance order); returns R (>= 0) or
 * an error. */
int asr_spec_debug_logits(asr_spec_handle h, float* out, int32_t max_rows);

/* Synchronise the stream, then return and clear the device status word
 * (ASR_ST_* bits; 0 = clean).  Negative on a CUDA error. */
int asr_spec_status(asr_spec_handle h);

/* Message of the last error on this handle (static storage of the handle). */
const char* asr_spec_last_error(asr_spec_handle h);

/* Free every device buffer of the handle.  NULL is a no-op. */
void asr_spec_destroy(asr_spec_handle h);

/* ---- Execution and measurement controls (not part of the paper's method) --
 * asr_spec_set_graphs: replay each (B, k) verify body as a captured CUDA graph
 * (default 1) or launch its kernels one by one (0).
 * asr_spec_profile: when enabled, verify launches its kernels directly and
 * brackets each kernel class with CUDA events on the handle's stream.
 * asr_spec_profile_read: synchronise, then return per class the summed event
 * time in ms (ms[ASR_PROF_N]), the kernel launches since the last read
 * (launches[ASR_PROF_N]), and the algorithmic traffic counters
 * (traffic[8]: verify calls, self K/V bytes, encoder K/V bytes, anchor key
 * bytes, scored rows; weight bytes follow from the dims), then reset all. */
#define ASR_PROF_QKV 0        /* self-attention Q/K/V projection (+ cache append) */
#define ASR_PROF_RESID 1      /* projections added to the residual: self out, cross out, MLP down */
#define ASR_PROF_QUERY 2      /* cross-attention query projection */
#define ASR_PROF_UP 3         /* MLP up projection + GELU */
#define ASR_PROF_SELF 4       /* self-attention */
#define ASR_PROF_CROSS 5      /* cross-attention */
#define ASR_PROF_LMHEAD 6     /* LM head with fused argmax */
#define ASR_PROF_LAYERNORM 7  /* stand-alone LayerNorm */
#define ASR_PROF_OTHER 8      /* row plan, embedding, accept + anchor, encoder cache build, prefill steps */
#define ASR_PROF_QKV_SELF 9   /* few rows: LayerNorm + QKV projection + self-attention, one cluster per head */
#define ASR_PROF_QUERY_CROSS 10  /* few rows: LayerNorm + cross query + cross-attention, one cluster per head */
#define ASR_PROF_N 11
int asr_spec_set_graphs(asr_spec_handle h, int enable);
int asr_spec_profile(asr_spec_handle h, int enable);
int asr_spec_profile_read(asr_spec_handle h, double* ms, int64_t* launches, uint64_t* traffic);

/* ---- Launch timeline (diagnostics; no counterpart in the paper) ----------
 * asr_spec_timeline: when enabled, verify launches its kernels directly (no
 * graph) and each launch of the verify chain records, from the GPU's global
 * timer (ns), when its first CTA started, when its first CTA was past its
 * wait on the previous kernel (programmatic dependent launch; the kernel's
 * own prefetch of constant operands comes before that point), when its last
 * CTA reached the kernel's midpoint (GEMM: its tensor-core MMAs done;
 * attention: its key loop done; others: not recorded), and when its last CTA
 * ended.  Enabling or disabling clears the record.  Each launch
 * costs three atomics per CTA; up to ASR_TL_CAP launches are recorded.
 * asr_spec_timeline_read: synchronise, then write up to `cap` launches in
 * launch order: ns[4 * i + 0..3] = (start, past the wait, midpoint, end), 0
 * where nothing was recorded, kind[i] as below; *count = the
 * launches recorded since the last read; then clear.  Host pointers. */
#define ASR_TL_CAP 65536
#define ASR_TL_OTHER 0
#define ASR_TL_PLAN 1          /* row plan of a verify step */
#define ASR_TL_EMBED 2         /* token + position embedding */
#define ASR_TL_LAYERNORM 3     /* stand-alone LayerNorm */
#define ASR_TL_ATTN_SELF 4     /* self-attention */
#define ASR_TL_ATTN_CROSS 5    /* cross-attention */
#define ASR_TL_ACCEPT 6        /* acceptance, commit and anchor readout */
#define ASR_TL_QKV_SELF 8      /* few rows: LayerNorm + QKV + self-attention, one cluster per head */
#define ASR_TL_QUERY_CROSS 9   /* few rows: LayerNorm + cross query + cross-attention, one cluster per head */
#define ASR_TL_GEMM 16         /* + epilogue: 0 plain, 1 QKV + cache append, 2 residual, 3 query, 4 GELU, 6 argmax */
#define ASR_TL_LN_FUSED 32     /* added to a GEMM kind whose input LayerNorm is folded into it (no LayerNorm launch) */
int asr_spec_timeline(asr_spec_handle h, int32_t enable);
int asr_spec_timeline_read(asr_spec_handle h, uint64_t* ns, int32_t* kind, int32_t cap, int32_t* count);


/* ---- Diagnostics of the few-row layers (not part of the paper's method) ---
 * asr_spec_fewrow_trace: when enabled, every verify that runs the few-row
 * layers (bf16 models, batch x (k + 1) <= 9 rows) records, per CTA of each of
 * its 6 L layer launches, the GPU global timer (ns) at 12 phases: entry, past
 * the wait on the previous launch, input rows ready, weights landed,
 * projection reduced, exchange landed, attention done, exit, first K/V chunk
 * landed, first chunk combined, merge inputs landed, bf16 input rows landed
 * (GEMVs without a LayerNorm) (0 where a launch has no such phase); verify
 * then launches directly (no graph).  A
 * verify of more rows records its 6 L tensor-core projections instead (in
 * layer order: QKV, self out, cross query, cross out, MLP up, MLP down), for
 * their first 320 CTAs: 0 entry, 1 set-up done, 2 first k-block landed,
 * 3 MMAs done, 4 exit, 5 K-split partial staged (one CTA per tile: tile
 * staged in shared memory), 6 partials landed (staging barrier passed),
 * 7 reduction done (rows written), 8 past the wait on the previous launch,
 * 9 last k-block issued, 10 epilogue operands loaded, 11 first rows written
 * (many-row kernel).  ASR_E_INVAL for an fp32 model.
 * asr_spec_fewrow_trace_read: synchronise and copy the last traced call's
 * stamps, [n_launches][320 CTAs][12] words in launch order, up to `cap` words. */
int asr_spec_fewrow_trace(asr_spec_handle h, int32_t enable);
int asr_spec_fewrow_trace_read(asr_spec_handle h, uint64_t* out, int64_t cap, int32_t* n_launches);

/* ---- Workload utility (not part of the paper's method) -------------------
 * Synthetic draft source used by benchmarks in place of a trained draft
 * model: draft i (1-based) of a round at committed length P is
 * truth[b][P+i] (or truth[b][P+i-1] when shift[b][P] = s > 0 and i >= s),
 * replaced by repl[b][P][i-1] when that is >= 0.  lens[b] = -1 once
 * P + 1 >= total_len[b], else min(k, total_len[b] - P - 2).
 *   truth [B][max_pos], total_len [B], repl [B][max_pos][k_repl], shift [B][max_pos];
 *   draft_out [B][k], lens_out [B].  Device pointers only. */
int asr_spec_synth_drafts(asr_spec_handle h, const int32_t* truth, const int32_t* total_len,
                          const int32_t* repl, int32_t k_repl, const int32_t* shift, int32_t k,
                          int32_t* draft_out, int32_t* lens_out);

/* ---- Kernel test entry (not part of the paper's method) ------------------
 * C[m][n] = sum_k A[m][k] * B[n][k] through the tcgen05 tensor-core GEMM
 * (impl 0), the same with a 3-way K split over a global workspace (impl 2) or
 * with K split inside a thread-block cluster and wide N tiles (impl 4), or
 * the SIMT GEMM (impl 1);
 * impl 3 runs the LM-head epilogue instead and writes C[n] = the index m of
 * the largest value of column n (lowest m on ties).  Impls 5 - 7 run the
 * many-row kernel (one tile per SM; K split over a cluster pair from 48
 * k-blocks in 7) with zero bias and write C transposed, [n][m]: 5 the query
 * epilogue, 6 GELU (bf16 result widened to fp32), 7 the residual epilogue
 * onto x = 0; M % 128 == 0.  A, B bf16 row-major device arrays, C fp32.
 * K % 64 == 0.  Synchronous. */
int asr_spec_test_gemm(int32_t impl, const void* A, const void* B, float* C, int32_t M, int32_t N,
                       int32_t K, void* stream);

/* ---- Split-K GEMM without device allocation ------------------------------
 * The paper has no counterpart to this entry: it serves callers that may not
 * allocate device memory at all, such as a host framework that owns every
 * device byte through its own pool, a serving loop that forbids allocation
 * after start-up because cudaMalloc/cudaFree can synchronise the whole device,
 * or code running while another thread captures a CUDA graph in a mode that
 * rejects such calls.
 * Computes C[m][n] = sum_k A[m][k] * B[n][k] with the tcgen05 GEMM, K split
 * into `splits` ranges (1 <= splits <= K / 64) whose partial sums are added in
 * split order; A [M][K], B [N][K] bf16 row-major, C [M][N] fp32, all device
 * pointers owned by the caller; K % 64 == 0.  It calls no cudaMalloc, cudaFree
 * or allocating library routine: the split-K partial sums, tile tickets and
 * status word live in one fixed device array of about 8 MiB (2^21 partial
 * floats, 4096 output tiles) that every GPU loading the library keeps until
 * the process exits.  Calls needing more return ASR_E_CAPACITY.  The first
 * call on a device looks the array's address up (make it before any stream
 * capture on that device).  All calls share the array: each one clears the
 * tickets and status before its kernel, and calls that overlap on the GPU
 * race.  Synchronises `stream` before returning; ASR_E_DEVICE if a bounded
 * pipeline wait gave up, ASR_E_INVAL for bad arguments. */
int asr_spec_gemm_noalloc(const void* A, const void* B, float* C, int32_t M, int32_t N, int32_t K,
                          int32_t splits, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* ASRSPEC_H_ */
