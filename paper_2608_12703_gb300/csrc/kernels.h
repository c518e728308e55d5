// Host-side launchers of the draft-verify kernels (internal to libasrspec).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>
#include <cuda.h>

#include "epilogue.cuh"

namespace asrspec {

// ---- GEMM: C[m][n] = sum_k A[m][k] B[n][k] (+ epilogue) ---------------------
// tcgen05 path: A, B bf16 K-major, described by 2-D tensor maps (box 64 x 128
// for A, 64 x BN for B, 128-byte swizzle).  K % 64 == 0.
struct TcGemm {
  CUtensorMap mapA;
  CUtensorMap mapB;
  int M, N, K;
  int bn;        // N tile: 16, 32, 64, 128, 192, 224 or 256
  int splits;    // split-K factor (1 = none)
  float* ws;     // workspace split: partials (splits * tiles * 128 * bn floats)
  int* tickets;  // workspace split: one zeroed int per output tile
  bool cluster = false;  // split K inside a thread-block cluster (splits in {2,4,8,16})
  bool pdl = false;      // programmatic dependent launch after the previous kernel
};

bool make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows);
int tc_pick_bn(int n_max);
int tc_pick_bn_wide(int n);
void launch_gemm_tc(const TcGemm& g, int mode, const Epi& epi, int* status, cudaStream_t st);
size_t tc_smem_bytes(int bn);
// 2-D fp32 tensor map over [rows][cols], no swizzle, box {box_cols, box_rows}.
bool make_tmap_f32(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                   uint32_t box_rows);

// Many-row projections (csrc/gemm_wide.cuh): one 128 x bn tile per CTA, about
// one CTA per SM; modes QKV, Q, GELU, RESID (M % 128 == 0, K % 64 == 0).
struct WideGemm {
  CUtensorMap mapA;   // weights [M][K], box 64 x 128
  CUtensorMap mapB;   // rows [R][K], box 64 x bn
  CUtensorMap mapX;   // RESID: the residual stream [R][d] fp32, box 128 x bn (others: unused)
  int M, N, K;
  int bn, split;      // N tile (32 .. 160, RESID <= 96); 1, or 2 = K split over a cluster pair
  int stages = 0;     // stages per pipeline, at least 1 (0: as deep as shared memory allows)
  bool pdl = false;
};
bool wide_pick(int M, int N, int K, int mode, int sms, int* bn, int* split);
void launch_gemm_wide(const WideGemm& g, int mode, const Epi& epi, int* status, cudaStream_t st);
void configure_gemm_tc();
void configure_attention();

// SIMT path (fp32 models, and a cross-check of the tensor-core path).
// A: [M][K] of type a_bf16 ? bf16 : fp32; B: [N][K] likewise.
void launch_gemm_simt(const void* A, int a_bf16, const void* B, int b_bf16, int M, int N, int K, int mode,
                      const Epi& epi, cudaStream_t st);

// ---- Row bookkeeping, embedding, LayerNorm ---------------------------------
struct RowPlan {
  int* row_b;       // [R_max]
  int* row_i;       // [R_max]
  int* row_pos;     // [R_max] cache slot of the row's K/V (its position, but for tree nodes)
  int* row_epos;    // [R_max] position of the row's token (positional embedding)
  unsigned* row_mask;   // [R_max] tree verify: the row's ancestors (bit j = node j of its utterance)
  int* row_tok;     // [R_max]
  int* row_start;   // [B_max + 1]
  int* n_rows;      // [1] rows of this step (0 when the step is refused)
  int* n_utt_rows;  // [B_max] rows of utterance b this step (lens+1, or 0)
};

// Per-step algorithmic traffic, accumulated on the device (bench support):
// counters[0] verify calls, [1] self K/V bytes, [2] cross K/V bytes,
// [3] anchor key bytes, [4] scored rows.
struct TrafficArgs {
  unsigned long long* counters;
  const int* enc_len;
  int n_layers, d, elem_bytes;
};

// Validate the step's inputs, lay out the rows and reset the argmax keys.
// parent (tree verify, else null): [B][k], the parent node of node i + 1 in
// [0, i] (node 0 is the pending token); node i goes to cache slot kv_len + i
// at position kv_len + depth(i).
void launch_plan_verify(const int* draft, const int* lens, int k, int B, int vocab, int max_pos, const int* kv_len,
                        const int* pending, const int* ready, RowPlan plan, unsigned long long* row_key,
                        int* status, const TrafficArgs& tr, cudaStream_t st, unsigned long long* tl = nullptr,
                        const int* parent = nullptr);
void launch_plan_prefill_chunk(const int* prompt, int P0, int p0, int c, int B, int vocab, const int* ready,
                               RowPlan plan, int* status, cudaStream_t st);
// xg / gain / st_part: the folded first LayerNorm's operand bf16(gain * x) [R][d]
// and the rows' statistics (one slice of d features), or null.
void launch_embed(const void* tok_emb, const void* pos_emb, int w_bf16, RowPlan plan, int R_max, int d, float* x,
                  cudaStream_t st, bool pdl, unsigned long long* tl, __nv_bfloat16* xg, const float* gain,
                  float2* st_part, int vocab, int max_pos, int* status);
// c1[m] = sum_k W[m][k] g[k], c2[m] = sum_k W[m][k] b[k] for a bf16 W [M][K].
void launch_ln_fold(const void* W, const float* g, const float* b, int M, int K, float* c1, float* c2,
                    cudaStream_t st);
// y = LN(x) * g + b over rows < n_rows, written as bf16 or fp32.
void launch_layernorm(const float* x, const float* g, const float* b, void* y, int y_bf16, const int* n_rows,
                      int R_max, int d, cudaStream_t st, bool pdl = false, unsigned long long* tl = nullptr);

// ---- Attention ---------------------------------------------------------------
struct AttnArgs {
  const float* q;          // [R][d] fp32 queries
  const void* kc;          // key cache base of this layer:   [B_max][H][T_alloc][64]
  const void* vc;          // value cache base of this layer
  int kv_bf16;
  int t_alloc;             // rows per (b, h) in the cache (max_pos or max_enc)
  int causal;              // 1: self-attention, keys 0..row_pos; 0: cross, keys 0..enc_len-1
  const int* enc_len;      // [B_max] (cross)
  const int* kv_len;       // [B_max] committed lengths (self; keys up to kv_len + i)
  RowPlan plan;
  int B, H, d, k1;         // utterances, heads, d_model, rows per utterance slot (k + 1)
  int chunk;               // keys per split
  int n_chunks;            // splits per (b, h)
  float* part;             // [B][H][n_chunks][k1] x (64 + 2) partials
  void* out;               // [R][d] attention output (bf16 or fp32)
  int out_bf16;
  float* ml_out;           // optional [R][H][2] (max, sum) of the full softmax
  // tensor-core path (bf16 caches): 2-D tensor maps over the whole K and V
  // caches ([rows][64], 128-byte swizzle) and the row of (b = 0, h = 0, t = 0)
  // of this layer in each; per-(b, h) tickets for the in-kernel chunk merge
  const CUtensorMap* kmap = nullptr;
  const CUtensorMap* vmap = nullptr;
  long long k_row0 = 0, v_row0 = 0;
  int* tickets = nullptr;
  int rows_max = 0;        // most rows of one utterance in this call
  int splits = 1;          // CTAs (one cluster) per (utterance, head)
  bool pdl = false;        // programmatic dependent launch
  bool tree = false;       // self-attention of a tree verify: slots past kv_len visible by plan.row_mask
  unsigned long long* tl = nullptr;   // launch timeline slot (tl_mark), or null
  int* status = nullptr;   // device status word (bounds-check mode)
};
void launch_attention(const AttnArgs& a, cudaStream_t st);
void launch_attention_tc(const AttnArgs& a, int* status, cudaStream_t st);
// Tensor map over a [rows][64] bf16 cache with `box_rows`-row boxes.
bool make_tmap_cache(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows);

// Acceptance + commit + anchor readout (one kernel).
struct AcceptAnchorArgs {
  const int* draft;                 // [B][k]
  int k, B, H, d, t_alloc, kv_bf16;
  RowPlan plan;
  const unsigned long long* row_key;
  int* kv_len;
  int* pending;
  int *accepted, *bonus, *kv_len_out, *anchor_out;
  int* restart;                     // [B]: 1 when the next round restarts (a draft was rejected), else 0
  float* profile;                   // [B][t_alloc]: the head-mean profile of the anchor row (test readback)
  const float* q_anchor;            // [R][d] cross-attention queries at the anchor layer
  const float* ml;                  // [R][H][2] their softmax (max, sum)
  const void* kc;                   // anchor layer's encoder keys [B_max][H][t_alloc][64]
  const int* enc_len;
  unsigned long long* frame_key;    // [B_max], zero between calls
  int* tickets;                     // [B_max], zero between calls
  int* status;                      // wait time-outs (ST_WAIT_TIMEOUT)
  const int* parent = nullptr;      // tree verify: [B][k] parents (as the plan), else null
  int* path = nullptr;              // tree verify: [B][k] accepted nodes by depth (-1 past the path)
  bool pdl;
  unsigned long long* tl = nullptr;   // launch timeline slot (tl_mark), or null
};
void launch_accept_anchor(const AcceptAnchorArgs& a, cudaStream_t st);
// Tree verify commit: the accepted path's self K/V (every layer and head) from
// the nodes' slots kv_len_old + path[j] to the positions kv_len_old + j + 1.
// Reads the new kv_len and the accepted count (kv_len_old = kv_len - 1 - n).
void launch_tree_commit(const int* path, int k, const int* accepted, const int* kv_len, int B, int L, int H,
                        int max_pos, int b_max, void* kself, void* vself, int es, int* status, cudaStream_t st);

// ---- Few-row verify layers (csrc/fewrow.cu) ------------------------------------
// A step of at most VF_ROWS rows runs each decoder layer as six launches:
// LayerNorm + QKV + self-attention (one cluster per head), output projection,
// LayerNorm + cross query + cross-attention (one cluster per head), output
// projection, LayerNorm + MLP up, MLP down; the projections as GEMVs over
// 8-feature tiles (no split-K exchange).
constexpr int VF_ROWS = 9;
enum FrMode : int { FR_RESID = 0, FR_GELU = 1 };
struct FrGemv {
  const __nv_bfloat16* W;   // [N][K] weights
  const float* bias;        // [N]
  int N, K;                 // outputs, inputs
  int tiles_max;            // 8-feature tiles per CTA, at most (<= 5): ceil(N / 8 / groups)
  const float* x;           // FR_GELU: the residual stream [R][K] (LayerNorm input)
  const float *ln_g, *ln_b;
  const __nv_bfloat16* a;   // FR_RESID: bf16 input rows [R][K]
  float* x_out;             // FR_RESID: x[r][m] += y + bias  ([R][N])
  __nv_bfloat16* h_out;     // FR_GELU: bf16(gelu(y + bias))  ([R][N])
  const int* n_rows;
  int* status;
  unsigned long long* tl;
  unsigned long long* trace;   // per-CTA phase stamps [CTA][FR_TRACE_PHASES] (diagnostics), or null
  const void* pf;              // a later launch's weights, prefetched into L2 (or null)
  uint32_t pf_bytes;
};
struct FrHead {
  const __nv_bfloat16* W;   // self: fused QKV weights [3d][d]; cross: query weights [d][d]
  const float* bias;
  const float *x, *ln_g, *ln_b;   // the residual stream and the LayerNorm in front of W
  int d, H, C, B, max_pos;
  int tiles_max;            // weight tiles per CTA, at most
  int mrg_slots;            // partials a merging CTA can hold per row
  RowPlan plan;
  const int* kv_len;
  const int* enc_len;
  __nv_bfloat16 *ks, *vs;   // self: this layer's caches [B_max][H][max_pos][64] (new rows appended)
  long long row0;           // tensor-map row of this layer's (utterance 0, head 0, key 0)
  long long vofs;           // cross: rows from the K half to the V half of the encoder cache
  int t_alloc;              // tensor-map rows per (utterance, head)
  __nv_bfloat16* att;       // [R][d] attention output
  float* q_anchor;          // cross at the anchor layer: fp32 queries [R][d], else null
  float* ml;                // cross at the anchor layer: softmax (max, sum) [R][H][2], else null
  int* status;
  unsigned long long* tl;
  unsigned long long* trace;   // per-CTA phase stamps [CTA][FR_TRACE_PHASES] (diagnostics), or null
  const void* pf;              // a later launch's weights, prefetched into L2 (or null)
  uint32_t pf_bytes;
};
// Phase stamps of a traced few-row launch, GPU global timer (ns), thread 0 of
// each CTA: 0 entry, 1 past the wait on the previous launch, 2 input rows
// ready, 3 weights landed, 4 projection reduced, 5 exchange landed (head:
// gathered q/k/v; K-split group: the other ranks' partials), 6 attention
// done (head), 7 exit; head kernels also 8 first K/V chunk landed, 9 first
// chunk's attention combined, 10 merge inputs landed, 11 (GEMVs without a
// LayerNorm) bf16 input rows landed.  Up to FR_TRACE_CTAS
// CTAs per launch.
constexpr int FR_TRACE_PHASES = 12;
constexpr int FR_TRACE_CTAS = 320;
// 1 and the cluster size per head when the kernels run for these dimensions on this device
// (gd_out: the MLP down-projection's groups of F / d CTAs)
int fr_configure(int d, int F, int H, int max_pos, int* C_out, int* sms_out, int* gd_out);
size_t fr_gemv_smem(int d, int K, int tiles_max, int ks);
size_t fr_head_smem(int d, int tiles_max, bool self_attn, int mrg_slots);
// groups: CTA groups of ks (one cluster each); a.tiles_max = ceil(N / 8 / groups)
// Pack a bf16 [N][K] weight matrix (N, K multiples of 8) into the few-row
// kernels' tile layout: 8-row tiles, contiguous, 16-byte pieces piece-major.
cudaError_t launch_fr_pack(const void* src, void* dst, int N, int K, cudaStream_t st);
cudaError_t launch_fr_gemv(const FrGemv& a, int mode, int ks, int groups, int d, cudaStream_t st, bool pdl);
cudaError_t launch_fr_self(const CUtensorMap* kmap, const CUtensorMap* vmap, const FrHead& a, cudaStream_t st,
                           bool pdl);
cudaError_t launch_fr_cross(const CUtensorMap* xmap, const FrHead& a, cudaStream_t st, bool pdl);

// ---- Draft side (csrc/draft.cu) ---------------------------------------------------
// Window centre of the draft's audio cross-attention for proposals
// (App. "Window geometry"): the verification anchor (deployed), 500 ms later
// (shifted control), a given frame (random control), or no window.
enum DraftWin : int { DRAFT_WIN_ANCHOR = 0, DRAFT_WIN_SHIFTED = 1, DRAFT_WIN_RANDOM = 2, DRAFT_WIN_NONE = 3 };
struct DraftArgs {
  int B, d, k, k_verify, win_kind;
  int vocab, max_pos, r_max;   // token ids, positions, rows of the pass buffers
  int* status;               // device status word (ASR_ST_* bits)
  int after_verify;          // 1: a verification ran since the last round (catch-up rows)
  const int *kv_len, *pending, *enc_len, *total_len;
  const int *v_row_start, *v_n_utt_rows;   // the last verification's row plan
  const int *accepted, *anchor;             // its outputs
  const int* v_draft;        // [B][k_verify] its drafts
  const int* centers;        // [B] window centres of the random control, or null
  const float* taps;         // [R][4][d] tapped target rows (verification or prefill chunk)
  float* last_tap;           // [B_max][4][d] the tap of the last prompt row per utterance
  const float* x_prev;       // [R][d] the previous pass's block output (continuation rows)
  RowPlan plan;              // the draft pass's rows
  int *row_src, *row_lo, *row_hi;   // [R_max] feature source; audio window [lo, hi) per row
  int *win_lo, *win_hi;      // [B_max] the round's window
  int *lens, *n_prop, *last_row, *prev_pos;   // [B_max]
  int* draft_out;            // [B][k] proposals
  unsigned long long* row_key;   // [R_max] LM-head argmax keys of the pass
  __nv_bfloat16* x_in;       // [R_max][4 d] the pass's input representations
  float threshold;           // confidence threshold on the proposal's probability (0 = off)
  const float* row_p;        // [R_max] softmax probability of each row's argmax (threshold on)
};
struct DraftAttn {
  const float* q;            // [R][d] fp32
  const __nv_bfloat16 *kc, *vc;   // [B_max][H][t_alloc][64]
  int t_alloc, B, H, d, causal;
  RowPlan plan;
  const int *row_lo, *row_hi;
  __nv_bfloat16* out;        // [R][d]
  int* status;               // device status word (bounds-check mode)
};
void launch_draft_round_plan(const DraftArgs& a, cudaStream_t st);
void launch_draft_next_plan(const DraftArgs& a, int i, cudaStream_t st);
void launch_draft_gather(const DraftArgs& a, int rows_max, cudaStream_t st);
void launch_draft_prefill_gather(const DraftArgs& a, int rows_max, cudaStream_t st);
void launch_draft_embed(const DraftArgs& a, int rows_max, const void* tok_emb, const void* pos_emb, float* x,
                        cudaStream_t st);
void launch_draft_take(const DraftArgs& a, cudaStream_t st);
void launch_draft_finish(const DraftArgs& a, int* lens_out, cudaStream_t st);
void launch_draft_attn(const DraftAttn& a, cudaStream_t st);
// Per row of logits [rows][V] (fp32): the argmax key (as the LM-head epilogue
// writes it: lowest index on ties) and the softmax probability of the argmax.
void launch_draft_softmax(const float* logits, int V, const int* n_rows, int rows_max, unsigned long long* row_key,
                          float* row_p, cudaStream_t st);

// ---- Accept / commit ------------------------------------------------------------
void launch_prefill_advance(int B, int c, const int* n_utt_rows, int* kv_len, cudaStream_t st);
void launch_prefill_finish(const int* prompt, int P0, int B, int* pending, const int* ready, cudaStream_t st);
void launch_rollback(const int* new_len, const int* new_pending, int B, int vocab, int* kv_len, int* pending,
                     int* status, cudaStream_t st);
void launch_synth_drafts(const int* truth, const int* total_len, const int* repl, int k_repl, const int* shift, int k,
                         int B, int max_pos, const int* kv_len, int* draft_out, int* lens_out, cudaStream_t st);
void launch_mark_ready(const int* enc_len, int B, int t_max, int* ready, int* kv_len, int* pending, int* status,
                       cudaStream_t st);
int attn_chunk_len(int kv_bf16);

// Bounds-check mode switches, one per translation unit (see bounds_bad).
void set_check_gemm_tc(int on);
void set_check_gemm_simt(int on);
void set_check_gemm_wide(int on);
void set_check_rows(int on);
void set_check_attention(int on);
void set_check_attention_tc(int on);
void set_check_fewrow(int on);
void set_check_draft(int on);

}  // namespace asrspec
