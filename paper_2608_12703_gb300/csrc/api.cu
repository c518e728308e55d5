// C ABI of the draft-verify step: handle, weights upload, per-utterance
// encoder cache, prefill, verify, rollback.  See include/asrspec.h.
#include <algorithm>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <map>
#include <string>
#include <vector>

#include "kernels.h"

using namespace asrspec;

namespace {

constexpr int NUM_SMS_TARGET = 152;

struct LayerW {
  void *wqkv, *wo, *wcq, *wco, *w1, *w2;
  float *bqkv, *bo, *bcq, *bco, *b1, *b2;
  float *ln1g, *ln1b, *ln2g, *ln2b, *ln3g, *ln3b;
  // folded LayerNorm constants (c1 = W g, c2 = W b) of the three projections
  // whose input is a LayerNorm output
  float *c1_qkv = nullptr, *c2_qkv = nullptr, *c1_cq = nullptr, *c2_cq = nullptr, *c1_fc1 = nullptr, *c2_fc1 = nullptr;
  CUtensorMap m_wqkv, m_wo, m_wcq, m_wco, m_w1, m_w2;
  // the same weights packed for the few-row kernels (launch_fr_pack), or null
  void *p_qkv = nullptr, *p_wo = nullptr, *p_wcq = nullptr, *p_wco = nullptr, *p_w1 = nullptr, *p_w2 = nullptr;
};

}  // namespace

// The one-block draft (asr_spec_draft_create): weights as the target layer's,
// feed-forward width 2 d, its own cross K/V projections and final LayerNorm.
struct DraftW {
  void *w_in = nullptr, *wqkv = nullptr, *wo = nullptr, *wcq = nullptr, *wco = nullptr, *w1 = nullptr, *w2 = nullptr,
       *w_cross = nullptr;
  float *b_in = nullptr, *bqkv = nullptr, *bo = nullptr, *bcq = nullptr, *bco = nullptr, *b1 = nullptr, *b2 = nullptr,
        *b_cross = nullptr;
  float *ln1g = nullptr, *ln1b = nullptr, *ln2g = nullptr, *ln2b = nullptr, *ln3g = nullptr, *ln3b = nullptr,
        *lnfg = nullptr, *lnfb = nullptr;
  CUtensorMap m_in, m_qkv, m_wo, m_wcq, m_wco, m_w1, m_w2;
};

struct asr_spec {
  asr_model_dims dims{};
  int L = 0, d = 0, H = 0, F = 0, V = 0, maxpos = 0, Bmax = 0, kmax = 0, Tmax = 0, anchor = 0;
  bool bf16 = true;
  size_t es = 2;  // element size of weights / caches / GEMM inputs
  cudaStream_t st = nullptr;
  bool own_stream = false;
  int host_io = 0;
  int state = 0;  // 0 created, 1 encoder cache built, 2 prefilled
  int B = 0, t_max = 0;
  std::string err;

  std::vector<void*> allocs;
  void *w_tok = nullptr, *w_pos = nullptr, *w_cross = nullptr;
  float *b_cross = nullptr, *lnf_g = nullptr, *lnf_b = nullptr;
  float *c1_lm = nullptr, *c2_lm = nullptr;   // folded final LayerNorm of the LM head
  CUtensorMap m_tok{};
  std::vector<LayerW> lw;

  void *kself = nullptr, *vself = nullptr, *xkv = nullptr;
  int *enc_len = nullptr, *kv_len = nullptr, *pending = nullptr, *ready = nullptr;

  int R_max = 0, R_pad = 0;
  float *x = nullptr, *q = nullptr, *q_anchor = nullptr, *ml = nullptr, *part = nullptr;
  void *xn = nullptr, *att = nullptr, *hbuf = nullptr, *xf = nullptr;
  RowPlan plan{};
  unsigned long long* row_key = nullptr;
  unsigned long long* frame_key = nullptr;  // [Bmax] keys + [Bmax] int tickets
  int* anchor_row = nullptr;
  // out4: accepted, bonus, kv_len, anchor and restart of the last verify, [Bmax] each
  int *draft_buf = nullptr, *lens_buf = nullptr, *prompt_buf = nullptr, *out4 = nullptr, *misc = nullptr;
  float* anchor_prof = nullptr;   // [Bmax][Tmax] head-mean profile of the last verify's anchor rows
  int* status = nullptr;
  float* ws = nullptr;
  size_t ws_floats = 0;
  int* tickets = nullptr;
  int n_tickets = 0;
  int* attn_tickets = nullptr;                       // [B_max * H], tensor-core attention merge
  CUtensorMap m_kself[2], m_vself[2], m_xkv[2];      // boxes of 128 and 256 rows
  std::map<std::pair<int, int>, CUtensorMap> bmaps;  // (buffer id, BN) -> map
  std::map<int, CUtensorMap> xmaps;                   // BN -> map of the residual stream (fp32, box 128 x BN)
  int n_sms = 0;
  bool use_wide = true;   // many-row projections on the one-tile-per-SM kernel (ASRSPEC_WIDE=0: the split-K chain)
  int fr_prefetch = 3;    // few-row launches prefetch the weights of the launch this many ahead into L2 (0: none)
  int wide_stages = 0;    // its stages per pipeline (ASRSPEC_WIDE_STAGES; 0 = as deep as shared memory allows)

  // profiling: CUDA events around each kernel class (direct launches only)
  bool prof = false;
  bool capturing = false;
  std::vector<cudaEvent_t> ev_pool;
  size_t ev_used = 0;
  std::vector<std::pair<int, size_t>> marks;      // (class, index of start event)
  long long launches[ASR_PROF_N] = {};
  long long cur[ASR_PROF_N] = {};                 // launches of the call being enqueued
  unsigned long long* counters = nullptr;         // device traffic counters [8]
  // CUDA graphs of the verify body, keyed by (B, k)
  bool use_graphs = true;
  bool use_pdl = true;   // programmatic dependent launch between verify kernels
  // LayerNorm folded into its neighbours (bf16, d % 128 == 0, N tiles <= 64):
  // the producer of x writes bf16(g * x) into xn and slice statistics into
  // ln_part; the consumer GEMM corrects its accumulators.  ln_S / ln_c: the
  // slices of the last producer.
  bool ln_fold = false;
  float2* ln_part = nullptr;
  int ln_S = 0, ln_c = 0;
  // few-row verify layers (csrc/fewrow.cu) for steps of at most VF_ROWS rows:
  // the cluster size per head (0 = unavailable for this model or device);
  // ASRSPEC_FEWROW=0 keeps the tensor-core chain for every step
  bool use_fewrow = true;
  int fr_C = 0;
  int fr_sms = 0;   // SMs of the device: the GEMVs run one CTA (group) per SM
  int fr_gd = 0;    // groups of the MLP down-projection (clusters resident at once)
  bool last_fused = false;    // the last verify ran the few-row layers (LM-head input in xf)
  // per-CTA phase stamps of the few-row launches of the last traced call
  // (diagnostics): [6 L][FR_TRACE_CTAS][FR_TRACE_PHASES]
  unsigned long long* fr_trace = nullptr;
  bool fr_trace_on = false;
  int fr_trace_n = 0;
  // tree verify: the nodes' parents and the accepted path ([B_max][max_draft]),
  // and whether the step being enqueued is one
  int *parent_buf = nullptr, *path_buf = nullptr;
  bool cur_tree = false;
  int wide_bn = 64;      // N tile for many rows (ASRSPEC_WIDE_BN: 64, 128, 192, 224, 256)
  int wide_target = 2 * 152;   // CTAs a many-row GEMM may fill by splitting K (ASRSPEC_WIDE_TARGET)
  int few_target = 2 * 152;    // the same for few rows (ASRSPEC_FEW_TARGET)
  // encoder-cache GEMM: N tile (ASRSPEC_ENC_BN) and M tiles per band of the
  // grouped order (ASRSPEC_ENC_GROUP, 0 = plain); measured at 64 utterances x
  // 1500 frames: 14.5 ms (128, 64) against 16.7 (256, 32) and 23.6 (256, plain)
  int enc_bn = 128;
  int enc_group = 64;
  // launch timeline (diagnostics): [ASR_TL_CAP][4] device slots, the kind of
  // each recorded launch, and the slot of the launch being enqueued
  bool tl_on = false;
  unsigned long long* tl_buf = nullptr;
  std::vector<int> tl_kind;
  unsigned long long* tl_cur = nullptr;
  struct Graph {
    cudaGraphExec_t exec;
    long long launches[ASR_PROF_N];
    int ln_S, ln_c;   // the folded LayerNorm slices the captured body leaves (for debug_logits)
    bool fused;       // the body runs the few-row layers
  };
  std::map<std::pair<int, int>, Graph> graphs;
  // the draft: weights, caches, the tapped target rows and its pass buffers
  bool has_draft = false;
  DraftW dw;
  int taps[4] = {0, 0, 0, 0};   // target layers whose outputs the draft reads
  void *d_ks = nullptr, *d_vs = nullptr, *d_xkv = nullptr;
  float *d_taps = nullptr, *d_last_tap = nullptr, *d_x = nullptr, *d_q = nullptr;
  void *d_xin = nullptr, *d_xn = nullptr, *d_att = nullptr, *d_h = nullptr, *d_xf = nullptr;
  RowPlan d_plan{};
  int *d_row_src = nullptr, *d_row_lo = nullptr, *d_row_hi = nullptr, *d_win_lo = nullptr, *d_win_hi = nullptr;
  int *d_lens = nullptr, *d_nprop = nullptr, *d_last_row = nullptr, *d_prev_pos = nullptr, *d_out = nullptr;
  int *d_total = nullptr, *d_centers = nullptr, *d_lens_out = nullptr;
  unsigned long long* d_row_key = nullptr;
  bool d_after_verify = false;
  float d_threshold = 0.f;            // confidence threshold of the proposals (0 = off)
  float* d_logits = nullptr;          // threshold on: the pass's logits [R_pad][V]
  float* d_row_p = nullptr;           // threshold on: [R_pad] probability of each row's argmax
  int last_k = 0;   // k of the last linear verification (stride of its drafts)
};

namespace {

int fail(asr_spec* h, int code, const std::string& msg) {
  if (h) h->err = msg;
  return code;
}

cudaEvent_t next_event(asr_spec* h) {
  if (h->ev_used == h->ev_pool.size()) {
    cudaEvent_t e;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    h->ev_pool.push_back(e);
  }
  return h->ev_pool[h->ev_used++];
}

// Counts the launches of one kernel class and, when profiling, brackets them
// with CUDA events on the handle's stream.
struct Prof {
  asr_spec* h;
  int cls;
  size_t idx = 0;
  bool on = false;
  Prof(asr_spec* h_, int cls_, int n_launch) : h(h_), cls(cls_) {
    if (h->capturing) h->cur[cls] += n_launch;   // replayed with the graph
    else h->launches[cls] += n_launch;
    if (h->prof && !h->capturing) {
      cudaEvent_t e1 = next_event(h);
      cudaEvent_t e2 = next_event(h);
      if (e1 && e2) {
        idx = h->ev_used - 2;
        cudaEventRecord(e1, h->st);
        on = true;
      }
    }
  }
  ~Prof() {
    if (on) {
      cudaEventRecord(h->ev_pool[idx + 1], h->st);
      h->marks.emplace_back(cls, idx);
    }
  }
};

// Gives the next launch a timeline slot (h->tl_cur) when the timeline is on.
struct Tl {
  asr_spec* h;
  Tl(asr_spec* h_, int kind) : h(h_) {
    h->tl_cur = nullptr;
    if (h->tl_on && !h->capturing && h->tl_buf && (int)h->tl_kind.size() < ASR_TL_CAP) {
      h->tl_cur = h->tl_buf + 4 * h->tl_kind.size();
      h->tl_kind.push_back(kind);
    }
  }
  ~Tl() { h->tl_cur = nullptr; }
};

#define CK(call)                                                                       \
  do {                                                                                 \
    cudaError_t e_ = (call);                                                           \
    if (e_ != cudaSuccess) return fail(h, ASR_E_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

template <typename T>
int dalloc(asr_spec* h, T** p, size_t bytes) {
  void* v = nullptr;
  if (cudaMalloc(&v, bytes) != cudaSuccess) return fail(h, ASR_E_OOM, "cudaMalloc failed");
  h->allocs.push_back(v);
  *p = static_cast<T*>(v);
  return 0;
}

// Round fp32 -> bf16 (nearest, ties to even), host side.
uint16_t f2bf_host(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  if ((u & 0x7fffffffu) > 0x7f800000u) return 0x7fc0;
  u += 0x7fffu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

// Upload `n` consecutive fp32 values as the model's storage type.
int upload(asr_spec* h, void* dst, const float* src, size_t n) {
  if (!h->bf16) {
    CK(cudaMemcpy(dst, src, n * 4, cudaMemcpyHostToDevice));
    return 0;
  }
  std::vector<uint16_t> tmp(n);
  for (size_t i = 0; i < n; ++i) tmp[i] = f2bf_host(src[i]);
  CK(cudaMemcpy(dst, tmp.data(), n * 2, cudaMemcpyHostToDevice));
  return 0;
}
int upload_f32(asr_spec* h, float* dst, const float* src, size_t n) {
  CK(cudaMemcpy(dst, src, n * 4, cudaMemcpyHostToDevice));
  return 0;
}

const CUtensorMap* bmap(asr_spec* h, int id, const void* buf, int rows, int cols, int bn) {
  auto key = std::make_pair(id, bn);
  auto it = h->bmaps.find(key);
  if (it != h->bmaps.end()) return &it->second;
  CUtensorMap m;
  if (!make_tmap_bf16(&m, buf, rows, cols, bn)) return nullptr;
  return &(h->bmaps[key] = m);
}

const CUtensorMap* xmap(asr_spec* h, int bn) {
  auto it = h->xmaps.find(bn);
  if (it != h->xmaps.end()) return &it->second;
  CUtensorMap m;
  if (!make_tmap_f32(&m, h->x, h->R_pad, h->d, 128, bn)) return nullptr;
  return &(h->xmaps[bn] = m);
}

// The next launch's slot of the per-CTA phase trace, or null (tracing off or the buffer full).
unsigned long long* trace_slot(asr_spec* h) {
  if (!h->fr_trace_on || h->fr_trace_n >= 6 * h->L) return nullptr;
  return h->fr_trace + (size_t)(h->fr_trace_n++) * FR_TRACE_CTAS * FR_TRACE_PHASES;
}

// One projection over the verify rows: out-features m (weights = A), rows n (activations = B).
int gemm_rows(asr_spec* h, const void* W, const CUtensorMap* mW, int M, int K, const void* X, int x_id, int N,
              int mode, const Epi& epi_in) {
  Epi epi = epi_in;
  epi.M = M;
  epi.N = N;
  epi.status = h->status;
  if (mode == EPI_QKV) epi.b_max = h->Bmax;
  if (mode != EPI_ARGMAX && !epi.trace) epi.trace = trace_slot(h);
  const int cls = mode == EPI_QKV     ? ASR_PROF_QKV
                  : mode == EPI_RESID ? ASR_PROF_RESID
                  : mode == EPI_Q     ? ASR_PROF_QUERY
                  : mode == EPI_GELU  ? ASR_PROF_UP
                                      : ASR_PROF_LMHEAD;
  Prof p(h, cls, 1);
  if (!h->bf16) {
    launch_gemm_simt(W, 0, X, 0, M, N, K, mode, epi, h->st);
    return 0;
  }
  WideGemm w{};
  if (N > 64 && h->use_wide && wide_pick(M, N, K, mode, h->n_sms, &w.bn, &w.split) &&
      (mode != EPI_RESID || epi.x == h->x)) {
    const CUtensorMap* mb = bmap(h, x_id, X, h->R_pad, K, w.bn);
    const CUtensorMap* mx = mode == EPI_RESID ? xmap(h, w.bn) : mW;
    if (!mb || !mx) return fail(h, ASR_E_CUDA, "tensor map encode failed");
    w.mapA = *mW;
    w.mapB = *mb;
    w.mapX = *mx;
    w.M = M;
    w.N = N;
    w.K = K;
    w.pdl = h->use_pdl;
    w.stages = h->wide_stages;
    Tl t(h, ASR_TL_GEMM + mode + (epi.ln_part ? ASR_TL_LN_FUSED : 0));
    epi.tl = h->tl_cur;
    launch_gemm_wide(w, mode, epi, h->status, h->st);
    if (epi.xg) {   // every tile wrote the statistics of its 128-feature slice
      h->ln_c = 128;
      h->ln_S = M / 128;
    }
    return 0;
  }
  TcGemm g{};
  g.mapA = *mW;
  // Few rows (batch 1): one narrow N tile and K split across the CTAs of a
  // cluster so that every SM streams weights.  Many rows: 64-wide N tiles
  // (two CTAs per SM; measured best at batch 64 against 128 and 256), K split
  // in a cluster while the grid stays within one wave and every split keeps at
  // least four k-blocks.  Split factors are powers of two up to 16.
  // the LM head (argmax epilogue, 406 weight tiles) takes 128-wide row tiles
  // for many rows: its weights are read half as often (measured 95 vs 116 us
  // at 448 rows)
  g.bn = N <= 64 ? tc_pick_bn(N) : (mode == EPI_ARGMAX ? 128 : h->wide_bn);
  const CUtensorMap* mb = bmap(h, x_id, X, h->R_pad, K, g.bn);
  if (!mb) return fail(h, ASR_E_CUDA, "tensor map encode failed");
  g.mapB = *mb;
  g.M = M;
  g.N = N;
  g.K = K;
  const int tiles = ((M + 127) / 128) * ((N + g.bn - 1) / g.bn);
  const int nkb = K / 64;
  const int target = N <= 64 ? h->few_target : h->wide_target;
  g.splits = 1;
  if (mode != EPI_ARGMAX && mode != EPI_F32)
    while (g.splits < 16 && tiles * g.splits * 2 <= target && g.splits * 2 <= (N <= 64 ? nkb : nkb / 4))
      g.splits *= 2;
  g.cluster = g.splits > 1;
  g.pdl = h->use_pdl;
  g.ws = h->ws;
  g.tickets = h->tickets;
  Tl t(h, ASR_TL_GEMM + mode + (epi.ln_part ? ASR_TL_LN_FUSED : 0));
  epi.tl = h->tl_cur;
  launch_gemm_tc(g, mode, epi, h->status, h->st);
  if (epi.xg) {   // the slices the residual epilogue wrote statistics for
    h->ln_c = g.splits > 1 ? 128 / g.splits : 128;
    h->ln_S = M / h->ln_c;
  }
  return 0;
}

enum BufId { BUF_XN = 1, BUF_ATT = 2, BUF_H = 3, BUF_XF = 4, BUF_DIN = 5, BUF_DXN = 6, BUF_DATT = 7, BUF_DH = 8,
             BUF_DXF = 9 };

// Folded LayerNorm of a consumer GEMM: B = xn (bf16(g * x), written by the
// producer of x) and the producer's slice statistics.
void fold_consumer(asr_spec* h, Epi& e, const float* c1, const float* c2) {
  e.ln_part = h->ln_part;
  e.ln_S = h->ln_S;
  e.ln_c = h->ln_c;
  e.ln_stride = h->R_pad;
  e.ln_c1 = c1;
  e.ln_c2 = c2;
}

// A projection whose input is LayerNorm(x).  Folded (bf16): no LayerNorm
// launch; the GEMM reads xn and corrects its accumulators.  Otherwise a
// LayerNorm kernel writes `ln_out` and the GEMM loads it by TMA.
int gemm_rows_ln(asr_spec* h, const void* W, const CUtensorMap* mW, int M, int K, const float* g, const float* b,
                 const float* c1, const float* c2, void* ln_out, int ln_out_id, int N, int mode, const Epi& epi_in) {
  Epi e = epi_in;
  if (h->ln_fold) {
    fold_consumer(h, e, c1, c2);
    return gemm_rows(h, W, mW, M, K, h->xn, BUF_XN, N, mode, e);
  }
  {
    Prof p(h, ASR_PROF_LAYERNORM, 1);
    Tl t(h, ASR_TL_LAYERNORM);
    launch_layernorm(h->x, g, b, ln_out, h->bf16, h->plan.n_rows, N, K, h->st, h->use_pdl, h->tl_cur);
  }
  return gemm_rows(h, W, mW, M, K, ln_out, ln_out_id, N, mode, e);
}

// The decoder layers over the rows laid out by the last plan kernel.
// CTAs per (utterance, head) for the tensor-core attention: few utterances
// (batch 1) split the keys over a cluster of up to 8 CTAs.
int attn_splits_for(asr_spec* h, int t_alloc) {
  const int nc_max = (t_alloc + 127) / 128;
  int S = 1;
  // split until every SM has two CTAs (the ring of each keeps 96 KB in flight)
  while (S < 8 && S * 2 <= nc_max && h->B * h->H * S < 2 * NUM_SMS_TARGET) S *= 2;
  return S;
}

void attention(asr_spec* h, AttnArgs& a, bool self_attn, int layer) {
  if (!h->bf16) {
    launch_attention(a, h->st);
    return;
  }
  a.splits = attn_splits_for(h, a.t_alloc);
  const int ci = 0;   // 128-row boxes
  if (self_attn) {
    a.kmap = &h->m_kself[ci];
    a.vmap = &h->m_vself[ci];
    a.k_row0 = a.v_row0 = (long long)layer * h->Bmax * h->H * h->maxpos;
  } else {
    a.kmap = a.vmap = &h->m_xkv[ci];
    a.k_row0 = (long long)layer * 2 * h->Bmax * h->H * h->Tmax;
    a.v_row0 = a.k_row0 + (long long)h->Bmax * h->H * h->Tmax;
  }
  a.tickets = h->attn_tickets;
  a.pdl = h->use_pdl;
  Tl t(h, self_attn ? ASR_TL_ATTN_SELF : ASR_TL_ATTN_CROSS);
  a.tl = h->tl_cur;
  launch_attention_tc(a, h->status, h->st);
  a.tl = nullptr;
}

// With a draft: the residual stream after a tapped layer into its column of
// the tap rows [R][4][d] (the draft's inputs, App. "Draft architecture").
int tap_copy(asr_spec* h, int l, int rows) {
  if (!h->has_draft) return 0;
  for (int i = 0; i < 4; ++i)
    if (h->taps[i] == l)
      CK(cudaMemcpy2DAsync(h->d_taps + (size_t)i * h->d, 4 * (size_t)h->d * 4, h->x, (size_t)h->d * 4,
                           (size_t)h->d * 4, rows, cudaMemcpyDeviceToDevice, h->st));
  return 0;
}

int run_layers(asr_spec* h, int N) {
  const int rows_max = N / std::max(h->B, 1);
  const int d = h->d;
  Epi base{};
  base.n_valid = h->plan.n_rows;
  base.d = d;
  base.row_b = h->plan.row_b;
  base.row_pos = h->plan.row_pos;
  base.kv_bf16 = h->bf16;
  base.act_bf16 = h->bf16;
  base.max_pos = h->maxpos;
  base.n_heads = h->H;
  const size_t self_layer = (size_t)h->Bmax * h->H * h->maxpos * 64 * h->es;
  const size_t cross_half = (size_t)h->Bmax * h->H * h->Tmax * 64 * h->es;
  {
    Prof p(h, ASR_PROF_OTHER, 1);
    Tl t(h, ASR_TL_EMBED);
    if (h->ln_fold) {   // the first LayerNorm's operand and statistics (one slice of d features)
      launch_embed(h->w_tok, h->w_pos, h->bf16, h->plan, N, d, h->x, h->st, h->use_pdl, h->tl_cur,
                   static_cast<__nv_bfloat16*>(h->xn), h->lw[0].ln1g, h->ln_part, h->V, h->maxpos, h->status);
      h->ln_S = 1;
      h->ln_c = d;
    } else {
      launch_embed(h->w_tok, h->w_pos, h->bf16, h->plan, N, d, h->x, h->st, h->use_pdl, h->tl_cur, nullptr, nullptr,
                   nullptr, h->V, h->maxpos, h->status);
    }
  }
  // a residual projection that also produces the next LayerNorm's folded operand
  auto producer = [&](Epi& e, const float* next_gain) {
    if (!h->ln_fold) return;
    e.xg = static_cast<__nv_bfloat16*>(h->xn);
    e.xg_gain = next_gain;
    e.st_part = h->ln_part;
    e.st_stride = h->R_pad;
  };
  for (int l = 0; l < h->L; ++l) {
    LayerW& w = h->lw[l];
    char* ks = static_cast<char*>(h->kself) + l * self_layer;
    char* vs = static_cast<char*>(h->vself) + l * self_layer;
    char* kx = static_cast<char*>(h->xkv) + (size_t)l * 2 * cross_half;
    char* vx = kx + cross_half;
    // self-attention block
    Epi e = base;
    e.bias = w.bqkv;
    e.out_f32 = h->q;
    e.kcache = ks;
    e.vcache = vs;
    if (int rc = gemm_rows_ln(h, w.wqkv, &w.m_wqkv, 3 * d, d, w.ln1g, w.ln1b, w.c1_qkv, w.c2_qkv, h->xn, BUF_XN, N,
                              EPI_QKV, e))
      return rc;
    AttnArgs a{};
    a.status = h->status;
    a.q = h->q;
    a.kc = ks;
    a.vc = vs;
    a.kv_bf16 = h->bf16;
    a.t_alloc = h->maxpos;
    a.causal = 1;
    a.enc_len = h->enc_len;
    a.kv_len = h->kv_len;
    a.plan = h->plan;
    a.B = h->B;
    a.H = h->H;
    a.d = d;
    a.k1 = h->kmax + 1;
    a.chunk = attn_chunk_len(h->bf16);
    a.n_chunks = (h->maxpos + a.chunk - 1) / a.chunk;
    a.part = h->part;
    a.out = h->att;
    a.out_bf16 = h->bf16;
    a.ml_out = nullptr;
    a.rows_max = rows_max;
    a.tree = h->cur_tree;
    {
      Prof p(h, ASR_PROF_SELF, h->bf16 ? 1 : 2);
      attention(h, a, true, l);
    }
    a.tree = false;
    e = base;
    e.bias = w.bo;
    e.x = h->x;
    producer(e, w.ln2g);
    if (int rc = gemm_rows(h, w.wo, &w.m_wo, d, d, h->att, BUF_ATT, N, EPI_RESID, e)) return rc;
    // cross-attention block
    float* qc = (l == h->anchor) ? h->q_anchor : h->q;
    e = base;
    e.bias = w.bcq;
    e.out_f32 = qc;
    if (int rc = gemm_rows_ln(h, w.wcq, &w.m_wcq, d, d, w.ln2g, w.ln2b, w.c1_cq, w.c2_cq, h->xn, BUF_XN, N, EPI_Q, e))
      return rc;
    a.q = qc;
    a.kc = kx;
    a.vc = vx;
    a.t_alloc = h->Tmax;
    a.causal = 0;
    a.n_chunks = (h->Tmax + a.chunk - 1) / a.chunk;
    a.ml_out = (l == h->anchor) ? h->ml : nullptr;
    {
      Prof p(h, ASR_PROF_CROSS, h->bf16 ? 1 : 2);
      attention(h, a, false, l);
    }
    e = base;
    e.bias = w.bco;
    e.x = h->x;
    producer(e, w.ln3g);
    if (int rc = gemm_rows(h, w.wco, &w.m_wco, d, d, h->att, BUF_ATT, N, EPI_RESID, e)) return rc;
    // MLP block
    e = base;
    e.bias = w.b1;
    e.act = h->hbuf;
    if (int rc = gemm_rows_ln(h, w.w1, &w.m_w1, h->F, d, w.ln3g, w.ln3b, w.c1_fc1, w.c2_fc1, h->xn, BUF_XN, N, EPI_GELU,
                              e))
      return rc;
    e = base;
    e.bias = w.b2;
    e.x = h->x;
    producer(e, l + 1 < h->L ? h->lw[l + 1].ln1g : h->lnf_g);
    if (int rc = gemm_rows(h, w.w2, &w.m_w2, d, h->F, h->hbuf, BUF_H, N, EPI_RESID, e)) return rc;
    if (int rc = tap_copy(h, l, N)) return rc;
  }
  return 0;
}

// The decoder layers of a step with at most VF_ROWS rows (csrc/fewrow.cu):
// six launches per layer.
int run_layers_few(asr_spec* h) {
  const int d = h->d, F = h->F, H = h->H, C = h->fr_C, N = h->B * (h->kmax + 1);
  const int nt_o = d / 8, nt_f = F / 8, KS = F / d;
  const int g_o = std::min(nt_o, h->fr_sms), g_f = std::min(nt_f, h->fr_sms), g_d = h->fr_gd;
  const size_t self_layer = (size_t)h->Bmax * H * h->maxpos * 64;
  {
    Prof p(h, ASR_PROF_OTHER, 1);
    Tl t(h, ASR_TL_EMBED);
    launch_embed(h->w_tok, h->w_pos, h->bf16, h->plan, std::min(N, VF_ROWS), d, h->x, h->st, h->use_pdl, h->tl_cur,
                 nullptr, nullptr, nullptr, h->V, h->maxpos, h->status);
  }
  auto bf = [](void* p) { return static_cast<const __nv_bfloat16*>(p); };
  // the packed weights of the layers' six launches in launch order, for the
  // L2 prefetch of a later launch's weights
  auto later = [&](int l, int slot, const void** pf, uint32_t* bytes) {
    const int g = 6 * l + slot + h->fr_prefetch;
    *pf = nullptr;
    *bytes = 0;
    if (h->fr_prefetch <= 0 || g >= 6 * h->L) return;
    const LayerW& n = h->lw[g / 6];
    const uint32_t dd = (uint32_t)d * d * 2, fd = (uint32_t)F * d * 2;
    const void* p[6] = {n.p_qkv, n.p_wo, n.p_wcq, n.p_wco, n.p_w1, n.p_w2};
    const uint32_t b[6] = {3 * dd, dd, dd, dd, fd, fd};
    *pf = p[g % 6];
    *bytes = b[g % 6];
  };
  for (int l = 0; l < h->L; ++l) {
    LayerW& w = h->lw[l];
    FrHead hd{};
    hd.x = h->x;
    hd.d = d;
    hd.H = H;
    hd.C = C;
    hd.B = h->B;
    hd.max_pos = h->maxpos;
    hd.plan = h->plan;
    hd.kv_len = h->kv_len;
    hd.enc_len = h->enc_len;
    hd.att = static_cast<__nv_bfloat16*>(h->att);
    hd.status = h->status;
    // LayerNorm 1 -> QKV -> self-attention
    FrHead hs = hd;
    hs.W = bf(w.p_qkv);
    hs.bias = w.bqkv;
    hs.ln_g = w.ln1g;
    hs.ln_b = w.ln1b;
    hs.tiles_max = (24 + C - 1) / C;
    hs.mrg_slots = (h->maxpos + 127) / 128;
    hs.ks = static_cast<__nv_bfloat16*>(h->kself) + l * self_layer;
    hs.vs = static_cast<__nv_bfloat16*>(h->vself) + l * self_layer;
    hs.row0 = (long long)l * h->Bmax * H * h->maxpos;
    hs.t_alloc = h->maxpos;
    later(l, 0, &hs.pf, &hs.pf_bytes);
    {
      Prof p(h, ASR_PROF_QKV_SELF, 1);
      Tl t(h, ASR_TL_QKV_SELF);
      hs.tl = h->tl_cur;
      hs.trace = trace_slot(h);
      CK(launch_fr_self(&h->m_kself[0], &h->m_vself[0], hs, h->st, h->use_pdl));
    }
    FrGemv g{};
    g.n_rows = h->plan.n_rows;
    g.status = h->status;
    g.x = h->x;
    g.x_out = h->x;
    // self-attention output projection + residual
    FrGemv go = g;
    go.W = bf(w.p_wo);
    go.bias = w.bo;
    go.N = d;
    go.K = d;
    go.tiles_max = (nt_o + g_o - 1) / g_o;
    go.a = static_cast<const __nv_bfloat16*>(h->att);
    later(l, 1, &go.pf, &go.pf_bytes);
    {
      Prof p(h, ASR_PROF_RESID, 1);
      Tl t(h, ASR_TL_GEMM + EPI_RESID);
      go.tl = h->tl_cur;
      go.trace = trace_slot(h);
      CK(launch_fr_gemv(go, FR_RESID, 1, g_o, d, h->st, h->use_pdl));
    }
    // LayerNorm 2 -> cross query -> cross-attention
    FrHead hc = hd;
    hc.W = bf(w.p_wcq);
    hc.bias = w.bcq;
    hc.ln_g = w.ln2g;
    hc.ln_b = w.ln2b;
    hc.tiles_max = (8 + C - 1) / C;
    hc.mrg_slots = C;
    hc.row0 = (long long)l * 2 * h->Bmax * H * h->Tmax;
    hc.vofs = (long long)h->Bmax * H * h->Tmax;
    hc.t_alloc = h->Tmax;
    hc.q_anchor = l == h->anchor ? h->q_anchor : nullptr;
    hc.ml = l == h->anchor ? h->ml : nullptr;
    later(l, 2, &hc.pf, &hc.pf_bytes);
    {
      Prof p(h, ASR_PROF_QUERY_CROSS, 1);
      Tl t(h, ASR_TL_QUERY_CROSS);
      hc.tl = h->tl_cur;
      hc.trace = trace_slot(h);
      CK(launch_fr_cross(&h->m_xkv[0], hc, h->st, h->use_pdl));
    }
    // cross-attention output projection + residual
    FrGemv gc = go;
    gc.W = bf(w.p_wco);
    gc.bias = w.bco;
    later(l, 3, &gc.pf, &gc.pf_bytes);
    {
      Prof p(h, ASR_PROF_RESID, 1);
      Tl t(h, ASR_TL_GEMM + EPI_RESID);
      gc.tl = h->tl_cur;
      gc.trace = trace_slot(h);
      CK(launch_fr_gemv(gc, FR_RESID, 1, g_o, d, h->st, h->use_pdl));
    }
    // LayerNorm 3 -> MLP up + GELU
    FrGemv gu = g;
    gu.W = bf(w.p_w1);
    gu.bias = w.b1;
    gu.N = F;
    gu.K = d;
    gu.tiles_max = (nt_f + g_f - 1) / g_f;
    gu.ln_g = w.ln3g;
    gu.ln_b = w.ln3b;
    gu.h_out = static_cast<__nv_bfloat16*>(h->hbuf);
    later(l, 4, &gu.pf, &gu.pf_bytes);
    {
      Prof p(h, ASR_PROF_UP, 1);
      Tl t(h, ASR_TL_GEMM + EPI_GELU);
      gu.tl = h->tl_cur;
      gu.trace = trace_slot(h);
      CK(launch_fr_gemv(gu, FR_GELU, 1, g_f, d, h->st, h->use_pdl));
    }
    // MLP down + residual (K split over a cluster of F / d CTAs)
    FrGemv gd = g;
    gd.W = bf(w.p_w2);
    gd.bias = w.b2;
    gd.N = d;
    gd.K = F;
    gd.tiles_max = (nt_o + g_d - 1) / g_d;
    gd.a = static_cast<const __nv_bfloat16*>(h->hbuf);
    later(l, 5, &gd.pf, &gd.pf_bytes);
    {
      Prof p(h, ASR_PROF_RESID, 1);
      Tl t(h, ASR_TL_GEMM + EPI_RESID);
      gd.tl = h->tl_cur;
      gd.trace = trace_slot(h);
      CK(launch_fr_gemv(gd, FR_RESID, KS, g_d, d, h->st, h->use_pdl));
    }
    if (int rc = tap_copy(h, l, VF_ROWS)) return rc;
  }
  return 0;
}

// One pass of the draft's block over the rows of `plan` (at most `rows`):
// input combination w_in [f_1..f_4] + b_in + embeddings, LayerNorm ->
// self-attention over the draft's cache (K/V of the rows appended) -> out
// projection; LayerNorm -> cross-attention over the draft's encoder K/V
// (window per row) -> out projection; LayerNorm -> MLP (2 d, GELU); final
// LayerNorm -> the target's tied LM head with argmax (when `lm`).
int draft_block(asr_spec* h, const RowPlan& plan, int rows, bool lm) {
  const int d = h->d, F2 = 2 * h->d;
  DraftW& w = h->dw;
  Epi base{};
  base.n_valid = plan.n_rows;
  base.d = d;
  base.row_b = plan.row_b;
  base.row_pos = plan.row_pos;
  base.kv_bf16 = 1;
  base.act_bf16 = 1;
  base.max_pos = h->maxpos;
  base.n_heads = h->H;
  DraftArgs A{};
  A.B = h->B;
  A.d = d;
  A.vocab = h->V;
  A.max_pos = h->maxpos;
  A.r_max = h->R_pad;
  A.status = h->status;
  A.plan = plan;
  Epi e = base;
  e.bias = w.b_in;
  e.out_f32 = h->d_x;
  if (int rc = gemm_rows(h, w.w_in, &w.m_in, d, 4 * d, h->d_xin, BUF_DIN, rows, EPI_Q, e)) return rc;
  launch_draft_embed(A, rows, h->w_tok, h->w_pos, h->d_x, h->st);
  auto ln = [&](const float* g, const float* b, void* y) {
    launch_layernorm(h->d_x, g, b, y, 1, plan.n_rows, rows, d, h->st, false, nullptr);
  };
  DraftAttn at{};
  at.q = h->d_q;
  at.B = h->B;
  at.H = h->H;
  at.d = d;
  at.plan = plan;
  at.row_lo = h->d_row_lo;
  at.row_hi = h->d_row_hi;
  at.out = static_cast<__nv_bfloat16*>(h->d_att);
  at.status = h->status;
  // self-attention block
  ln(w.ln1g, w.ln1b, h->d_xn);
  e = base;
  e.bias = w.bqkv;
  e.out_f32 = h->d_q;
  e.kcache = h->d_ks;
  e.vcache = h->d_vs;
  if (int rc = gemm_rows(h, w.wqkv, &w.m_qkv, 3 * d, d, h->d_xn, BUF_DXN, rows, EPI_QKV, e)) return rc;
  at.kc = static_cast<const __nv_bfloat16*>(h->d_ks);
  at.vc = static_cast<const __nv_bfloat16*>(h->d_vs);
  at.t_alloc = h->maxpos;
  at.causal = 1;
  launch_draft_attn(at, h->st);
  e = base;
  e.bias = w.bo;
  e.x = h->d_x;
  if (int rc = gemm_rows(h, w.wo, &w.m_wo, d, d, h->d_att, BUF_DATT, rows, EPI_RESID, e)) return rc;
  // cross-attention block
  ln(w.ln2g, w.ln2b, h->d_xn);
  e = base;
  e.bias = w.bcq;
  e.out_f32 = h->d_q;
  if (int rc = gemm_rows(h, w.wcq, &w.m_wcq, d, d, h->d_xn, BUF_DXN, rows, EPI_Q, e)) return rc;
  const size_t half = (size_t)h->Bmax * h->H * h->Tmax * 64;
  at.kc = static_cast<const __nv_bfloat16*>(h->d_xkv);
  at.vc = static_cast<const __nv_bfloat16*>(h->d_xkv) + half;
  at.t_alloc = h->Tmax;
  at.causal = 0;
  launch_draft_attn(at, h->st);
  e = base;
  e.bias = w.bco;
  e.x = h->d_x;
  if (int rc = gemm_rows(h, w.wco, &w.m_wco, d, d, h->d_att, BUF_DATT, rows, EPI_RESID, e)) return rc;
  // MLP block
  ln(w.ln3g, w.ln3b, h->d_xn);
  e = base;
  e.bias = w.b1;
  e.act = h->d_h;
  if (int rc = gemm_rows(h, w.w1, &w.m_w1, F2, d, h->d_xn, BUF_DXN, rows, EPI_GELU, e)) return rc;
  e = base;
  e.bias = w.b2;
  e.x = h->d_x;
  if (int rc = gemm_rows(h, w.w2, &w.m_w2, d, F2, h->d_h, BUF_DH, rows, EPI_RESID, e)) return rc;
  if (!lm) return 0;
  ln(w.lnfg, w.lnfb, h->d_xf);
  e = Epi{};
  e.n_valid = plan.n_rows;
  e.row_key = h->d_row_key;
  e.d = d;
  if (h->d_threshold <= 0.f)
    return gemm_rows(h, h->w_tok, &h->m_tok, h->V, d, h->d_xf, BUF_DXF, rows, EPI_ARGMAX, e);
  // confidence threshold: the logits, then per row the argmax and its probability
  e.out_f32 = h->d_logits;
  e.ld = h->V;
  if (int rc = gemm_rows(h, h->w_tok, &h->m_tok, h->V, d, h->d_xf, BUF_DXF, rows, EPI_F32, e)) return rc;
  launch_draft_softmax(h->d_logits, h->V, plan.n_rows, rows, h->d_row_key, h->d_row_p, h->st);
  return 0;
}

bool dims_ok(const asr_model_dims& m) {
  return m.n_layers >= 1 && m.d_model >= 64 && m.d_model % 64 == 0 && m.d_model <= 2048 &&
         m.n_heads * 64 == m.d_model && m.d_ffn >= 64 && m.d_ffn % 64 == 0 && m.vocab >= 2 && m.max_pos >= 2 &&
         m.max_batch >= 1 && m.max_batch <= 1024 && m.max_draft >= 0 && m.max_draft <= 31 && m.max_enc >= 1 &&
         (m.dtype == 0 || m.dtype == 1) && m.anchor_layer >= -1 && m.anchor_layer < m.n_layers;
}

int copy_in(asr_spec* h, int* dst, const int32_t* src, size_t n) {
  CK(cudaMemcpyAsync(dst, src, n * 4, h->host_io ? cudaMemcpyHostToDevice : cudaMemcpyDeviceToDevice, h->st));
  return 0;
}
int copy_out(asr_spec* h, int32_t* dst, const int* src, size_t n) {
  CK(cudaMemcpyAsync(dst, src, n * 4, h->host_io ? cudaMemcpyDeviceToHost : cudaMemcpyDeviceToDevice, h->st));
  return 0;
}

// The verify body on the handle's stream: rows, decoder layers, LM head with
// fused argmax, acceptance and commit, anchor readout.  Reads the internal
// draft/lens buffers and writes the internal output block.
int enqueue_verify(asr_spec* h, int k) {
  const int B = h->B;
  h->fr_trace_n = 0;   // the phase trace (when on) holds this call's launches
  {
    Prof p(h, ASR_PROF_OTHER, 1);
    Tl t(h, ASR_TL_PLAN);
    TrafficArgs tr{h->counters, h->enc_len, h->L, h->d, (int)h->es};
    launch_plan_verify(h->draft_buf, h->lens_buf, k, B, h->V, h->maxpos, h->kv_len, h->pending, h->ready, h->plan,
                       h->row_key, h->status, tr, h->st, h->tl_cur, h->cur_tree ? h->parent_buf : nullptr);
  }
  const int N = B * (k + 1);
  h->last_fused = h->fr_C > 0 && h->use_fewrow && N <= VF_ROWS && B <= VF_ROWS && !h->cur_tree;
  if (h->last_fused) {   // few rows: six launches per layer, then LayerNorm + LM head
    if (int rc = run_layers_few(h)) return rc;
    {
      Prof p(h, ASR_PROF_LAYERNORM, 1);
      Tl t(h, ASR_TL_LAYERNORM);
      launch_layernorm(h->x, h->lnf_g, h->lnf_b, h->xf, h->bf16, h->plan.n_rows, N, h->d, h->st, h->use_pdl,
                       h->tl_cur);
    }
    Epi e{};
    e.n_valid = h->plan.n_rows;
    e.row_key = h->row_key;
    e.d = h->d;
    if (int rc = gemm_rows(h, h->w_tok, &h->m_tok, h->V, h->d, h->xf, BUF_XF, N, EPI_ARGMAX, e)) return rc;
  } else {
    if (int rc = run_layers(h, N)) return rc;
    Epi e{};
    e.n_valid = h->plan.n_rows;
    e.row_key = h->row_key;
    e.d = h->d;
    if (int rc = gemm_rows_ln(h, h->w_tok, &h->m_tok, h->V, h->d, h->lnf_g, h->lnf_b, h->c1_lm, h->c2_lm, h->xf,
                              BUF_XF, N, EPI_ARGMAX, e))
      return rc;
  }
  Prof p(h, ASR_PROF_OTHER, 1);
  AcceptAnchorArgs A{};
  A.draft = h->draft_buf;
  A.k = k;
  A.B = B;
  A.H = h->H;
  A.d = h->d;
  A.t_alloc = h->Tmax;
  A.kv_bf16 = h->bf16;
  A.plan = h->plan;
  A.row_key = h->row_key;
  A.kv_len = h->kv_len;
  A.pending = h->pending;
  A.accepted = h->out4;
  A.bonus = h->out4 + h->Bmax;
  A.kv_len_out = h->out4 + 2 * h->Bmax;
  A.anchor_out = h->out4 + 3 * h->Bmax;
  A.restart = h->out4 + 4 * h->Bmax;
  A.profile = h->anchor_prof;
  A.q_anchor = h->q_anchor;
  A.ml = h->ml;
  const size_t cross_half = (size_t)h->Bmax * h->H * h->Tmax * 64 * h->es;
  A.kc = static_cast<const char*>(h->xkv) + (size_t)h->anchor * 2 * cross_half;
  A.enc_len = h->enc_len;
  A.frame_key = h->frame_key;
  A.tickets = reinterpret_cast<int*>(h->frame_key + h->Bmax);
  A.status = h->status;
  A.pdl = h->use_pdl;
  if (h->cur_tree) {
    A.parent = h->parent_buf;
    A.path = h->path_buf;
  }
  {
    Tl t(h, ASR_TL_ACCEPT);
    A.tl = h->tl_cur;
    launch_accept_anchor(A, h->st);
  }
  if (h->cur_tree) {   // the accepted path's K/V to consecutive positions
    Prof p2(h, ASR_PROF_OTHER, 1);
    launch_tree_commit(h->path_buf, k, h->out4, h->kv_len, B, h->L, h->H, h->maxpos, h->Bmax, h->kself, h->vself,
                       (int)h->es, h->status, h->st);
  }
  return 0;
}

}  // namespace

extern "C" {

int asr_spec_create(const asr_model_dims* dims, const asr_weights* weights, void* stream, asr_spec_handle* out) {
  if (!dims || !weights || !weights->blob || !out) return ASR_E_INVAL;
  *out = nullptr;
  if (!dims_ok(*dims)) return ASR_E_INVAL;
  asr_spec* h = new asr_spec();
  h->dims = *dims;
  h->L = dims->n_layers;
  h->d = dims->d_model;
  h->H = dims->n_heads;
  h->F = dims->d_ffn;
  h->V = dims->vocab;
  h->maxpos = dims->max_pos;
  h->Bmax = dims->max_batch;
  h->kmax = dims->max_draft;
  h->Tmax = dims->max_enc;
  h->anchor = dims->anchor_layer >= 0 ? dims->anchor_layer : (3 * h->L) / 4;
  h->bf16 = dims->dtype == 1;
  {
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&h->n_sms, cudaDevAttrMultiProcessorCount, dev);
  }
  if (const char* e = std::getenv("ASRSPEC_WIDE")) h->use_wide = std::atoi(e) != 0;
  if (const char* e = std::getenv("ASRSPEC_FR_PREFETCH")) h->fr_prefetch = std::max(0, std::atoi(e));
  if (const char* e = std::getenv("ASRSPEC_WIDE_STAGES")) h->wide_stages = std::max(0, std::atoi(e));
  {   // bounds-check mode: process-wide (each kernel module's constant), set by every create
    const char* e = std::getenv("ASRSPEC_CHECK");
    const int on = e && std::atoi(e) != 0;
    set_check_gemm_tc(on);
    set_check_gemm_simt(on);
    set_check_gemm_wide(on);
    set_check_rows(on);
    set_check_attention(on);
    set_check_attention_tc(on);
    set_check_fewrow(on);
    set_check_draft(on);
  }
  if (const char* e = std::getenv("ASRSPEC_PDL")) h->use_pdl = std::atoi(e) != 0;
  if (const char* e = std::getenv("ASRSPEC_WIDE_BN")) {
    const int v = std::atoi(e);
    if (v == 64 || v == 128 || v == 192 || v == 224 || v == 256) h->wide_bn = v;
  }
  if (const char* e = std::getenv("ASRSPEC_WIDE_TARGET")) h->wide_target = std::max(1, std::atoi(e));
  if (const char* e = std::getenv("ASRSPEC_FEW_TARGET")) h->few_target = std::max(1, std::atoi(e));
  if (const char* e = std::getenv("ASRSPEC_ENC_BN")) {
    const int v = std::atoi(e);
    if (v == 64 || v == 128 || v == 256) h->enc_bn = v;
  }
  if (const char* e = std::getenv("ASRSPEC_ENC_GROUP")) h->enc_group = std::max(0, std::atoi(e));
  h->es = h->bf16 ? 2 : 4;
  h->ln_fold = h->bf16 && h->d % 128 == 0 && h->wide_bn <= 64;
  if (const char* e = std::getenv("ASRSPEC_LN_FOLD")) h->ln_fold = h->ln_fold && std::atoi(e) != 0;
  h->st = static_cast<cudaStream_t>(stream);
  if (!h->st) {
    // A blocking stream of our own: ordered with the legacy default stream,
    // and capturable into CUDA graphs (the legacy stream itself is not).
    if (cudaStreamCreate(&h->st) != cudaSuccess) {
      delete h;
      return ASR_E_CUDA;
    }
    h->own_stream = true;
  }
  const int d = h->d, F = h->F, L = h->L;
  const size_t per_layer = 8 * (size_t)d * d + 13 * (size_t)d + 2 * (size_t)F * d + F;
  const size_t expect = (size_t)h->V * d + (size_t)h->maxpos * d + L * per_layer + 2 * (size_t)d;
  if (weights->n_floats != expect) {
    if (h->own_stream) cudaStreamDestroy(h->st);
    delete h;
    return ASR_E_INVAL;
  }
  int rc = 0;
  auto finish = [&](int code) {
    if (code) asr_spec_destroy(h);
    else *out = h;
    return code;
  };
  const float* src = weights->blob;
  size_t off = 0;
  auto take = [&](size_t n) {
    const float* p = src + off;
    off += n;
    return p;
  };
  const size_t es = h->es;
  if ((rc = dalloc(h, &h->w_tok, (size_t)h->V * d * es))) return finish(rc);
  if ((rc = upload(h, h->w_tok, take((size_t)h->V * d), (size_t)h->V * d))) return finish(rc);
  if ((rc = dalloc(h, &h->w_pos, (size_t)h->maxpos * d * es))) return finish(rc);
  if ((rc = upload(h, h->w_pos, take((size_t)h->maxpos * d), (size_t)h->maxpos * d))) return finish(rc);
  if ((rc = dalloc(h, &h->w_cross, (size_t)L * 2 * d * d * es))) return finish(rc);
  if ((rc = dalloc(h, &h->b_cross, (size_t)L * 2 * d * 4))) return finish(rc);
  h->lw.resize(L);
  std::vector<float> tmp;
  for (int l = 0; l < L; ++l) {
    LayerW& w = h->lw[l];
    auto vec = [&](float** dst, size_t n, const float* s) {
      int r = dalloc(h, dst, n * 4);
      if (!r) r = upload_f32(h, *dst, s, n);
      return r;
    };
    auto mat = [&](void** dst, size_t n, const float* s) {
      int r = dalloc(h, dst, n * es);
      if (!r) r = upload(h, *dst, s, n);
      return r;
    };
    const float* ln1g = take(d);
    const float* ln1b = take(d);
    const float* wq = take((size_t)d * d);
    const float* bq = take(d);
    const float* wk = take((size_t)d * d);
    const float* wv = take((size_t)d * d);
    const float* bv = take(d);
    const float* wo = take((size_t)d * d);
    const float* bo = take(d);
    const float* ln2g = take(d);
    const float* ln2b = take(d);
    const float* wcq = take((size_t)d * d);
    const float* bcq = take(d);
    const float* wck = take((size_t)d * d);
    const float* wcv = take((size_t)d * d);
    const float* bcv = take(d);
    const float* wco = take((size_t)d * d);
    const float* bco = take(d);
    const float* ln3g = take(d);
    const float* ln3b = take(d);
    const float* w1 = take((size_t)F * d);
    const float* b1 = take(F);
    const float* w2 = take((size_t)d * F);
    const float* b2 = take(d);
    // fused [q; k; v] projection, no key bias
    tmp.assign((size_t)3 * d * d, 0.f);
    std::memcpy(tmp.data(), wq, (size_t)d * d * 4);
    std::memcpy(tmp.data() + (size_t)d * d, wk, (size_t)d * d * 4);
    std::memcpy(tmp.data() + (size_t)2 * d * d, wv, (size_t)d * d * 4);
    if ((rc = mat(&w.wqkv, (size_t)3 * d * d, tmp.data()))) return finish(rc);
    std::vector<float> bqkv(3 * d, 0.f);
    std::memcpy(bqkv.data(), bq, d * 4);
    std::memcpy(bqkv.data() + 2 * d, bv, d * 4);
    if ((rc = vec(&w.bqkv, 3 * d, bqkv.data()))) return finish(rc);
    if ((rc = mat(&w.wo, (size_t)d * d, wo)) || (rc = vec(&w.bo, d, bo))) return finish(rc);
    if ((rc = mat(&w.wcq, (size_t)d * d, wcq)) || (rc = vec(&w.bcq, d, bcq))) return finish(rc);
    if ((rc = mat(&w.wco, (size_t)d * d, wco)) || (rc = vec(&w.bco, d, bco))) return finish(rc);
    if ((rc = mat(&w.w1, (size_t)F * d, w1)) || (rc = vec(&w.b1, F, b1))) return finish(rc);
    if ((rc = mat(&w.w2, (size_t)d * F, w2)) || (rc = vec(&w.b2, d, b2))) return finish(rc);
    if ((rc = vec(&w.ln1g, d, ln1g)) || (rc = vec(&w.ln1b, d, ln1b)) || (rc = vec(&w.ln2g, d, ln2g)) ||
        (rc = vec(&w.ln2b, d, ln2b)) || (rc = vec(&w.ln3g, d, ln3g)) || (rc = vec(&w.ln3b, d, ln3b)))
      return finish(rc);
    // cross K/V projection of this layer: rows [k; v] of the stacked all-layer matrix
    char* wc = static_cast<char*>(h->w_cross) + (size_t)l * 2 * d * d * es;
    if ((rc = upload(h, wc, wck, (size_t)d * d))) return finish(rc);
    if ((rc = upload(h, wc + (size_t)d * d * es, wcv, (size_t)d * d))) return finish(rc);
    std::vector<float> bc(2 * d, 0.f);
    std::memcpy(bc.data() + d, bcv, d * 4);
    if ((rc = upload_f32(h, h->b_cross + (size_t)l * 2 * d, bc.data(), 2 * d))) return finish(rc);
    if (h->bf16) {
      bool ok = make_tmap_bf16(&w.m_wqkv, w.wqkv, 3 * d, d, 128) && make_tmap_bf16(&w.m_wo, w.wo, d, d, 128) &&
                make_tmap_bf16(&w.m_wcq, w.wcq, d, d, 128) && make_tmap_bf16(&w.m_wco, w.wco, d, d, 128) &&
                make_tmap_bf16(&w.m_w1, w.w1, F, d, 128) && make_tmap_bf16(&w.m_w2, w.w2, d, F, 128);
      if (!ok) return finish(fail(h, ASR_E_CUDA, "tensor map encode failed"));
    }
  }
  const float* lnfg = take(d);
  const float* lnfb = take(d);
  if ((rc = dalloc(h, &h->lnf_g, d * 4)) || (rc = upload_f32(h, h->lnf_g, lnfg, d))) return finish(rc);
  if ((rc = dalloc(h, &h->lnf_b, d * 4)) || (rc = upload_f32(h, h->lnf_b, lnfb, d))) return finish(rc);
  if (h->bf16 && !make_tmap_bf16(&h->m_tok, h->w_tok, h->V, d, 128))
    return finish(fail(h, ASR_E_CUDA, "tensor map encode failed"));
  if (h->ln_fold) {
    auto fold = [&](const void* W, const float* g, const float* b, int M, float** c1, float** c2) {
      int r = dalloc(h, c1, (size_t)M * 4);
      if (!r) r = dalloc(h, c2, (size_t)M * 4);
      if (!r) launch_ln_fold(W, g, b, M, d, *c1, *c2, h->st);
      return r;
    };
    for (int l = 0; l < L; ++l) {
      LayerW& w = h->lw[l];
      if ((rc = fold(w.wqkv, w.ln1g, w.ln1b, 3 * d, &w.c1_qkv, &w.c2_qkv)) ||
          (rc = fold(w.wcq, w.ln2g, w.ln2b, d, &w.c1_cq, &w.c2_cq)) ||
          (rc = fold(w.w1, w.ln3g, w.ln3b, F, &w.c1_fc1, &w.c2_fc1)))
        return finish(rc);
    }
    if ((rc = fold(h->w_tok, h->lnf_g, h->lnf_b, h->V, &h->c1_lm, &h->c2_lm))) return finish(rc);
    CK(cudaGetLastError());
  }

  // caches
  const size_t self_bytes = (size_t)L * h->Bmax * h->H * h->maxpos * 64 * es;
  const size_t cross_bytes = (size_t)L * 2 * h->Bmax * h->H * h->Tmax * 64 * es;
  if ((rc = dalloc(h, &h->kself, self_bytes)) || (rc = dalloc(h, &h->vself, self_bytes)) ||
      (rc = dalloc(h, &h->xkv, cross_bytes)))
    return finish(rc);
  // Attention reads whole 128-key chunks and masks the keys past a row's range;
  // rows never written (encoder padding, positions not yet cached) hold zeros,
  // so that a masked probability of 0 never meets a non-finite value.
  CK(cudaMemset(h->kself, 0, self_bytes));
  CK(cudaMemset(h->vself, 0, self_bytes));
  CK(cudaMemset(h->xkv, 0, cross_bytes));
  if ((rc = dalloc(h, &h->enc_len, h->Bmax * 4)) || (rc = dalloc(h, &h->kv_len, h->Bmax * 4)) ||
      (rc = dalloc(h, &h->pending, h->Bmax * 4)) || (rc = dalloc(h, &h->ready, h->Bmax * 4)))
    return finish(rc);
  CK(cudaMemset(h->ready, 0, h->Bmax * 4));
  CK(cudaMemset(h->kv_len, 0, h->Bmax * 4));
  CK(cudaMemset(h->pending, 0, h->Bmax * 4));
  CK(cudaMemset(h->enc_len, 0, h->Bmax * 4));

  // work buffers
  h->R_max = h->Bmax * (h->kmax + 1);
  h->R_pad = ((h->R_max + 255) / 256) * 256;
  const size_t R = h->R_pad;
  if ((rc = dalloc(h, &h->x, R * d * 4)) || (rc = dalloc(h, &h->q, R * d * 4)) ||
      (rc = dalloc(h, &h->q_anchor, R * d * 4)) || (rc = dalloc(h, &h->ml, R * h->H * 2 * 4)) ||
      (rc = dalloc(h, &h->xn, R * d * es)) || (rc = dalloc(h, &h->att, R * d * es)) ||
      (rc = dalloc(h, &h->hbuf, R * F * es)) || (rc = dalloc(h, &h->xf, R * d * es)))
    return finish(rc);
  CK(cudaMemset(h->xn, 0, R * d * es));
  CK(cudaMemset(h->att, 0, R * d * es));
  CK(cudaMemset(h->hbuf, 0, R * F * es));
  CK(cudaMemset(h->xf, 0, R * d * es));
  if (h->ln_fold) {   // slices of at least 8 features
    if ((rc = dalloc(h, &h->ln_part, (size_t)(d / 8) * R * sizeof(float2)))) return finish(rc);
    CK(cudaMemset(h->ln_part, 0, (size_t)(d / 8) * R * sizeof(float2)));
  }
  const int chunk = h->bf16 ? 128 : attn_chunk_len(0);   // the finest split either path uses
  const int n_chunks = (std::max(h->maxpos, h->Tmax) + chunk - 1) / chunk;
  if ((rc = dalloc(h, &h->part, (size_t)h->Bmax * h->H * n_chunks * (h->kmax + 1) * 66 * 4))) return finish(rc);
  if ((rc = dalloc(h, &h->plan.row_b, R * 4)) || (rc = dalloc(h, &h->plan.row_i, R * 4)) ||
      (rc = dalloc(h, &h->plan.row_pos, R * 4)) || (rc = dalloc(h, &h->plan.row_tok, R * 4)) ||
      (rc = dalloc(h, &h->plan.row_epos, R * 4)) || (rc = dalloc(h, &h->plan.row_mask, R * 4)) ||
      (rc = dalloc(h, &h->plan.row_start, (h->Bmax + 1) * 4)) || (rc = dalloc(h, &h->plan.n_rows, 4)) ||
      (rc = dalloc(h, &h->plan.n_utt_rows, h->Bmax * 4)))
    return finish(rc);
  CK(cudaMemset(h->plan.n_rows, 0, 4));
  if ((rc = dalloc(h, &h->row_key, R * 8)) || (rc = dalloc(h, &h->frame_key, h->Bmax * 12)) ||
      (rc = dalloc(h, &h->anchor_row, h->Bmax * 4)))
    return finish(rc);
  CK(cudaMemset(h->frame_key, 0, h->Bmax * 12));
  if ((rc = dalloc(h, &h->parent_buf, (size_t)h->Bmax * std::max(h->kmax, 1) * 4)) ||
      (rc = dalloc(h, &h->path_buf, (size_t)h->Bmax * std::max(h->kmax, 1) * 4)))
    return finish(rc);
  if ((rc = dalloc(h, &h->draft_buf, (size_t)h->Bmax * std::max(h->kmax, 1) * 4)) ||
      (rc = dalloc(h, &h->lens_buf, h->Bmax * 4)) || (rc = dalloc(h, &h->prompt_buf, (size_t)h->Bmax * h->maxpos * 4)) ||
      (rc = dalloc(h, &h->out4, 5 * h->Bmax * 4)) || (rc = dalloc(h, &h->misc, 64 * 4)) ||
      (rc = dalloc(h, &h->anchor_prof, (size_t)h->Bmax * h->Tmax * 4)) ||
      (rc = dalloc(h, &h->status, 4)))
    return finish(rc);
  CK(cudaMemset(h->status, 0, 4));
  h->ws_floats = (size_t)16 << 20;  // 64 MB of split-K partials
  h->n_tickets = 8192;
  if ((rc = dalloc(h, &h->ws, h->ws_floats * 4)) || (rc = dalloc(h, &h->tickets, h->n_tickets * 4))) return finish(rc);
  CK(cudaMemset(h->tickets, 0, h->n_tickets * 4));
  if ((rc = dalloc(h, &h->attn_tickets, (size_t)h->Bmax * h->H * 4))) return finish(rc);
  CK(cudaMemset(h->attn_tickets, 0, (size_t)h->Bmax * h->H * 4));
  if (h->bf16) {
    const uint64_t self_rows = (uint64_t)L * h->Bmax * h->H * h->maxpos;
    const uint64_t cross_rows = (uint64_t)L * 2 * h->Bmax * h->H * h->Tmax;
    for (int i = 0; i < 2; ++i) {
      const uint32_t box = i ? 256 : 128;
      if (!make_tmap_cache(&h->m_kself[i], h->kself, self_rows, box) ||
          !make_tmap_cache(&h->m_vself[i], h->vself, self_rows, box) ||
          !make_tmap_cache(&h->m_xkv[i], h->xkv, cross_rows, box))
        return finish(fail(h, ASR_E_CUDA, "tensor map encode failed"));
    }
  }
  if ((rc = dalloc(h, &h->counters, 8 * sizeof(unsigned long long)))) return finish(rc);
  CK(cudaMemset(h->counters, 0, 8 * sizeof(unsigned long long)));
  if (const char* e = std::getenv("ASRSPEC_FEWROW")) h->use_fewrow = std::atoi(e) != 0;
  if (h->bf16) {
    int C = 0;
    int n_sm = 0, gd = 0;
    if (fr_configure(d, F, h->H, h->maxpos, &C, &n_sm, &gd)) {
      h->fr_C = C;
      h->fr_sms = n_sm;
      h->fr_gd = gd;
      for (int l = 0; l < L; ++l) {   // packed copies of the layer weights
        LayerW& w = h->lw[l];
        struct {
          void* src;
          void** dst;
          int N, K;
        } mats[6] = {{w.wqkv, &w.p_qkv, 3 * d, d}, {w.wo, &w.p_wo, d, d},  {w.wcq, &w.p_wcq, d, d},
                     {w.wco, &w.p_wco, d, d},     {w.w1, &w.p_w1, F, d},   {w.w2, &w.p_w2, d, F}};
        for (auto& m : mats) {
          if ((rc = dalloc(h, m.dst, (size_t)m.N * m.K * 2))) return finish(rc);
          CK(launch_fr_pack(m.src, *m.dst, m.N, m.K, h->st));
        }
      }
    }
  }
  configure_gemm_tc();
  configure_attention();
  CK(cudaDeviceSynchronize());
  return finish(0);
}

int asr_spec_set_host_io(asr_spec_handle h, int host_io) {
  if (!h) return ASR_E_INVAL;
  h->host_io = host_io ? 1 : 0;
  return ASR_OK;
}

int asr_spec_encode_cache(asr_spec_handle h, int32_t B, const void* enc_states, int32_t t_max,
                          const int32_t* enc_lens) {
  if (!h) return ASR_E_INVAL;
  if (B < 1 || B > h->Bmax || !enc_states || !enc_lens || t_max < 1) return fail(h, ASR_E_INVAL, "bad arguments");
  if (t_max > h->Tmax) return fail(h, ASR_E_CAPACITY, "t_max exceeds max_enc");
  if (int rc = copy_in(h, h->enc_len, enc_lens, B)) return rc;
  Prof p(h, ASR_PROF_OTHER, 1);
  launch_mark_ready(h->enc_len, B, t_max, h->ready, h->kv_len, h->pending, h->status, h->st);
  const int d = h->d;
  Epi e{};
  e.bias = h->b_cross;
  e.d = d;
  e.kcache = h->xkv;
  e.kv_bf16 = h->bf16;
  e.n_heads = h->H;
  e.enc_len = h->enc_len;
  e.t_max = t_max;
  e.max_enc = h->Tmax;
  e.b_max = h->Bmax;
  e.status = h->status;
  const int M = B * t_max, N = h->L * 2 * d;
  e.M = M;
  e.N = N;
  if (h->bf16) {
    TcGemm g{};
    g.bn = h->enc_bn;
    if (!make_tmap_bf16(&g.mapA, enc_states, M, d, 128) || !make_tmap_bf16(&g.mapB, h->w_cross, N, d, g.bn))
      return fail(h, ASR_E_INVAL, "encoder states must be 16-byte aligned");
    g.M = M;
    g.N = N;
    g.K = d;
    e.group_m = h->enc_group;   // both operands exceed L2: bands of frame tiles sweep the weight tiles
    g.splits = 1;
    g.ws = h->ws;
    g.tickets = h->tickets;
    Prof pg(h, ASR_PROF_OTHER, 1);
    launch_gemm_tc(g, EPI_CROSSKV, e, h->status, h->st);
  } else {
    Prof pg(h, ASR_PROF_OTHER, 1);
    launch_gemm_simt(enc_states, 0, h->w_cross, 0, M, N, d, EPI_CROSSKV, e, h->st);
  }
  if (h->has_draft && h->bf16) {   // the draft's own cross K/V of the same encoder states
    Epi de = e;
    de.bias = h->dw.b_cross;
    de.kcache = h->d_xkv;
    de.N = 2 * d;
    TcGemm g{};
    g.bn = h->enc_bn;
    if (!make_tmap_bf16(&g.mapA, enc_states, M, d, 128) || !make_tmap_bf16(&g.mapB, h->dw.w_cross, 2 * d, d, g.bn))
      return fail(h, ASR_E_INVAL, "encoder states must be 16-byte aligned");
    g.M = M;
    g.N = 2 * d;
    g.K = d;
    g.splits = 1;
    g.ws = h->ws;
    g.tickets = h->tickets;
    Prof pg(h, ASR_PROF_OTHER, 1);
    launch_gemm_tc(g, EPI_CROSSKV, de, h->status, h->st);
  }
  CK(cudaGetLastError());
  h->B = B;
  h->t_max = t_max;
  h->state = 1;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_prefill(asr_spec_handle h, const int32_t* prompt, int32_t P0) {
  if (!h) return ASR_E_INVAL;
  if (h->state < 1) return fail(h, ASR_E_STATE, "prefill before encode_cache");
  if (!prompt || P0 < 1) return fail(h, ASR_E_INVAL, "bad arguments");
  if (P0 > h->maxpos) return fail(h, ASR_E_CAPACITY, "prompt longer than max_pos");
  if (int rc = copy_in(h, h->prompt_buf, prompt, (size_t)h->B * P0)) return rc;
  if (h->has_draft) {
    CK(cudaMemsetAsync(h->d_last_tap, 0, (size_t)h->Bmax * 4 * h->d * 4, h->st));
    h->d_after_verify = false;
  }
  const int c_max = h->kmax + 1;
  for (int p0 = 0; p0 < P0 - 1; p0 += c_max) {
    const int c = std::min(c_max, P0 - 1 - p0);
    {
      Prof p(h, ASR_PROF_OTHER, 1);
      launch_plan_prefill_chunk(h->prompt_buf, P0, p0, c, h->B, h->V, h->ready, h->plan, h->status, h->st);
    }
    if (int rc = run_layers(h, h->B * c)) return rc;
    if (h->has_draft) {   // the draft's cache of the same prompt rows (their taps as its inputs)
      DraftArgs A{};
      A.B = h->B;
      A.d = h->d;
      A.vocab = h->V;
      A.max_pos = h->maxpos;
      A.r_max = h->R_pad;
      A.status = h->status;
      A.enc_len = h->enc_len;
      A.taps = h->d_taps;
      A.last_tap = h->d_last_tap;
      A.plan = h->plan;
      A.row_lo = h->d_row_lo;
      A.row_hi = h->d_row_hi;
      A.x_in = static_cast<__nv_bfloat16*>(h->d_xin);
      launch_draft_prefill_gather(A, h->B * c, h->st);
      if (int rc = draft_block(h, h->plan, h->B * c, false)) return rc;
    }
    Prof p(h, ASR_PROF_OTHER, 1);
    launch_prefill_advance(h->B, c, h->plan.n_utt_rows, h->kv_len, h->st);
  }
  Prof p(h, ASR_PROF_OTHER, 1);
  launch_prefill_finish(h->prompt_buf, P0, h->B, h->pending, h->ready, h->st);
  CK(cudaGetLastError());
  h->state = 2;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

namespace {

// The verify call: inputs into the internal buffers, the body (a CUDA graph per
// (B, k, linear or tree), captured on first use), outputs out.
int verify_call(asr_spec* h, const int32_t* draft, const int32_t* parent, const int32_t* lens, int32_t k,
                int32_t* accepted, int32_t* bonus, int32_t* kv_len, int32_t* anchor, int32_t* path) {
  const bool tree = parent != nullptr;
  const int B = h->B;
  if (k > 0) {
    if (int rc = copy_in(h, h->draft_buf, draft, (size_t)B * k)) return rc;
    if (tree)
      if (int rc = copy_in(h, h->parent_buf, parent, (size_t)B * k)) return rc;
  }
  if (int rc = copy_in(h, h->lens_buf, lens, B)) return rc;
  for (int c = 0; c < ASR_PROF_N; ++c) h->cur[c] = 0;
  struct TreeScope {   // the enqueued layers read cur_tree; cleared on every way out
    asr_spec* h;
    ~TreeScope() { h->cur_tree = false; }
  } scope{h};
  h->cur_tree = tree;
  if (h->use_graphs && !h->prof && !h->tl_on && !h->fr_trace_on) {
    auto key = std::make_pair(B, tree ? 1000 + (int)k : (int)k);
    auto it = h->graphs.find(key);
    if (it == h->graphs.end()) {
      cudaGraph_t graph;
      CK(cudaStreamBeginCapture(h->st, cudaStreamCaptureModeThreadLocal));
      h->capturing = true;
      int rc = enqueue_verify(h, k);
      h->capturing = false;
      cudaError_t e = cudaStreamEndCapture(h->st, &graph);
      if (rc) return rc;
      if (e != cudaSuccess) return fail(h, ASR_E_CUDA, std::string("stream capture: ") + cudaGetErrorString(e));
      asr_spec::Graph g{};
      e = cudaGraphInstantiate(&g.exec, graph, 0);
      cudaGraphDestroy(graph);
      if (e != cudaSuccess) return fail(h, ASR_E_CUDA, std::string("graph instantiate: ") + cudaGetErrorString(e));
      for (int c = 0; c < ASR_PROF_N; ++c) g.launches[c] = h->cur[c];
      g.ln_S = h->ln_S;
      g.ln_c = h->ln_c;
      g.fused = h->last_fused;
      it = h->graphs.emplace(key, g).first;
    }
    CK(cudaGraphLaunch(it->second.exec, h->st));
    h->ln_S = it->second.ln_S;
    h->ln_c = it->second.ln_c;
    h->last_fused = it->second.fused;
    for (int c = 0; c < ASR_PROF_N; ++c) h->launches[c] += it->second.launches[c];
  } else {
    if (int rc = enqueue_verify(h, k)) return rc;
  }
  CK(cudaGetLastError());
  int* o = h->out4;
  if (int rc = copy_out(h, accepted, o, B)) return rc;
  if (int rc = copy_out(h, bonus, o + h->Bmax, B)) return rc;
  if (int rc = copy_out(h, kv_len, o + 2 * h->Bmax, B)) return rc;
  if (int rc = copy_out(h, anchor, o + 3 * h->Bmax, B)) return rc;
  if (tree && path && k > 0)
    if (int rc = copy_out(h, path, h->path_buf, (size_t)B * k)) return rc;
  h->d_after_verify = h->has_draft && !tree;
  if (!tree) h->last_k = k;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

}  // namespace

int asr_spec_verify(asr_spec_handle h, const int32_t* draft, const int32_t* lens, int32_t k, int32_t* accepted,
                    int32_t* bonus, int32_t* kv_len, int32_t* anchor) {
  if (!h) return ASR_E_INVAL;
  if (h->state < 2) return fail(h, ASR_E_STATE, "verify before prefill");
  if (k < 0 || k > h->kmax) return fail(h, ASR_E_INVAL, "k outside [0, max_draft]");
  if (!lens || (k > 0 && !draft) || !accepted || !bonus || !kv_len || !anchor)
    return fail(h, ASR_E_INVAL, "null pointer");
  return verify_call(h, draft, nullptr, lens, k, accepted, bonus, kv_len, anchor, nullptr);
}

int asr_spec_verify_tree(asr_spec_handle h, const int32_t* tokens, const int32_t* parent, const int32_t* lens,
                         int32_t n, int32_t* accepted, int32_t* bonus, int32_t* kv_len, int32_t* anchor,
                         int32_t* path) {
  if (!h) return ASR_E_INVAL;
  if (h->state < 2) return fail(h, ASR_E_STATE, "verify before prefill");
  if (!h->bf16) return fail(h, ASR_E_INVAL, "tree verify needs a bf16 model");
  if (n < 0 || n > h->kmax || n > 31) return fail(h, ASR_E_INVAL, "n outside [0, min(max_draft, 31)]");
  if (!lens || (n > 0 && (!tokens || !parent || !path)) || !accepted || !bonus || !kv_len || !anchor)
    return fail(h, ASR_E_INVAL, "null pointer");
  return verify_call(h, tokens, n > 0 ? parent : nullptr, lens, n, accepted, bonus, kv_len, anchor, path);
}

int asr_spec_draft_create(asr_spec_handle h, const asr_weights* dw) {
  if (!h || !dw || !dw->blob) return ASR_E_INVAL;
  if (!h->bf16) return fail(h, ASR_E_INVAL, "the draft needs a bf16 model");
  if (h->has_draft) return fail(h, ASR_E_STATE, "the handle already has a draft");
  if (h->state != 0) return fail(h, ASR_E_STATE, "create the draft before encode_cache");
  if (h->Bmax > 256) return fail(h, ASR_E_INVAL, "the draft serves at most 256 utterances");
  if (h->maxpos > 16384 || h->Tmax > 16384) return fail(h, ASR_E_INVAL, "the draft attends to at most 16384 keys");
  const int d = h->d, F2 = 2 * d, L = h->L;
  const size_t expect = 16 * (size_t)d * d + 18 * (size_t)d;
  if (dw->n_floats != expect) return fail(h, ASR_E_INVAL, "draft blob size");
  const float* src = dw->blob;
  size_t off = 0;
  auto take = [&](size_t n) {
    const float* p = src + off;
    off += n;
    return p;
  };
  DraftW& w = h->dw;
  int rc = 0;
  auto vec = [&](float** dst, size_t n, const float* v) {
    int r = dalloc(h, dst, n * 4);
    if (!r) r = upload_f32(h, *dst, v, n);
    return r;
  };
  auto mat = [&](void** dst, size_t n, const float* v) {
    int r = dalloc(h, dst, n * 2);
    if (!r) r = upload(h, *dst, v, n);
    return r;
  };
  const float* w_in = take((size_t)4 * d * d);
  const float* b_in = take(d);
  const float* ln1g = take(d);
  const float* ln1b = take(d);
  const float* wq = take((size_t)d * d);
  const float* bq = take(d);
  const float* wk = take((size_t)d * d);
  const float* wv = take((size_t)d * d);
  const float* bv = take(d);
  const float* wo = take((size_t)d * d);
  const float* bo = take(d);
  const float* ln2g = take(d);
  const float* ln2b = take(d);
  const float* wcq = take((size_t)d * d);
  const float* bcq = take(d);
  const float* wck = take((size_t)d * d);
  const float* wcv = take((size_t)d * d);
  const float* bcv = take(d);
  const float* wco = take((size_t)d * d);
  const float* bco = take(d);
  const float* ln3g = take(d);
  const float* ln3b = take(d);
  const float* w1 = take((size_t)F2 * d);
  const float* b1 = take(F2);
  const float* w2 = take((size_t)d * F2);
  const float* b2 = take(d);
  const float* lnfg = take(d);
  const float* lnfb = take(d);
  std::vector<float> tmp((size_t)3 * d * d);
  std::memcpy(tmp.data(), wq, (size_t)d * d * 4);
  std::memcpy(tmp.data() + (size_t)d * d, wk, (size_t)d * d * 4);
  std::memcpy(tmp.data() + (size_t)2 * d * d, wv, (size_t)d * d * 4);
  std::vector<float> bqkv(3 * d, 0.f), bx(2 * d, 0.f), wx((size_t)2 * d * d);
  std::memcpy(bqkv.data(), bq, d * 4);
  std::memcpy(bqkv.data() + 2 * d, bv, d * 4);
  std::memcpy(wx.data(), wck, (size_t)d * d * 4);
  std::memcpy(wx.data() + (size_t)d * d, wcv, (size_t)d * d * 4);
  std::memcpy(bx.data() + d, bcv, d * 4);
  if ((rc = mat(&w.w_in, (size_t)4 * d * d, w_in)) || (rc = vec(&w.b_in, d, b_in)) ||
      (rc = mat(&w.wqkv, (size_t)3 * d * d, tmp.data())) || (rc = vec(&w.bqkv, 3 * d, bqkv.data())) ||
      (rc = mat(&w.wo, (size_t)d * d, wo)) || (rc = vec(&w.bo, d, bo)) || (rc = mat(&w.wcq, (size_t)d * d, wcq)) ||
      (rc = vec(&w.bcq, d, bcq)) || (rc = mat(&w.w_cross, (size_t)2 * d * d, wx.data())) ||
      (rc = vec(&w.b_cross, 2 * d, bx.data())) || (rc = mat(&w.wco, (size_t)d * d, wco)) || (rc = vec(&w.bco, d, bco)) ||
      (rc = mat(&w.w1, (size_t)F2 * d, w1)) || (rc = vec(&w.b1, F2, b1)) || (rc = mat(&w.w2, (size_t)d * F2, w2)) ||
      (rc = vec(&w.b2, d, b2)) || (rc = vec(&w.ln1g, d, ln1g)) || (rc = vec(&w.ln1b, d, ln1b)) ||
      (rc = vec(&w.ln2g, d, ln2g)) || (rc = vec(&w.ln2b, d, ln2b)) || (rc = vec(&w.ln3g, d, ln3g)) ||
      (rc = vec(&w.ln3b, d, ln3b)) || (rc = vec(&w.lnfg, d, lnfg)) || (rc = vec(&w.lnfb, d, lnfb)))
    return rc;
  if (!make_tmap_bf16(&w.m_in, w.w_in, d, 4 * d, 128) || !make_tmap_bf16(&w.m_qkv, w.wqkv, 3 * d, d, 128) ||
      !make_tmap_bf16(&w.m_wo, w.wo, d, d, 128) || !make_tmap_bf16(&w.m_wcq, w.wcq, d, d, 128) ||
      !make_tmap_bf16(&w.m_wco, w.wco, d, d, 128) || !make_tmap_bf16(&w.m_w1, w.w1, F2, d, 128) ||
      !make_tmap_bf16(&w.m_w2, w.w2, d, F2, 128))
    return fail(h, ASR_E_CUDA, "tensor map encode failed");
  for (int i = 0; i < 4; ++i) h->taps[i] = std::max(0, (i + 1) * L / 4 - 1);
  const size_t Bm = h->Bmax, R = h->R_pad;
  const size_t self_b = Bm * h->H * h->maxpos * 64 * 2, cross_b = 2 * Bm * h->H * h->Tmax * 64 * 2;
  if ((rc = dalloc(h, &h->d_ks, self_b)) || (rc = dalloc(h, &h->d_vs, self_b)) || (rc = dalloc(h, &h->d_xkv, cross_b)) ||
      (rc = dalloc(h, &h->d_taps, R * 4 * d * 4)) || (rc = dalloc(h, &h->d_last_tap, Bm * 4 * d * 4)) ||
      (rc = dalloc(h, &h->d_x, R * d * 4)) || (rc = dalloc(h, &h->d_q, R * 3 * d * 4)) ||
      (rc = dalloc(h, &h->d_xin, R * 4 * d * 2)) || (rc = dalloc(h, &h->d_xn, R * d * 2)) ||
      (rc = dalloc(h, &h->d_att, R * d * 2)) || (rc = dalloc(h, &h->d_h, R * F2 * 2)) ||
      (rc = dalloc(h, &h->d_xf, R * d * 2)) || (rc = dalloc(h, &h->d_row_key, R * 8)))
    return rc;
  RowPlan& p = h->d_plan;
  int* ints = nullptr;
  const size_t n_int = 7 * R + (Bm + 1) + 1 + Bm + 3 * R + 9 * Bm + Bm * std::max(h->kmax, 1);
  if ((rc = dalloc(h, &ints, n_int * 4))) return rc;
  CK(cudaMemset(ints, 0, n_int * 4));
  int* q = ints;
  auto cut = [&](size_t n) {
    int* r = q;
    q += n;
    return r;
  };
  p.row_b = cut(R);
  p.row_i = cut(R);
  p.row_pos = cut(R);
  p.row_epos = cut(R);
  p.row_mask = reinterpret_cast<unsigned*>(cut(R));
  p.row_tok = cut(R);
  (void)cut(R);
  p.row_start = cut(Bm + 1);
  p.n_rows = cut(1);
  p.n_utt_rows = cut(Bm);
  h->d_row_src = cut(R);
  h->d_row_lo = cut(R);
  h->d_row_hi = cut(R);
  h->d_win_lo = cut(Bm);
  h->d_win_hi = cut(Bm);
  h->d_lens = cut(Bm);
  h->d_nprop = cut(Bm);
  h->d_last_row = cut(Bm);
  h->d_prev_pos = cut(Bm);
  h->d_total = cut(Bm);
  h->d_centers = cut(Bm);
  h->d_lens_out = cut(Bm);
  h->d_out = cut(Bm * std::max(h->kmax, 1));
  CK(cudaMemset(h->d_ks, 0, self_b));
  CK(cudaMemset(h->d_vs, 0, self_b));
  CK(cudaMemset(h->d_xkv, 0, cross_b));
  CK(cudaDeviceSynchronize());
  h->has_draft = true;
  return ASR_OK;
}

int asr_spec_draft_propose(asr_spec_handle h, int32_t k, int32_t window, const int32_t* centers,
                           const int32_t* total_len, int32_t* draft_out, int32_t* lens_out) {
  if (!h) return ASR_E_INVAL;
  if (!h->has_draft) return fail(h, ASR_E_STATE, "no draft (asr_spec_draft_create)");
  if (h->state < 2) return fail(h, ASR_E_STATE, "propose before prefill");
  if (k < 0 || k > h->kmax) return fail(h, ASR_E_INVAL, "k outside [0, max_draft]");
  if (window < DRAFT_WIN_ANCHOR || window > DRAFT_WIN_NONE) return fail(h, ASR_E_INVAL, "window kind");
  if (!total_len || !lens_out || (k > 0 && !draft_out) || (window == DRAFT_WIN_RANDOM && !centers))
    return fail(h, ASR_E_INVAL, "null pointer");
  const int B = h->B;
  if (int rc = copy_in(h, h->d_total, total_len, B)) return rc;
  if (window == DRAFT_WIN_RANDOM)
    if (int rc = copy_in(h, h->d_centers, centers, B)) return rc;
  DraftArgs A{};
  A.B = B;
  A.d = h->d;
  A.k = k;
  A.k_verify = h->last_k;
  A.win_kind = window;
  A.vocab = h->V;
  A.max_pos = h->maxpos;
  A.r_max = h->R_pad;
  A.status = h->status;
  A.after_verify = h->d_after_verify ? 1 : 0;
  A.kv_len = h->kv_len;
  A.pending = h->pending;
  A.enc_len = h->enc_len;
  A.total_len = h->d_total;
  A.v_row_start = h->plan.row_start;
  A.v_n_utt_rows = h->plan.n_utt_rows;
  A.accepted = h->out4;
  A.anchor = h->out4 + 3 * h->Bmax;
  A.v_draft = h->draft_buf;
  A.centers = h->d_centers;
  A.taps = h->d_taps;
  A.last_tap = h->d_last_tap;
  A.x_prev = h->d_x;
  A.plan = h->d_plan;
  A.row_src = h->d_row_src;
  A.row_lo = h->d_row_lo;
  A.row_hi = h->d_row_hi;
  A.win_lo = h->d_win_lo;
  A.win_hi = h->d_win_hi;
  A.lens = h->d_lens;
  A.n_prop = h->d_nprop;
  A.last_row = h->d_last_row;
  A.prev_pos = h->d_prev_pos;
  A.draft_out = h->d_out;
  A.row_key = h->d_row_key;
  A.x_in = static_cast<__nv_bfloat16*>(h->d_xin);
  A.threshold = h->d_threshold;
  A.row_p = h->d_row_p;
  // pass 0: catch-up of the last verification's accepted drafts + the restart
  const int rows0 = std::min(h->R_pad, B * (h->kmax + 1));
  launch_draft_round_plan(A, h->st);
  launch_draft_gather(A, rows0, h->st);
  if (int rc = draft_block(h, h->d_plan, rows0, true)) return rc;
  launch_draft_take(A, h->st);
  for (int i = 1; i < k; ++i) {   // continuation proposals, one row per utterance still proposing
    launch_draft_next_plan(A, i, h->st);
    launch_draft_gather(A, B, h->st);
    if (int rc = draft_block(h, h->d_plan, B, true)) return rc;
    launch_draft_take(A, h->st);
  }
  launch_draft_finish(A, h->d_lens_out, h->st);
  CK(cudaGetLastError());
  h->d_after_verify = false;
  if (k > 0)
    if (int rc = copy_out(h, draft_out, h->d_out, (size_t)B * k)) return rc;
  if (int rc = copy_out(h, lens_out, h->d_lens_out, B)) return rc;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_draft_set_threshold(asr_spec_handle h, float threshold) {
  if (!h) return ASR_E_INVAL;
  if (!h->has_draft) return fail(h, ASR_E_STATE, "no draft (asr_spec_draft_create)");
  if (!(threshold >= 0.f && threshold <= 1.f)) return fail(h, ASR_E_INVAL, "threshold outside [0, 1]");
  if (threshold > 0.f && !h->d_logits) {
    if (int rc = dalloc(h, &h->d_logits, (size_t)h->R_pad * h->V * 4)) return rc;
    if (int rc = dalloc(h, &h->d_row_p, (size_t)h->R_pad * 4)) return rc;
  }
  h->d_threshold = threshold;
  return ASR_OK;
}

int asr_spec_restart(asr_spec_handle h, int32_t* restart) {
  if (!h || !restart) return ASR_E_INVAL;
  if (h->state < 2) return fail(h, ASR_E_STATE, "restart flags before prefill");
  if (int rc = copy_out(h, restart, h->out4 + 4 * h->Bmax, h->B)) return rc;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_debug_anchor_profile(asr_spec_handle h, float* out) {
  if (!h || !out) return ASR_E_INVAL;
  if (h->state < 2) return fail(h, ASR_E_STATE, "anchor profile before prefill");
  const size_t bytes = (size_t)h->B * h->Tmax * 4;
  CK(cudaMemcpyAsync(out, h->anchor_prof, bytes, h->host_io ? cudaMemcpyDeviceToHost : cudaMemcpyDeviceToDevice,
                     h->st));
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_set_graphs(asr_spec_handle h, int enable) {
  if (!h) return ASR_E_INVAL;
  h->use_graphs = enable != 0;
  return ASR_OK;
}

int asr_spec_profile(asr_spec_handle h, int enable) {
  if (!h) return ASR_E_INVAL;
  h->prof = enable != 0;
  return ASR_OK;
}

int asr_spec_profile_read(asr_spec_handle h, double* ms, int64_t* launches, uint64_t* traffic) {
  if (!h) return ASR_E_INVAL;
  CK(cudaStreamSynchronize(h->st));
  if (ms) {
    for (int c = 0; c < ASR_PROF_N; ++c) ms[c] = 0.0;
    for (auto& m : h->marks) {
      float t = 0.f;
      CK(cudaEventElapsedTime(&t, h->ev_pool[m.second], h->ev_pool[m.second + 1]));
      ms[m.first] += t;
    }
  }
  if (launches)
    for (int c = 0; c < ASR_PROF_N; ++c) launches[c] = h->launches[c];
  if (traffic) {
    unsigned long long tmp[8];
    CK(cudaMemcpy(tmp, h->counters, sizeof(tmp), cudaMemcpyDeviceToHost));
    for (int i = 0; i < 8; ++i) traffic[i] = tmp[i];
  }
  h->marks.clear();
  h->ev_used = 0;
  for (int c = 0; c < ASR_PROF_N; ++c) h->launches[c] = 0;
  CK(cudaMemset(h->counters, 0, 8 * sizeof(unsigned long long)));
  return ASR_OK;
}

int asr_spec_timeline(asr_spec_handle h, int32_t enable) {
  if (!h) return ASR_E_INVAL;
  const size_t bytes = (size_t)ASR_TL_CAP * 4 * sizeof(unsigned long long);
  if (enable && !h->tl_buf) {
    if (int rc = dalloc(h, &h->tl_buf, bytes)) return rc;
  }
  if (h->tl_buf) CK(cudaMemsetAsync(h->tl_buf, 0, bytes, h->st));
  h->tl_kind.clear();
  h->tl_on = enable != 0;
  return ASR_OK;
}

int asr_spec_timeline_read(asr_spec_handle h, uint64_t* ns, int32_t* kind, int32_t cap, int32_t* count) {
  if (!h || cap < 0 || !count || (cap > 0 && (!ns || !kind))) return ASR_E_INVAL;
  CK(cudaStreamSynchronize(h->st));
  const int n = (int)h->tl_kind.size();
  *count = n;
  const int m = std::min(n, (int)cap);
  if (m > 0) {
    std::vector<unsigned long long> raw((size_t)m * 4);
    CK(cudaMemcpy(raw.data(), h->tl_buf, raw.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
    for (int i = 0; i < m; ++i) {
      const unsigned long long* s = &raw[(size_t)i * 4];
      ns[4 * i + 0] = s[0] ? ~s[0] : 0;   // entries were recorded complemented (max of ~t = min of t)
      ns[4 * i + 1] = s[1] ? ~s[1] : 0;
      ns[4 * i + 2] = s[3];
      ns[4 * i + 3] = s[2];
      kind[i] = h->tl_kind[i];
    }
  }
  if (h->tl_buf) CK(cudaMemsetAsync(h->tl_buf, 0, (size_t)ASR_TL_CAP * 4 * sizeof(unsigned long long), h->st));
  h->tl_kind.clear();
  return ASR_OK;
}

int asr_spec_fewrow_trace(asr_spec_handle h, int32_t enable) {
  if (!h) return ASR_E_INVAL;
  if (enable && !h->bf16) return fail(h, ASR_E_INVAL, "the phase trace needs a bf16 model");
  if (enable && !h->fr_trace) {
    const size_t n = (size_t)6 * h->L * FR_TRACE_CTAS * FR_TRACE_PHASES;
    int rc = dalloc(h, &h->fr_trace, n * sizeof(unsigned long long));
    if (rc) return rc;
    CK(cudaMemset(h->fr_trace, 0, n * sizeof(unsigned long long)));
  }
  h->fr_trace_on = enable != 0;
  return ASR_OK;
}

int asr_spec_fewrow_trace_read(asr_spec_handle h, uint64_t* out, int64_t cap, int32_t* n_launches) {
  if (!h || !n_launches || cap < 0 || (cap > 0 && !out)) return ASR_E_INVAL;
  *n_launches = h->fr_trace ? h->fr_trace_n : 0;
  const size_t n = std::min((size_t)cap, (size_t)(*n_launches) * FR_TRACE_CTAS * FR_TRACE_PHASES);
  CK(cudaStreamSynchronize(h->st));
  if (n > 0) CK(cudaMemcpy(out, h->fr_trace, n * sizeof(unsigned long long), cudaMemcpyDeviceToHost));
  return ASR_OK;
}

int asr_spec_rollback(asr_spec_handle h, const int32_t* new_len, const int32_t* new_pending) {
  if (!h) return ASR_E_INVAL;
  if (h->state < 2) return fail(h, ASR_E_STATE, "rollback before prefill");
  if (!new_len || !new_pending) return fail(h, ASR_E_INVAL, "null pointer");
  if (int rc = copy_in(h, h->misc, new_len, h->B)) return rc;
  if (int rc = copy_in(h, h->lens_buf, new_pending, h->B)) return rc;
  Prof p(h, ASR_PROF_OTHER, 1);
  launch_rollback(h->misc, h->lens_buf, h->B, h->V, h->kv_len, h->pending, h->status, h->st);
  CK(cudaGetLastError());
  h->d_after_verify = false;   // the draft has no verification rows of the rewound state
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_state(asr_spec_handle h, int32_t* kv_len, int32_t* pending) {
  if (!h || !kv_len || !pending) return ASR_E_INVAL;
  if (int rc = copy_out(h, kv_len, h->kv_len, h->B)) return rc;
  if (int rc = copy_out(h, pending, h->pending, h->B)) return rc;
  if (h->host_io) CK(cudaStreamSynchronize(h->st));
  return ASR_OK;
}

int asr_spec_debug_logits(asr_spec_handle h, float* out, int32_t max_rows) {
  if (!h || !out) return ASR_E_INVAL;
  int R = 0;
  CK(cudaMemcpyAsync(&R, h->plan.n_rows, 4, cudaMemcpyDeviceToHost, h->st));
  CK(cudaStreamSynchronize(h->st));
  if (R > max_rows) return fail(h, ASR_E_INVAL, "output too small");
  if (R == 0) return 0;
  float* dst = out;
  float* tmp = nullptr;
  if (h->host_io) {
    CK(cudaMalloc(&tmp, (size_t)R * h->V * 4));
    dst = tmp;
  }
  Epi e{};
  e.out_f32 = dst;
  e.ld = h->V;
  e.n_valid = h->plan.n_rows;
  int rc;
  if (h->ln_fold && !h->last_fused) {   // the same operand and statistics as the last verify's LM head
    fold_consumer(h, e, h->c1_lm, h->c2_lm);
    rc = gemm_rows(h, h->w_tok, &h->m_tok, h->V, h->d, h->xn, BUF_XN, R, EPI_F32, e);
  } else {
    rc = gemm_rows(h, h->w_tok, &h->m_tok, h->V, h->d, h->xf, BUF_XF, R, EPI_F32, e);
  }
  if (!rc && h->host_io) {
    CK(cudaMemcpyAsync(out, tmp, (size_t)R * h->V * 4, cudaMemcpyDeviceToHost, h->st));
  }
  CK(cudaStreamSynchronize(h->st));
  if (tmp) cudaFree(tmp);
  return rc ? rc : R;
}

int asr_spec_status(asr_spec_handle h) {
  if (!h) return ASR_E_INVAL;
  int s = 0;
  CK(cudaStreamSynchronize(h->st));
  CK(cudaMemcpy(&s, h->status, 4, cudaMemcpyDeviceToHost));
  CK(cudaMemset(h->status, 0, 4));
  return s;
}

const char* asr_spec_last_error(asr_spec_handle h) { return h ? h->err.c_str() : "null handle"; }

void asr_spec_destroy(asr_spec_handle h) {
  if (!h) return;
  cudaStreamSynchronize(h->st);
  for (auto& g : h->graphs) cudaGraphExecDestroy(g.second.exec);
  for (cudaEvent_t e : h->ev_pool) cudaEventDestroy(e);
  for (void* p : h->allocs) cudaFree(p);
  if (h->own_stream) cudaStreamDestroy(h->st);
  delete h;
}

int asr_spec_synth_drafts(asr_spec_handle h, const int32_t* truth, const int32_t* total_len, const int32_t* repl,
                          int32_t k_repl, const int32_t* shift, int32_t k, int32_t* draft_out, int32_t* lens_out) {
  if (!h || !truth || !total_len || !repl || !shift || !draft_out || !lens_out) return ASR_E_INVAL;
  if (k < 1 || k > k_repl) return fail(h, ASR_E_INVAL, "k outside [1, k_repl]");
  Prof p(h, ASR_PROF_OTHER, 1);
  launch_synth_drafts(truth, total_len, repl, k_repl, shift, k, h->B, h->maxpos, h->kv_len, draft_out, lens_out,
                      h->st);
  CK(cudaGetLastError());
  return ASR_OK;
}

int asr_spec_test_gemm(int32_t impl, const void* A, const void* B, float* C, int32_t M, int32_t N, int32_t K,
                       void* stream) {
  asr_spec* h = nullptr;
  if (!A || !B || !C || M < 1 || N < 1 || K < 64 || K % 64) return ASR_E_INVAL;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  Epi e{};
  e.M = M;
  e.N = N;
  e.out_f32 = C;
  e.ld = N;
  if (impl == 1) {
    launch_gemm_simt(A, 1, B, 1, M, N, K, EPI_F32_MN, e, st);
  } else if (impl == 3) {
    // fused argmax over m for every n: C[n] = index of the largest C[.][n]
    TcGemm g{};
    g.bn = tc_pick_bn(N);
    if (!make_tmap_bf16(&g.mapA, A, M, K, 128) || !make_tmap_bf16(&g.mapB, B, N, K, g.bn)) return ASR_E_INVAL;
    g.M = M;
    g.N = N;
    g.K = K;
    g.splits = 1;
    unsigned long long* keys = nullptr;
    int* status = nullptr;
    CK(cudaMalloc(&keys, (size_t)N * 8));
    CK(cudaMalloc(&status, 4));
    CK(cudaMemsetAsync(keys, 0, (size_t)N * 8, st));
    CK(cudaMemsetAsync(status, 0, 4, st));
    e.row_key = keys;
    launch_gemm_tc(g, EPI_ARGMAX, e, status, st);
    CK(cudaGetLastError());
    std::vector<unsigned long long> hk(N);
    std::vector<float> idx(N);
    CK(cudaMemcpyAsync(hk.data(), keys, (size_t)N * 8, cudaMemcpyDeviceToHost, st));
    CK(cudaStreamSynchronize(st));
    for (int n = 0; n < N; ++n) idx[n] = (float)(0xFFFFFFFFu - (uint32_t)(hk[n] & 0xFFFFFFFFull));
    CK(cudaMemcpy(C, idx.data(), (size_t)N * 4, cudaMemcpyHostToDevice));
    cudaFree(keys);
    cudaFree(status);
  } else if (impl >= 5 && impl <= 7) {
    // the many-row kernel: 5 = query epilogue, 6 = GELU (bf16 out), 7 = residual (onto x = 0);
    // zero bias, outputs [N][M]
    const int mode = impl == 5 ? EPI_Q : impl == 6 ? EPI_GELU : EPI_RESID;
    int sms = 0, dev = 0;
    CK(cudaGetDevice(&dev));
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    WideGemm w{};
    if (!wide_pick(M, N, K, mode, sms, &w.bn, &w.split)) return ASR_E_INVAL;
    if (!make_tmap_bf16(&w.mapA, A, M, K, 128) || !make_tmap_bf16(&w.mapB, B, N, K, w.bn)) return ASR_E_INVAL;
    w.mapX = w.mapA;
    if (mode == EPI_RESID && !make_tmap_f32(&w.mapX, C, N, M, 128, w.bn)) return ASR_E_INVAL;
    w.M = M;
    w.N = N;
    w.K = K;
    float* bias = nullptr;
    int* status = nullptr;
    __nv_bfloat16* act = nullptr;
    CK(cudaMalloc(&bias, (size_t)M * 4));
    CK(cudaMalloc(&status, 4));
    CK(cudaMemsetAsync(bias, 0, (size_t)M * 4, st));
    CK(cudaMemsetAsync(status, 0, 4, st));
    e.d = M;
    e.bias = bias;
    if (mode == EPI_GELU) {
      CK(cudaMalloc(&act, (size_t)M * N * 2));
      e.act = act;
      e.act_bf16 = 1;
    } else if (mode == EPI_RESID) {
      CK(cudaMemsetAsync(C, 0, (size_t)M * N * 4, st));
      e.x = C;
    }
    launch_gemm_wide(w, mode, e, status, st);
    CK(cudaGetLastError());
    CK(cudaStreamSynchronize(st));
    if (mode == EPI_GELU) {   // bf16 -> fp32 through the host
      std::vector<uint16_t> hb((size_t)M * N);
      std::vector<float> hf((size_t)M * N);
      CK(cudaMemcpy(hb.data(), act, hb.size() * 2, cudaMemcpyDeviceToHost));
      for (size_t i = 0; i < hb.size(); ++i) {
        const uint32_t u = (uint32_t)hb[i] << 16;
        std::memcpy(&hf[i], &u, 4);
      }
      CK(cudaMemcpy(C, hf.data(), hf.size() * 4, cudaMemcpyHostToDevice));
      cudaFree(act);
    }
    int hs = 0;
    CK(cudaMemcpy(&hs, status, 4, cudaMemcpyDeviceToHost));
    cudaFree(bias);
    cudaFree(status);
    if (hs) return ASR_E_DEVICE;
  } else {
    TcGemm g{};
    g.bn = impl == 4 && N > 64 ? tc_pick_bn_wide(N) : tc_pick_bn(N);
    if (!make_tmap_bf16(&g.mapA, A, M, K, 128) || !make_tmap_bf16(&g.mapB, B, N, K, g.bn)) return ASR_E_INVAL;
    g.M = M;
    g.N = N;
    g.K = K;
    const int tiles = ((M + 127) / 128) * ((N + g.bn - 1) / g.bn);
    g.splits = impl == 2 ? std::min(3, K / 64) : 1;
    if (impl == 4) {   // split K inside a cluster
      g.splits = 1;
      while (g.splits < 8 && g.splits * 2 <= K / 64) g.splits *= 2;
      g.cluster = g.splits > 1;
    }
    int* status = nullptr;
    CK(cudaMalloc(&status, 4));
    CK(cudaMemset(status, 0, 4));
    if (g.splits > 1 && !g.cluster) {
      CK(cudaMalloc(&g.ws, (size_t)g.splits * tiles * 128 * g.bn * 4));
      CK(cudaMalloc(&g.tickets, (size_t)tiles * 4));
      CK(cudaMemset(g.tickets, 0, (size_t)tiles * 4));
    }
    launch_gemm_tc(g, EPI_F32_MN, e, status, st);
    CK(cudaGetLastError());
    CK(cudaStreamSynchronize(st));
    int s = 0;
    CK(cudaMemcpy(&s, status, 4, cudaMemcpyDeviceToHost));
    cudaFree(status);
    if (g.ws) cudaFree(g.ws);
    if (g.tickets) cudaFree(g.tickets);
    if (s) return ASR_E_DEVICE;
  }
  CK(cudaGetLastError());
  CK(cudaStreamSynchronize(st));
  return ASR_OK;
}

}  // extern "C"
