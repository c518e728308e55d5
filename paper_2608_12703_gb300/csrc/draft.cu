// The draft side of the speculative loop on the device (App. "Draft
// architecture"; Sec. 3 "Speculative Loop"; App. "Decoding and Intervention
// Protocol": the real cached loop): row plans of the draft's passes, the
// gathers of its inputs (four tapped target representations, or its own
// block output for continuation proposals), the pick-up of its proposals,
// and the attention of its one block, whose audio cross-attention may be
// restricted to a window of encoder frames around a centre (App. "Window
// geometry"; Sec. 5 "Verification-Attention Correction").
//
// A round: pass 0 scores, per utterance, the positions the last
// verification committed (the accepted drafts, fed by the verification
// rows' target representations: the catch-up) and then the pending token at
// the new committed length (the restart, whose argmax is proposal 1); passes
// 1 .. k - 1 score one continuation row per utterance still proposing.  The
// block itself runs on the library's GEMMs; these kernels only lay out rows
// and move inputs.
#include <cmath>

#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_draft)

namespace {

constexpr int DP_T = 256;                  // threads of the one-CTA plan kernels (B <= 256 per pass)
constexpr int WIN_HALF = 20;               // window half-width: 400 ms on the 20 ms encoder grid
constexpr int WIN_SHIFT = 25;              // shifted control: +500 ms

// exclusive prefix sum over the CTA (DP_T threads)
__device__ int excl_scan(int v, int* total) {
  __shared__ int s[DP_T];
  s[threadIdx.x] = v;
  __syncthreads();
  for (int o = 1; o < DP_T; o <<= 1) {
    const int a = threadIdx.x >= o ? s[threadIdx.x - o] : 0;
    __syncthreads();
    s[threadIdx.x] += a;
    __syncthreads();
  }
  const int incl = s[threadIdx.x];
  *total = s[DP_T - 1];
  __syncthreads();
  return incl - v;
}

__device__ __forceinline__ void window_of(int kind, int anchor, int T, const int* centers, int b, int& lo, int& hi) {
  if (kind == DRAFT_WIN_NONE) {
    lo = 0;
    hi = T;
    return;
  }
  int c;
  if (kind == DRAFT_WIN_RANDOM) c = centers[b];
  else if (kind == DRAFT_WIN_SHIFTED) c = max(anchor, 0) + WIN_SHIFT;
  else c = max(anchor, 0);
  c = min(max(c, 0), T - 1);
  lo = max(c - WIN_HALF, 0);
  hi = min(c + WIN_HALF + 1, T);
}

// Pass 0 of a round.  Per utterance b: lens[b] = -1 once it holds its
// transcript (kv_len + 1 >= total), else min(k, total - kv_len - 2); after a
// verification that scored it, one catch-up row per accepted draft j
// (position P_old + j, token draft j, features of verification row j - 1);
// then, unless lens[b] < 0, the restart row (position kv_len, the pending
// token, features of the verification row that scored it, or after the
// prefill the saved tap of the last prompt row).  Row sources: >= 0 a tap
// row, -1 the saved tap of utterance b, -2 zeros.
__global__ void __launch_bounds__(DP_T) draft_round_plan_kernel(DraftArgs A) {
  const int b = threadIdx.x;
  int n_rows = 0, n_acc = 0, lens = -1, r0v = 0;
  bool scored = false;
  if (b < A.B) {
    const int P = A.kv_len[b], N = A.total_len[b];
    lens = P + 1 >= N ? -1 : min(A.k, N - P - 2);
    // the round's verification must fit the context: kv_len + lens + 1 <= max_pos
    if (lens >= 0 && lens > A.max_pos - 1 - P) {
      lens = P >= A.max_pos ? -1 : A.max_pos - 1 - P;
      atomicOr(A.status, ST_CAPACITY);
    }
    if (A.after_verify) {
      scored = A.v_n_utt_rows[b] > 0;
      if (scored) {
        n_acc = min(max(A.accepted[b], 0), min(A.k_verify, P - 1));
        r0v = A.v_row_start[b];
      }
    }
    n_rows = n_acc + (lens >= 0 ? 1 : 0);
  }
  int total;
  const int start = excl_scan(n_rows, &total);
  if (b < A.B) {
    const int P = A.kv_len[b], T = A.enc_len[b];
    int lo, hi;
    window_of(A.win_kind, A.after_verify ? A.anchor[b] : 0, T, A.centers, b, lo, hi);
    A.plan.row_start[b] = start;
    A.plan.n_utt_rows[b] = n_rows;
    A.lens[b] = lens;
    A.n_prop[b] = 0;
    A.win_lo[b] = lo;
    A.win_hi[b] = hi;
    A.last_row[b] = lens >= 0 ? start + n_acc : -1;
    const int P_old = P - 1 - n_acc;   // committed length before the verification (after_verify)
    for (int j = 1; j <= n_acc; ++j) {   // catch-up: unrestricted audio attention
      const int r = start + j - 1;
      A.plan.row_b[r] = b;
      A.plan.row_i[r] = j - 1;
      A.plan.row_pos[r] = P_old + j;
      A.plan.row_epos[r] = P_old + j;
      const int tok = A.v_draft[(size_t)b * A.k_verify + j - 1];
      A.plan.row_tok[r] = (tok >= 0 && tok < A.vocab) ? tok : 0;
      A.row_src[r] = r0v + j - 1;
      A.row_lo[r] = 0;
      A.row_hi[r] = T;
      A.row_key[r] = 0ull;
    }
    if (lens >= 0) {   // restart
      const int r = start + n_acc;
      A.plan.row_b[r] = b;
      A.plan.row_i[r] = n_acc;
      A.plan.row_pos[r] = P;
      A.plan.row_epos[r] = P;
      A.plan.row_tok[r] = A.pending[b];
      A.row_src[r] = scored ? r0v + n_acc : (A.after_verify ? -2 : -1);
      A.row_lo[r] = lo;
      A.row_hi[r] = hi;
      A.row_key[r] = 0ull;
    }
  }
  if (threadIdx.x == 0) {
    A.plan.row_start[A.B] = total;
    *A.plan.n_rows = total;
  }
}

// Pass i >= 1: one continuation row per utterance whose i proposals so far
// leave it short of lens[b]: position one past its previous row, the
// previous proposal as token, the previous row's block output (for all four
// representations) as features, the round's window.
__global__ void __launch_bounds__(DP_T) draft_next_plan_kernel(DraftArgs A, int i) {
  const int b = threadIdx.x;
  const bool on = b < A.B && A.lens[b] > i && A.n_prop[b] == i && A.last_row[b] >= 0;
  int total;
  const int r = excl_scan(on ? 1 : 0, &total);
  if (b < A.B) {
    A.plan.row_start[b] = r;
    A.plan.n_utt_rows[b] = on ? 1 : 0;
    if (on) {
      const int pr = A.last_row[b];
      const int pos = A.prev_pos[b] + 1;
      A.plan.row_b[r] = b;
      A.plan.row_i[r] = 0;
      A.plan.row_pos[r] = pos;
      A.plan.row_epos[r] = pos;
      A.plan.row_tok[r] = A.draft_out[(size_t)b * A.k + i - 1];
      A.row_src[r] = -3 - pr;   // the previous pass's block output of row pr
      A.row_lo[r] = A.win_lo[b];
      A.row_hi[r] = A.win_hi[b];
      A.row_key[r] = 0ull;
      A.last_row[b] = r;
    } else if (b < A.B) {
      A.last_row[b] = -1;
    }
  }
  if (threadIdx.x == 0) {
    A.plan.row_start[A.B] = total;
    *A.plan.n_rows = total;
  }
}

// x_in[r] = bf16 of the row's four representations ([4][d]): a tap row, the
// saved tap of its utterance, zeros, or (continuation) the previous pass's
// block output x_prev[pr] four times.  Grid-stride over rows x 4 d / 2.
__global__ void draft_gather_kernel(DraftArgs A) {
  const int R = *A.plan.n_rows, d = A.d;
  const int per = 2 * d;   // bf16 pairs per row
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < R * per; e += gridDim.x * blockDim.x) {
    const int r = e / per, c = 2 * (e - r * per);   // column c, c + 1 of [4 d]
    const int src = A.row_src[r];
    if (bounds_bad(A.status, src >= A.r_max || (src <= -3 && -3 - src >= A.r_max) || r >= A.r_max ||
                                 (src == -1 && (A.plan.row_b[r] < 0 || A.plan.row_b[r] >= A.B))))
      continue;
    float2 v;
    if (src >= 0) v = *reinterpret_cast<const float2*>(A.taps + (size_t)src * 4 * d + c);
    else if (src == -1) v = *reinterpret_cast<const float2*>(A.last_tap + (size_t)A.plan.row_b[r] * 4 * d + c);
    else if (src == -2) v = make_float2(0.f, 0.f);
    else v = *reinterpret_cast<const float2*>(A.x_prev + (size_t)(-3 - src) * d + (c % d));
    *reinterpret_cast<__nv_bfloat162*>(A.x_in + (size_t)r * 4 * d + c) = __floats2bfloat162_rn(v.x, v.y);
  }
}

// Prefill: the draft scores the target's prefill rows (the target's row plan
// of the chunk: prompt token p at position p); row r's representations are
// the tap of the target row at position p - 1 (the previous row of its
// utterance in this chunk, or the saved tap of the previous chunk's last row,
// zeros at p = 0); afterwards the chunk's last row of each utterance becomes
// the saved tap.  Unrestricted audio attention.
__global__ void draft_prefill_gather_kernel(DraftArgs A) {
  const int R = *A.plan.n_rows, d = A.d;
  const int per = 2 * d;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < R * per; e += gridDim.x * blockDim.x) {
    const int r = e / per, c = 2 * (e - r * per);
    const int b = A.plan.row_b[r], p = A.plan.row_pos[r];
    if (bounds_bad(A.status, r >= A.r_max || b < 0 || b >= A.B)) continue;
    float2 v = make_float2(0.f, 0.f);
    if (p > 0) v = A.plan.row_i[r] > 0 ? *reinterpret_cast<const float2*>(A.taps + (size_t)(r - 1) * 4 * d + c)
                                      : *reinterpret_cast<const float2*>(A.last_tap + (size_t)b * 4 * d + c);
    *reinterpret_cast<__nv_bfloat162*>(A.x_in + (size_t)r * 4 * d + c) = __floats2bfloat162_rn(v.x, v.y);
    if (c == 0) {
      A.row_lo[r] = 0;
      A.row_hi[r] = A.enc_len[b];
    }
  }
}

// The saved tap of each utterance := its last row of the prefill chunk (after
// the chunk's gather has read the old one).
__global__ void draft_prefill_save_kernel(DraftArgs A) {
  const int B = A.B, d = A.d;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < B * 4 * d; e += gridDim.x * blockDim.x) {
    const int b = e / (4 * d), c = e - b * 4 * d;
    const int n = A.plan.n_utt_rows[b];
    if (n > 0) A.last_tap[(size_t)b * 4 * d + c] = A.taps[(size_t)(A.plan.row_start[b] + n - 1) * 4 * d + c];
  }
}

// x[r] += tok_emb[token] + pos_emb[position]  (the draft's input combination:
// w_in [f_1; ..; f_4] + b_in was written by the input GEMM)
__global__ void draft_embed_kernel(DraftArgs A, const __nv_bfloat16* tok_emb, const __nv_bfloat16* pos_emb, float* x) {
  const int R = *A.plan.n_rows, d = A.d;
  for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < R * d; e += gridDim.x * blockDim.x) {
    const int r = e / d, c = e - r * d;
    const int tok = A.plan.row_tok[r], pos = A.plan.row_epos[r];
    if (bounds_bad(A.status, tok < 0 || tok >= A.vocab || pos < 0 || pos >= A.max_pos || r >= A.r_max)) continue;
    x[e] += __bfloat162float(tok_emb[(size_t)A.plan.row_tok[r] * d + c]) +
            __bfloat162float(pos_emb[(size_t)A.plan.row_epos[r] * d + c]);
  }
}

// After a pass's LM head: each utterance with a row in the pass takes its
// argmax as the next proposal (until it holds lens[b] of them, or, with the
// confidence threshold on, until the argmax's probability falls below it:
// the block then ends unproposed) and keeps the row's position for the next
// continuation row.
__global__ void draft_take_kernel(DraftArgs A) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= A.B) return;
  const int r = A.last_row[b];
  if (r < 0) return;
  const int n = A.n_prop[b];
  A.prev_pos[b] = A.plan.row_pos[r];
  if (n < A.lens[b]) {
    if (A.threshold > 0.f && A.row_p[r] < A.threshold) {   // not confident: the block ends here
      A.lens[b] = n;
      return;
    }
    const uint32_t tok = argmax_index(A.row_key[r]);
    A.draft_out[(size_t)b * A.k + n] = tok < (uint32_t)A.vocab ? (int)tok : 0;
    A.n_prop[b] = n + 1;
  }
}

// Softmax statistics of one row of logits (one CTA per row, fixed reduction
// order): the argmax (lowest index on ties) and its probability
// 1 / sum_v exp(l_v - l_max) (App. "Draft length and confidence threshold").
__global__ void __launch_bounds__(256) draft_softmax_kernel(const float* __restrict__ logits, int V,
                                                            const int* n_rows, unsigned long long* row_key,
                                                            float* row_p) {
  __shared__ float s_m[8], s_s[8];
  __shared__ int s_i[8];
  const int r = blockIdx.x;
  if (r >= *n_rows) return;   // uniform over the CTA
  const float* l = logits + (size_t)r * V;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  float m = -INFINITY;
  int mi = 0x7fffffff;
  for (int v = tid; v < V; v += 256) {
    const float x = l[v];
    if (x > m) {   // increasing v per thread: the first maximum is kept
      m = x;
      mi = v;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, m, o);
    const int oi = __shfl_xor_sync(0xffffffffu, mi, o);
    if (om > m || (om == m && oi < mi)) {
      m = om;
      mi = oi;
    }
  }
  if (lane == 0) {
    s_m[warp] = m;
    s_i[warp] = mi;
  }
  __syncthreads();
  m = s_m[0];
  mi = s_i[0];
  for (int w = 1; w < 8; ++w)
    if (s_m[w] > m || (s_m[w] == m && s_i[w] < mi)) {
      m = s_m[w];
      mi = s_i[w];
    }
  float sum = 0.f;
  for (int v = tid; v < V; v += 256) sum += __expf(l[v] - m);
  sum = warp_sum(sum);
  if (lane == 0) s_s[warp] = sum;
  __syncthreads();
  if (tid == 0) {
    float t = 0.f;
    for (int w = 0; w < 8; ++w) t += s_s[w];
    row_key[r] = argmax_key(m, (uint32_t)mi);
    row_p[r] = 1.0f / t;
  }
}

// lens_out[b] = proposals made (or -1 for an utterance that holds its transcript)
__global__ void draft_finish_kernel(DraftArgs A, int* lens_out) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < A.B) lens_out[b] = A.lens[b] < 0 ? -1 : A.n_prop[b];
}

// Attention of the draft's block for the rows of one (utterance, head):
// keys [0, pos + 1) of the self cache (causal) or [row_lo, row_hi) of the
// encoder K/V (cross); fp32 scores, softmax and sums over the bf16 caches.
// Cache layout [B_max][H][t_alloc][64]; q [R][d] fp32; out [R][d] bf16.
__global__ void __launch_bounds__(128) draft_attn_kernel(DraftAttn a) {
  extern __shared__ float s_p[];   // [t_alloc] scores / probabilities
  __shared__ float s_q[64], s_red[8], s_o[2][64];
  const int hh = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int n = a.plan.n_utt_rows[b];
  const int r0 = a.plan.row_start[b];
  const size_t head = ((size_t)b * a.H + hh) * a.t_alloc;
  const __nv_bfloat16* K = a.kc + head * 64;
  const __nv_bfloat16* V = a.vc + head * 64;
  for (int i = 0; i < n; ++i) {
    const int r = r0 + i;
    const int lo = a.causal ? 0 : a.row_lo[r];
    const int hi = a.causal ? a.plan.row_pos[r] + 1 : a.row_hi[r];
    if (bounds_bad(a.status, lo < 0 || hi > a.t_alloc || hi <= lo)) continue;   // uniform over the CTA
    if (tid < 64) s_q[tid] = a.q[(size_t)r * a.d + hh * 64 + tid] * 0.125f;
    __syncthreads();
    float m = -INFINITY;
    for (int j = lo + tid; j < hi; j += 128) {
      const __nv_bfloat162* kr = reinterpret_cast<const __nv_bfloat162*>(K + (size_t)j * 64);
      float s = 0.f;
#pragma unroll 8
      for (int c = 0; c < 32; ++c) {
        const float2 kv = __bfloat1622float2(kr[c]);
        s = fmaf(s_q[2 * c], kv.x, fmaf(s_q[2 * c + 1], kv.y, s));
      }
      s_p[j - lo] = s;
      m = fmaxf(m, s);
    }
    m = warp_max(m);
    if ((tid & 31) == 0) s_red[tid >> 5] = m;
    __syncthreads();
    m = fmaxf(fmaxf(s_red[0], s_red[1]), fmaxf(s_red[2], s_red[3]));
    float l = 0.f;
    for (int j = lo + tid; j < hi; j += 128) {
      const float p = expf(s_p[j - lo] - m);
      s_p[j - lo] = p;
      l += p;
    }
    l = warp_sum(l);
    __syncthreads();
    if ((tid & 31) == 0) s_red[4 + (tid >> 5)] = l;
    __syncthreads();
    l = (s_red[4] + s_red[5]) + (s_red[6] + s_red[7]);
    // output column c = tid & 63 over the keys of half tid >> 6
    const int c = tid & 63, half = tid >> 6;
    float o = 0.f;
    for (int j = lo + half; j < hi; j += 2) o = fmaf(s_p[j - lo], __bfloat162float(V[(size_t)j * 64 + c]), o);
    s_o[half][c] = o;
    __syncthreads();
    if (tid < 64) a.out[(size_t)r * a.d + hh * 64 + tid] = __float2bfloat16_rn((s_o[0][tid] + s_o[1][tid]) / l);
    __syncthreads();
  }
}

}  // namespace

void launch_draft_round_plan(const DraftArgs& a, cudaStream_t st) {
  draft_round_plan_kernel<<<1, DP_T, 0, st>>>(a);
}
void launch_draft_next_plan(const DraftArgs& a, int i, cudaStream_t st) {
  draft_next_plan_kernel<<<1, DP_T, 0, st>>>(a, i);
}
void launch_draft_gather(const DraftArgs& a, int rows_max, cudaStream_t st) {
  const int blocks = std::max(1, std::min(1024, (rows_max * 2 * a.d + 255) / 256));
  draft_gather_kernel<<<blocks, 256, 0, st>>>(a);
}
void launch_draft_prefill_gather(const DraftArgs& a, int rows_max, cudaStream_t st) {
  const int blocks = std::max(1, std::min(1024, (rows_max * 2 * a.d + 255) / 256));
  draft_prefill_gather_kernel<<<blocks, 256, 0, st>>>(a);
  draft_prefill_save_kernel<<<std::max(1, std::min(1024, (a.B * 4 * a.d + 255) / 256)), 256, 0, st>>>(a);
}
void launch_draft_embed(const DraftArgs& a, int rows_max, const void* tok_emb, const void* pos_emb, float* x,
                        cudaStream_t st) {
  const int blocks = std::max(1, std::min(1024, (rows_max * a.d + 255) / 256));
  draft_embed_kernel<<<blocks, 256, 0, st>>>(a, static_cast<const __nv_bfloat16*>(tok_emb),
                                              static_cast<const __nv_bfloat16*>(pos_emb), x);
}
void launch_draft_take(const DraftArgs& a, cudaStream_t st) {
  draft_take_kernel<<<(a.B + 255) / 256, 256, 0, st>>>(a);
}
void launch_draft_finish(const DraftArgs& a, int* lens_out, cudaStream_t st) {
  draft_finish_kernel<<<(a.B + 255) / 256, 256, 0, st>>>(a, lens_out);
}
void launch_draft_softmax(const float* logits, int V, const int* n_rows, int rows_max, unsigned long long* row_key,
                          float* row_p, cudaStream_t st) {
  draft_softmax_kernel<<<std::max(1, rows_max), 256, 0, st>>>(logits, V, n_rows, row_key, row_p);
}
void launch_draft_attn(const DraftAttn& a, cudaStream_t st) {
  static bool configured = false;
  if (!configured) {
    cudaFuncSetAttribute(draft_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 64 * 1024);
    configured = true;
  }
  draft_attn_kernel<<<dim3(a.H, a.B), 128, (size_t)a.t_alloc * 4, st>>>(a);
}

}  // namespace asrspec
