// Row bookkeeping of the verify step: input validation and row layout,
// embeddings, LayerNorm, greedy longest-prefix acceptance with the KV-length
// commit, rollback, and the synthetic draft source used by benchmarks.
#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_rows)

constexpr int PLAN_THREADS = 1024;

// Exclusive block scan of one int per thread (PLAN_THREADS threads).
__device__ int block_excl_scan(int v, int* total) {
  __shared__ int warp_sums[PLAN_THREADS / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = warp_sums[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    warp_sums[lane] = w;
  }
  __syncthreads();
  const int incl = x + (warp > 0 ? warp_sums[warp - 1] : 0);
  *total = warp_sums[PLAN_THREADS / 32 - 1];
  return incl - v;
}

// Verify rows: utterance b contributes lens[b] + 1 rows (pending, then drafts),
// at positions kv_len[b] + i.  A tree verify (parent set) lays out the nodes
// the same way, node i in cache slot kv_len[b] + i, with its position
// kv_len[b] + depth(i) and its ancestors (itself included) as a bit mask.  Any
// invalid input refuses the whole step (n_rows = 0, nothing is written) and
// sets the status word.
__global__ void __launch_bounds__(PLAN_THREADS)
plan_verify_kernel(const int* __restrict__ draft, const int* __restrict__ lens, int k, int B, int vocab, int max_pos,
                   const int* __restrict__ kv_len, const int* __restrict__ pending, const int* __restrict__ ready,
                   RowPlan plan, unsigned long long* row_key, int* status, TrafficArgs tr,
                   unsigned long long* tl, const int* __restrict__ parent) {
  __shared__ int s_err;
  __shared__ unsigned long long s_cnt[4];
  tl_mark(tl, TL_ENTRY);
  tl_mark(tl, TL_WORK);
  if (threadIdx.x == 0) s_err = 0;
  if (threadIdx.x < 4) s_cnt[threadIdx.x] = 0;
  __syncthreads();
  const int b = threadIdx.x;
  int n_b = 0, err = 0;
  if (b < B) {
    const int l = lens[b];
    if (l < -1 || l > k) err |= ST_BAD_LENS;
    else if (l >= 0) {
      if (!ready[b]) err |= ST_NOT_READY;
      if (kv_len[b] + l + 1 > max_pos) err |= ST_CAPACITY;
      for (int i = 0; i < l; ++i) {
        const int t = draft[(size_t)b * k + i];
        if (t < 0 || t >= vocab) err |= ST_BAD_TOKEN;
        if (parent != nullptr) {
          const int p = parent[(size_t)b * k + i];
          if (p < 0 || p > i) err |= ST_BAD_TREE;
        }
      }
      n_b = l + 1;
    }
  }
  if (err) atomicOr(&s_err, err);
  __syncthreads();
  if (s_err) {
    n_b = 0;
    if (threadIdx.x == 0) set_status(status, s_err);
  }
  int total;
  const int start = block_excl_scan(n_b, &total);
  if (b < B) {
    plan.row_start[b] = start;
    plan.n_utt_rows[b] = n_b;
    int depth[32];
    unsigned anc[32];
    for (int i = 0; i < n_b; ++i) {
      const int r = start + i;
      plan.row_b[r] = b;
      plan.row_i[r] = i;
      plan.row_pos[r] = kv_len[b] + i;
      plan.row_tok[r] = i == 0 ? pending[b] : draft[(size_t)b * k + i - 1];
      if (parent != nullptr) {   // n_b <= 32 (k <= 31)
        const int p = i == 0 ? 0 : parent[(size_t)b * k + i - 1];
        depth[i] = i == 0 ? 0 : depth[p] + 1;
        anc[i] = (i == 0 ? 0u : anc[p]) | (1u << i);
        plan.row_epos[r] = kv_len[b] + depth[i];
        plan.row_mask[r] = anc[i];
      } else {
        plan.row_epos[r] = kv_len[b] + i;
      }
      row_key[r] = 0ull;
    }
    if (n_b > 0 && tr.counters) {
      // algorithmic bytes of this utterance: self K/V read over the visible
      // keys of all layers, encoder K/V read by cross-attention, and one
      // anchor-layer key pass
      const unsigned long long es = (unsigned long long)tr.elem_bytes, d = tr.d, L = tr.n_layers;
      const unsigned long long T = (unsigned long long)tr.enc_len[b];
      atomicAdd(&s_cnt[0], 2ull * L * (unsigned long long)(kv_len[b] + n_b) * d * es);
      atomicAdd(&s_cnt[1], 2ull * L * T * d * es);
      atomicAdd(&s_cnt[2], T * d * es);
      atomicAdd(&s_cnt[3], (unsigned long long)n_b);
    }
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    plan.row_start[B] = total;
    *plan.n_rows = total;
    if (tr.counters) {
      atomicAdd(tr.counters + 0, 1ull);
      for (int c = 0; c < 4; ++c) atomicAdd(tr.counters + 1 + c, s_cnt[c]);
    }
  }
  tl_mark(tl, TL_EXIT);
}

// Prefill rows: prompt tokens p0 .. p0+c-1 of every utterance at positions p0 + i.
__global__ void __launch_bounds__(PLAN_THREADS)
plan_prefill_kernel(const int* __restrict__ prompt, int P0, int p0, int c, int B, int vocab,
                    const int* __restrict__ ready, RowPlan plan, int* status) {
  __shared__ int s_err;
  if (threadIdx.x == 0) s_err = 0;
  __syncthreads();
  const int b = threadIdx.x;
  int err = 0;
  if (b < B) {
    if (!ready[b]) err |= ST_NOT_READY;
    for (int i = 0; i < P0; ++i) {
      const int t = prompt[(size_t)b * P0 + i];
      if (t < 0 || t >= vocab) err |= ST_BAD_TOKEN;
    }
  }
  if (err) atomicOr(&s_err, err);
  __syncthreads();
  const int n_b = (b < B && !s_err) ? c : 0;
  if (s_err && threadIdx.x == 0) set_status(status, s_err);
  int total;
  const int start = block_excl_scan(n_b, &total);
  if (b < B) {
    plan.row_start[b] = start;
    plan.n_utt_rows[b] = n_b;
    for (int i = 0; i < n_b; ++i) {
      const int r = start + i;
      plan.row_b[r] = b;
      plan.row_i[r] = i;
      plan.row_pos[r] = p0 + i;
      plan.row_epos[r] = p0 + i;
      plan.row_tok[r] = prompt[(size_t)b * P0 + p0 + i];
    }
  }
  if (threadIdx.x == 0) {
    plan.row_start[B] = total;
    *plan.n_rows = total;
  }
}

void launch_plan_verify(const int* draft, const int* lens, int k, int B, int vocab, int max_pos, const int* kv_len,
                        const int* pending, const int* ready, RowPlan plan, unsigned long long* row_key,
                        int* status, const TrafficArgs& tr, cudaStream_t st, unsigned long long* tl,
                        const int* parent) {
  plan_verify_kernel<<<1, PLAN_THREADS, 0, st>>>(draft, lens, k, B, vocab, max_pos, kv_len, pending, ready, plan,
                                                 row_key, status, tr, tl, parent);
}

void launch_plan_prefill_chunk(const int* prompt, int P0, int p0, int c, int B, int vocab, const int* ready,
                               RowPlan plan, int* status, cudaStream_t st) {
  plan_prefill_kernel<<<1, PLAN_THREADS, 0, st>>>(prompt, P0, p0, c, B, vocab, ready, plan, status);
}

// x[r] = tok_emb[token] + pos_emb[position]  (fp32 residual stream).  With a
// folded first LayerNorm (xg set) also bf16(g * x) and the row's statistics as
// one slice of d features: st_part[r] = (mean, sum of squared deviations).
// One CTA of 128 threads per row (d <= 2048: 16 values per thread).
template <typename T>
__global__ void __launch_bounds__(128)
embed_kernel(const T* __restrict__ tok_emb, const T* __restrict__ pos_emb, RowPlan plan, int d,
             float* __restrict__ x, __nv_bfloat16* __restrict__ xg, const float* __restrict__ gain,
             float2* __restrict__ st_part, unsigned long long* tl, int vocab, int max_pos, int* status) {
  __shared__ float red[4];
  tl_mark(tl, TL_ENTRY);
  pdl_wait();
  tl_mark(tl, TL_WORK);
  pdl_launch();
  const int r = blockIdx.x;
  if (r >= *plan.n_rows) return;   // uniform over the CTA
  const int t = plan.row_tok[r], p = plan.row_epos[r];
  if (bounds_bad(status, t < 0 || t >= vocab || p < 0 || p >= max_pos)) return;   // uniform over the CTA
  float v[16];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < 16; ++i) {
    const int c = threadIdx.x + 128 * i;
    v[i] = c < d ? to_f<T>(tok_emb[(size_t)t * d + c]) + to_f<T>(pos_emb[(size_t)p * d + c]) : 0.f;
    if (c < d) x[(size_t)r * d + c] = v[i];
    s += v[i];
  }
  if (xg != nullptr) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    s = warp_sum(s);
    if (lane == 0) red[warp] = s;
    __syncthreads();
    const float mean = ((red[0] + red[1]) + (red[2] + red[3])) / (float)d;
    __syncthreads();
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
      const int c = threadIdx.x + 128 * i;
      if (c < d) {
        const float dv = v[i] - mean;
        q += dv * dv;
        xg[(size_t)r * d + c] = __float2bfloat16_rn(gain[c] * v[i]);
      }
    }
    q = warp_sum(q);
    if (lane == 0) red[warp] = q;
    __syncthreads();
    if (threadIdx.x == 0) st_part[r] = make_float2(mean, (red[0] + red[1]) + (red[2] + red[3]));
  }
  tl_mark(tl, TL_EXIT);
}

// Folded-LayerNorm constants of a projection W [M][K] (bf16) whose input is
// LayerNorm(x) with gain g and bias b: c1[m] = sum_k W[m][k] g[k],
// c2[m] = sum_k W[m][k] b[k].  One warp per row, fp32 sums.
__global__ void __launch_bounds__(256)
ln_fold_kernel(const __nv_bfloat16* __restrict__ W, const float* __restrict__ g, const float* __restrict__ b, int M,
               int K, float* __restrict__ c1, float* __restrict__ c2) {
  const int m = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
  if (m >= M) return;
  const __nv_bfloat16* w = W + (size_t)m * K;
  float s1 = 0.f, s2 = 0.f;
  for (int k = lane; k < K; k += 32) {
    const float wk = bf2f(w[k]);
    s1 = fmaf(wk, g[k], s1);
    s2 = fmaf(wk, b[k], s2);
  }
  s1 = warp_sum(s1);
  s2 = warp_sum(s2);
  if (lane == 0) {
    c1[m] = s1;
    c2[m] = s2;
  }
}
void launch_ln_fold(const void* W, const float* g, const float* b, int M, int K, float* c1, float* c2,
                    cudaStream_t st) {
  ln_fold_kernel<<<(M + 7) / 8, 256, 0, st>>>(static_cast<const __nv_bfloat16*>(W), g, b, M, K, c1, c2);
}

void launch_embed(const void* tok_emb, const void* pos_emb, int w_bf16, RowPlan plan, int R_max, int d, float* x,
                  cudaStream_t st, bool pdl, unsigned long long* tl, __nv_bfloat16* xg, const float* gain,
                  float2* st_part, int vocab, int max_pos, int* status) {
  if (w_bf16)
    launch_ex(embed_kernel<__nv_bfloat16>, dim3(R_max), dim3(128), 0, st, pdl, 1,
              static_cast<const __nv_bfloat16*>(tok_emb), static_cast<const __nv_bfloat16*>(pos_emb), plan, d, x, xg,
              gain, st_part, tl, vocab, max_pos, status);
  else
    launch_ex(embed_kernel<float>, dim3(R_max), dim3(128), 0, st, pdl, 1, static_cast<const float*>(tok_emb),
              static_cast<const float*>(pos_emb), plan, d, x, xg, gain, st_part, tl, vocab, max_pos, status);
}

// LayerNorm for any d % 4 == 0: a sum pass, a centred sum-of-squares pass over the
// row (L2-resident), then the affine write.
template <typename TO>
__global__ void __launch_bounds__(256)
layernorm_any_kernel(const float* __restrict__ x, const float* __restrict__ g, const float* __restrict__ bta,
                 TO* __restrict__ y, const int* __restrict__ n_rows, int d, unsigned long long* tl) {
  tl_mark(tl, TL_ENTRY);
  pdl_wait();
  tl_mark(tl, TL_WORK);
  pdl_launch();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int r = blockIdx.x * 8 + warp;
  if (r >= *n_rows) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)r * d);
  const int n4 = d >> 2;
  float s = 0.f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = xr[i];
    s += (v.x + v.y) + (v.z + v.w);
  }
  const float mean = warp_sum(s) / (float)d;
  float q = 0.f;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = xr[i];
    const float a = v.x - mean, b = v.y - mean, c = v.z - mean, e = v.w - mean;
    q += (a * a + b * b) + (c * c + e * e);
  }
  const float rstd = rsqrtf(warp_sum(q) / (float)d + 1e-5f);
  TO* yr = y + (size_t)r * d;
  for (int i = lane; i < n4; i += 32) {
    const float4 v = xr[i];
    const float4 gg = reinterpret_cast<const float4*>(g)[i];
    const float4 bb = reinterpret_cast<const float4*>(bta)[i];
    yr[4 * i + 0] = from_f<TO>((v.x - mean) * rstd * gg.x + bb.x);
    yr[4 * i + 1] = from_f<TO>((v.y - mean) * rstd * gg.y + bb.y);
    yr[4 * i + 2] = from_f<TO>((v.z - mean) * rstd * gg.z + bb.z);
    yr[4 * i + 3] = from_f<TO>((v.w - mean) * rstd * gg.w + bb.w);
  }
  tl_mark(tl, TL_EXIT);
}

// LayerNorm, one warp per row, statistics in fp32.  The gain and bias (weights)
// are loaded before the wait on the previous kernel; the row is read once into
// registers (N4 float4 per lane), then mean, centred variance and the affine
// write come from the registers.
template <typename TO, int N4>
__global__ void __launch_bounds__(256)
layernorm_kernel(const float* __restrict__ x, const float* __restrict__ g, const float* __restrict__ bta,
                 TO* __restrict__ y, const int* __restrict__ n_rows, int d, unsigned long long* tl) {
  tl_mark(tl, TL_ENTRY);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float4 gw[N4], bw[N4];
#pragma unroll
  for (int i = 0; i < N4; ++i) {
    gw[i] = __ldg(reinterpret_cast<const float4*>(g) + lane + 32 * i);
    bw[i] = __ldg(reinterpret_cast<const float4*>(bta) + lane + 32 * i);
  }
  pdl_wait();
  tl_mark(tl, TL_WORK);
  pdl_launch();
  const int r = blockIdx.x * 8 + warp;
  if (r >= *n_rows) return;
  const float4* xr = reinterpret_cast<const float4*>(x + (size_t)r * d);
  float4 v[N4];
  float s = 0.f;
#pragma unroll
  for (int i = 0; i < N4; ++i) {
    v[i] = xr[lane + 32 * i];
    s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
  }
  const float mean = warp_sum(s) / (float)d;
  float q = 0.f;
#pragma unroll
  for (int i = 0; i < N4; ++i) {
    const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, e = v[i].w - mean;
    q += (a * a + b * b) + (c * c + e * e);
  }
  const float rstd = rsqrtf(warp_sum(q) / (float)d + 1e-5f);
  TO* yr = y + (size_t)r * d;
#pragma unroll
  for (int i = 0; i < N4; ++i) {
    const int c4 = lane + 32 * i;
    const float4 gg = gw[i], bb = bw[i];
    yr[4 * c4 + 0] = from_f<TO>((v[i].x - mean) * rstd * gg.x + bb.x);
    yr[4 * c4 + 1] = from_f<TO>((v[i].y - mean) * rstd * gg.y + bb.y);
    yr[4 * c4 + 2] = from_f<TO>((v[i].z - mean) * rstd * gg.z + bb.z);
    yr[4 * c4 + 3] = from_f<TO>((v[i].w - mean) * rstd * gg.w + bb.w);
  }
  tl_mark(tl, TL_EXIT);
}

template <typename TO>
static void launch_ln_t(const float* x, const float* g, const float* b, TO* y, const int* n_rows, int R_max, int d,
                        cudaStream_t st, bool pdl, unsigned long long* tl) {
  const dim3 grid((R_max + 7) / 8), block(256);
  switch (d / 128) {   // d is a multiple of 64; d % 128 == 64 rounds up with a guarded tail
    case 1: launch_ex(layernorm_kernel<TO, 1>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 2: launch_ex(layernorm_kernel<TO, 2>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 3: launch_ex(layernorm_kernel<TO, 3>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 4: launch_ex(layernorm_kernel<TO, 4>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 5: launch_ex(layernorm_kernel<TO, 5>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 6: launch_ex(layernorm_kernel<TO, 6>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 8: launch_ex(layernorm_kernel<TO, 8>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 10: launch_ex(layernorm_kernel<TO, 10>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 12: launch_ex(layernorm_kernel<TO, 12>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    case 16: launch_ex(layernorm_kernel<TO, 16>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
    default: launch_ex(layernorm_any_kernel<TO>, grid, block, 0, st, pdl, 1, x, g, b, y, n_rows, d, tl); break;
  }
}

void launch_layernorm(const float* x, const float* g, const float* b, void* y, int y_bf16, const int* n_rows,
                      int R_max, int d, cudaStream_t st, bool pdl, unsigned long long* tl) {
  if (d % 128) {   // widths that are not a whole number of float4 per lane
    const dim3 grid((R_max + 7) / 8);
    if (y_bf16)
      launch_ex(layernorm_any_kernel<__nv_bfloat16>, grid, dim3(256), 0, st, pdl, 1, x, g, b,
                static_cast<__nv_bfloat16*>(y), n_rows, d, tl);
    else
      launch_ex(layernorm_any_kernel<float>, grid, dim3(256), 0, st, pdl, 1, x, g, b, static_cast<float*>(y),
                n_rows, d, tl);
    return;
  }
  if (y_bf16) launch_ln_t(x, g, b, static_cast<__nv_bfloat16*>(y), n_rows, R_max, d, st, pdl, tl);
  else launch_ln_t(x, g, b, static_cast<float*>(y), n_rows, R_max, d, st, pdl, tl);
}

// After a prefill chunk: the rows' K/V are cached, so the committed length moves on.
__global__ void prefill_advance_kernel(int B, int c, const int* n_utt_rows, int* kv_len) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B && n_utt_rows[b] > 0) kv_len[b] += c;
}
__global__ void prefill_finish_kernel(const int* __restrict__ prompt, int P0, int B, int* pending,
                                      const int* ready) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b < B && ready[b]) pending[b] = prompt[(size_t)b * P0 + P0 - 1];
}
void launch_prefill_advance(int B, int c, const int* n_utt_rows, int* kv_len, cudaStream_t st) {
  prefill_advance_kernel<<<(B + 127) / 128, 128, 0, st>>>(B, c, n_utt_rows, kv_len);
}
void launch_prefill_finish(const int* prompt, int P0, int B, int* pending, const int* ready, cudaStream_t st) {
  prefill_finish_kernel<<<(B + 127) / 128, 128, 0, st>>>(prompt, P0, B, pending, ready);
}

// Rollback: all-or-nothing over the batch.
__global__ void __launch_bounds__(PLAN_THREADS)
rollback_kernel(const int* __restrict__ new_len, const int* __restrict__ new_pending, int B, int vocab, int* kv_len,
                int* pending, int* status) {
  __shared__ int s_err;
  if (threadIdx.x == 0) s_err = 0;
  __syncthreads();
  const int b = threadIdx.x;
  int nl = -1, np = 0;
  if (b < B) {
    nl = new_len[b];
    np = new_pending[b];
    if (nl >= 0) {
      if (nl > kv_len[b]) atomicOr(&s_err, ST_CAPACITY);
      if (np < 0 || np >= vocab) atomicOr(&s_err, ST_BAD_TOKEN);
    } else if (nl < -1) {
      atomicOr(&s_err, ST_CAPACITY);
    }
  }
  __syncthreads();
  if (s_err) {
    if (threadIdx.x == 0) set_status(status, s_err);
    return;
  }
  if (b < B && nl >= 0) {
    kv_len[b] = nl;
    pending[b] = np;
  }
}
void launch_rollback(const int* new_len, const int* new_pending, int B, int vocab, int* kv_len, int* pending,
                     int* status, cudaStream_t st) {
  rollback_kernel<<<1, PLAN_THREADS, 0, st>>>(new_len, new_pending, B, vocab, kv_len, pending, status);
}

// Synthetic draft source (workload utility, stands in for a trained draft model).
__global__ void synth_drafts_kernel(const int* __restrict__ truth, const int* __restrict__ total_len,
                                    const int* __restrict__ repl, int k_repl, const int* __restrict__ shift, int k,
                                    int B, int max_pos, const int* __restrict__ kv_len, int* draft_out,
                                    int* lens_out) {
  const int b = blockIdx.x;
  if (b >= B) return;
  const int P = kv_len[b], N = min(total_len[b], max_pos);
  const int l = (P + 1 >= N) ? -1 : min(k, N - P - 2);
  if (threadIdx.x == 0) lens_out[b] = l;
  for (int i = 1 + threadIdx.x; i <= k; i += blockDim.x) {
    int t = 0;
    if (i <= l) {
      const int s = shift[(size_t)b * max_pos + P];
      const int j = (s > 0 && i >= s) ? P + i - 1 : P + i;
      t = truth[(size_t)b * max_pos + j];
      const int rp = repl[((size_t)b * max_pos + P) * k_repl + i - 1];
      if (rp >= 0) t = rp;
    }
    draft_out[(size_t)b * k + i - 1] = t;
  }
}
void launch_synth_drafts(const int* truth, const int* total_len, const int* repl, int k_repl, const int* shift, int k,
                         int B, int max_pos, const int* kv_len, int* draft_out, int* lens_out, cudaStream_t st) {
  synth_drafts_kernel<<<B, 32, 0, st>>>(truth, total_len, repl, k_repl, shift, k, B, max_pos, kv_len, draft_out,
                                        lens_out);
}

// After encode_cache: slot b is ready iff 1 <= enc_len[b] <= t_max; its decoder state is cleared.
__global__ void mark_ready_kernel(const int* __restrict__ enc_len, int B, int t_max, int* ready, int* kv_len,
                                  int* pending, int* status) {
  const int b = blockIdx.x * blockDim.x + threadIdx.x;
  if (b >= B) return;
  const int T = enc_len[b];
  const int ok = (T >= 1 && T <= t_max);
  if (!ok) set_status(status, ST_CAPACITY);
  ready[b] = ok;
  kv_len[b] = 0;
  pending[b] = 0;
}
void launch_mark_ready(const int* enc_len, int B, int t_max, int* ready, int* kv_len, int* pending, int* status,
                       cudaStream_t st) {
  mark_ready_kernel<<<(B + 127) / 128, 128, 0, st>>>(enc_len, B, t_max, ready, kv_len, pending, status);
}


}  // namespace asrspec
