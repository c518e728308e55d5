// Split-KV attention over the verify rows, and the re-anchoring readout.
//
// Self-attention (Sec. 3 "Speculative Loop": the target checks the whole
// draft block in one pass): row i of utterance b sits at position P_b + i and
// attends to cached keys 0 .. P_b + i, i.e. the committed cache plus rows
// 0..i of its own block (a block-causal mask).  Cross-attention: every row
// attends to the utterance's enc_len[b] encoder frames.
//
// One CTA takes one (utterance, head, key chunk): it stages the chunk's K and V
// in shared memory once and serves every row of that utterance from it.  Each
// chunk leaves (max, sum, unnormalised output) per row; a merge kernel
// combines the chunks in chunk order.
//
// Anchor (Sec. 5 "Verification-Attention Correction"; App. "Runtime anchor
// construction"): the head mean of the per-head softmax attention of one row
// at the anchor layer, recomputed from the cached keys with the (max, sum) that
// the attention pass left, then its peak frame.
#include <mutex>

#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_attention)

constexpr float ATTN_SCALE = 0.125f;  // 1 / sqrt(64)

// q . k over 64 dims, visiting the 32 element pairs starting at pair (j mod 32):
// consecutive rows of a shared-memory tile then hit different banks.  The same
// order is used by the anchor readout so both compute identical scores.
template <typename T>
__device__ __forceinline__ float dot64_rot(const float* q, const T* k, int j) {
  float acc = 0.f;
#pragma unroll 8
  for (int t = 0; t < 32; ++t) {
    const int w = (t + j) & 31;
    acc = fmaf(q[2 * w], to_f<T>(k[2 * w]), acc);
    acc = fmaf(q[2 * w + 1], to_f<T>(k[2 * w + 1]), acc);
  }
  return acc;
}

constexpr int ATTN_THREADS = 256;
constexpr int ATTN_MAX_ROWS = 32;   // rows per utterance served by one CTA (k + 1 <= 32)

template <typename T, int CHUNK>
__global__ void __launch_bounds__(ATTN_THREADS) attn_chunk_kernel(AttnArgs a) {
  extern __shared__ __align__(16) uint8_t smem[];
  T* Ks = reinterpret_cast<T*>(smem);
  T* Vs = Ks + CHUNK * 64;
  float* Qs = reinterpret_cast<float*>(Vs + CHUNK * 64);     // [rows][64]
  float* S = Qs + ATTN_MAX_ROWS * 64;                        // [rows][CHUNK]
  __shared__ float s_m[ATTN_MAX_ROWS], s_l[ATTN_MAX_ROWS];

  const int chunk = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int nr = a.plan.n_utt_rows[b];
  if (nr == 0) return;
  const int row0 = a.plan.row_start[b];
  const int n_keys = a.causal ? a.kv_len[b] + nr : a.enc_len[b];
  if (bounds_bad(a.status, n_keys > a.t_alloc || n_keys > a.n_chunks * a.chunk)) return;
  const int key0 = chunk * CHUNK;
  if (key0 >= n_keys) return;
  const int nk = min(CHUNK, n_keys - key0);
  const int tid = threadIdx.x;

  // stage K, V (contiguous [nk][64] for this (b, h)) and the rows' queries
  const size_t base = (((size_t)b * a.H + h) * a.t_alloc + key0) * 64;
  const T* gK = static_cast<const T*>(a.kc) + base;
  const T* gV = static_cast<const T*>(a.vc) + base;
  constexpr int VEC = 16 / sizeof(T);
  const int nvec = nk * 64 / VEC;
  for (int v = tid; v < nvec; v += ATTN_THREADS) {
    reinterpret_cast<uint4*>(Ks)[v] = __ldg(reinterpret_cast<const uint4*>(gK) + v);
    reinterpret_cast<uint4*>(Vs)[v] = __ldg(reinterpret_cast<const uint4*>(gV) + v);
  }
  for (int e = tid; e < nr * 64; e += ATTN_THREADS) {
    const int i = e >> 6, c = e & 63;
    Qs[e] = a.q[(size_t)(row0 + i) * a.d + h * 64 + c];
  }
  __syncthreads();

  // scores
  for (int e = tid; e < nr * nk; e += ATTN_THREADS) {
    const int i = e / nk, j = e - i * nk;
    const int key = key0 + j;
    float s = dot64_rot<T>(Qs + i * 64, Ks + j * 64, j) * ATTN_SCALE;
    if (a.causal && key > a.plan.row_pos[row0 + i]) s = -INFINITY;
    S[i * CHUNK + j] = s;
  }
  __syncthreads();

  // per-row max and sum over the chunk (one warp per row)
  const int warp = tid >> 5, lane = tid & 31;
  for (int i = warp; i < nr; i += ATTN_THREADS / 32) {
    float m = -INFINITY;
    for (int j = lane; j < nk; j += 32) m = fmaxf(m, S[i * CHUNK + j]);
    m = warp_max(m);
    float l = 0.f;
    for (int j = lane; j < nk; j += 32) {
      const float s = S[i * CHUNK + j];
      const float p = (s == -INFINITY) ? 0.f : expf(s - m);
      S[i * CHUNK + j] = p;
      l += p;
    }
    l = warp_sum(l);
    if (lane == 0) {
      s_m[i] = m;
      s_l[i] = l;
    }
  }
  __syncthreads();

  // unnormalised output of the chunk
  float* part = a.part + (((size_t)b * a.H + h) * a.n_chunks + chunk) * a.k1 * 66;
  for (int e = tid; e < nr * 64; e += ATTN_THREADS) {
    const int i = e >> 6, c = e & 63;
    float o = 0.f;
    const float* p = S + i * CHUNK;
    for (int j = 0; j < nk; ++j) o = fmaf(p[j], to_f<T>(Vs[j * 64 + c]), o);
    part[i * 66 + c] = o;
  }
  if (tid < nr) {
    part[tid * 66 + 64] = s_m[tid];
    part[tid * 66 + 65] = s_l[tid];
  }
}

// Merge the chunks of one (row, head) in chunk order.
__global__ void attn_merge_kernel(AttnArgs a, int chunk_len) {
  const int i = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int nr = a.plan.n_utt_rows[b];
  if (i >= nr) return;
  const int r = a.plan.row_start[b] + i;
  const int n_keys = a.causal ? a.kv_len[b] + nr : a.enc_len[b];
  if (bounds_bad(a.status, n_keys > a.t_alloc || n_keys > a.n_chunks * chunk_len)) return;
  const int nc = (n_keys + chunk_len - 1) / chunk_len;
  const float* part = a.part + ((size_t)b * a.H + h) * a.n_chunks * a.k1 * 66 + (size_t)i * 66;
  const size_t cstride = (size_t)a.k1 * 66;
  float M = -INFINITY;
  for (int c = 0; c < nc; ++c) M = fmaxf(M, part[c * cstride + 64]);
  float l = 0.f, o = 0.f;
  const int cc = threadIdx.x;   // 64 threads, one per output dim
  for (int c = 0; c < nc; ++c) {
    const float m_c = part[c * cstride + 64];
    const float w = (m_c == -INFINITY) ? 0.f : expf(m_c - M);
    l += part[c * cstride + 65] * w;
    o += part[c * cstride + cc] * w;
  }
  o = o / l;
  const size_t oi = (size_t)r * a.d + h * 64 + cc;
  if (a.out_bf16) reinterpret_cast<__nv_bfloat16*>(a.out)[oi] = f2bf(o);
  else reinterpret_cast<float*>(a.out)[oi] = o;
  if (a.ml_out && cc == 0) {
    a.ml_out[((size_t)r * a.H + h) * 2 + 0] = M;
    a.ml_out[((size_t)r * a.H + h) * 2 + 1] = l;
  }
}

template <typename T, int CHUNK>
static size_t attn_smem() {
  return (size_t)2 * CHUNK * 64 * sizeof(T) + (size_t)ATTN_MAX_ROWS * 64 * 4 + (size_t)ATTN_MAX_ROWS * CHUNK * 4;
}

void configure_attention() {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(attn_chunk_kernel<__nv_bfloat16, 256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attn_smem<__nv_bfloat16, 256>());
    cudaFuncSetAttribute(attn_chunk_kernel<float, 128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         (int)attn_smem<float, 128>());
  });
}

template <typename T, int CHUNK>
static void launch_attn_t(const AttnArgs& a, cudaStream_t st) {
  const size_t sm = attn_smem<T, CHUNK>();
  dim3 grid(a.n_chunks, a.H, a.B);
  attn_chunk_kernel<T, CHUNK><<<grid, ATTN_THREADS, sm, st>>>(a);
  dim3 mgrid(a.k1, a.H, a.B);
  attn_merge_kernel<<<mgrid, 64, 0, st>>>(a, CHUNK);
}

void launch_attention(const AttnArgs& a, cudaStream_t st) {
  configure_attention();
  if (a.kv_bf16) launch_attn_t<__nv_bfloat16, 256>(a, st);
  else launch_attn_t<float, 128>(a, st);
}

int attn_chunk_len(int kv_bf16) { return kv_bf16 ? 256 : 128; }

// ---------------------------------------------------------------------------
// Acceptance, commit and anchor readout, fused
// ---------------------------------------------------------------------------
// One CTA per (FB encoder frames, utterance).  The anchor layer's encoder keys
// do not change during a verify call, so each CTA starts copying its frames'
// keys (all heads) into shared memory before it waits for the LM head.  Then
// one warp recomputes the accepted length n from the per-row argmax keys (one
// ballot); the first CTA commits: accepted, bonus, kv_len += 1 + n, pending =
// bonus (Sec. 3 "Speculative Loop"; a round advances 1 + L tokens, App.
// "Correction and Cost").  Each CTA then evaluates, for its frames, the head
// mean of the per-head softmax attention of row n at the anchor layer (Sec. 5
// "Verification-Attention Correction"), with the (max, sum) the attention pass
// left: a fixed-order head sum per frame, an order-free atomicMax of packed
// (value, frame) keys, and the last CTA of the utterance (ticket) writes the
// peak frame.  Only CTAs that hold frames (and the first) take part.  A tree
// verify (A.parent set; App. tree decoder control) replaces the prefix ballot
// by a walk: from the root, one ballot per step finds the first child whose
// token is the current node's argmax; the path goes to A.path and the anchor
// row is the path's last node.
constexpr int ANCHOR_HMAX = 32;   // heads (d_model <= 2048)

template <typename T>
struct AnchorCfg {
  static constexpr int FB = sizeof(T) == 2 ? 16 : 8;   // frames per CTA (40 KB of keys for 20 heads)
  static constexpr int ROW_BYTES = 64 * (int)sizeof(T);
  static constexpr int SMEM = ANCHOR_HMAX * FB * ROW_BYTES;   // keys [H][FB][64]; <= 64 KB
};

template <typename T>
__global__ void __launch_bounds__(256)
accept_anchor_kernel(AcceptAnchorArgs A) {
  using C = AnchorCfg<T>;
  constexpr int FB = C::FB;
  extern __shared__ __align__(128) uint8_t anchor_keys[];
  __shared__ float qs[ANCHOR_HMAX][64];
  __shared__ float ph[ANCHOR_HMAX][FB + 1];
  __shared__ float sM[ANCHOR_HMAX], sL[ANCHOR_HMAX];
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_n, s_node, s_last;
  tl_mark(A.tl, TL_ENTRY);
  const int b = blockIdx.y, f0 = blockIdx.x * FB, tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int H = A.H;
  const int n_frames = A.enc_len[b];                  // constant during a verify call
  if (blockIdx.x > 0 && f0 >= n_frames) {             // no frames here
    pdl_wait();
    return;
  }
  const int rows = min(FB, n_frames - f0) > 0 ? min(FB, n_frames - f0) : 0;
  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    if (rows > 0) {
      mbar_arrive_expect_tx(&bar, (uint32_t)(H * rows * C::ROW_BYTES));
      const char* kc = static_cast<const char*>(A.kc);
      for (int h = 0; h < H; ++h)
        bulk_load(anchor_keys + h * FB * C::ROW_BYTES,
                  kc + (((size_t)b * H + h) * A.t_alloc + f0) * C::ROW_BYTES, (uint32_t)(rows * C::ROW_BYTES), &bar);
    }
  }
  pdl_wait();
  tl_mark(A.tl, TL_WORK);
  pdl_launch();
  const int nr = A.plan.n_utt_rows[b];
  if (nr == 0) {                                      // uniform over the utterance's CTAs
    if (blockIdx.x == 0 && tid == 0 && A.path != nullptr)
      for (int j = 0; j < A.k; ++j) A.path[(size_t)b * A.k + j] = -1;
    if (blockIdx.x == 0 && tid == 0) {
      A.accepted[b] = 0;
      A.bonus[b] = -1;
      A.kv_len_out[b] = A.kv_len[b];
      A.anchor_out[b] = -1;
      A.restart[b] = 0;
    }
    __syncthreads();
    if (rows > 0) mbar_wait(&bar, 0, A.status);       // no CTA leaves with copies in flight
    return;
  }
  const int r0 = A.plan.row_start[b];
  if (warp == 0 && A.parent != nullptr) {
    // tree: from the root, follow the first child whose token is the target's
    // argmax at its parent; n accepted nodes, the bonus is the argmax at the
    // last of them (lane j < nr holds node j: its argmax, and for j >= 1 its
    // token and parent)
    const int l = nr - 1;
    const unsigned long long key = lane < nr ? A.row_key[r0 + lane] : 0ull;
    const int tok = (int)argmax_index(key);
    const int my_tok = (lane >= 1 && lane <= l) ? A.draft[(size_t)b * A.k + lane - 1] : -1;
    const int my_par = (lane >= 1 && lane <= l) ? A.parent[(size_t)b * A.k + lane - 1] : -1;
    int c = 0, n = 0;
    while (true) {   // at most l steps: every step moves to a deeper node
      const int g = __shfl_sync(0xffffffffu, tok, c);
      const unsigned hit = __ballot_sync(0xffffffffu, my_par == c && my_tok == g);
      if (hit == 0u) break;
      c = __ffs(hit) - 1;
      if (lane == 0 && blockIdx.x == 0) A.path[(size_t)b * A.k + n] = c;
      ++n;
    }
    const int g = __shfl_sync(0xffffffffu, tok, c);
    const unsigned kids = __ballot_sync(0xffffffffu, my_par == c);   // the last node's children
    if (lane == 0) {
      s_n = n;
      s_node = c;
      if (blockIdx.x == 0) {
        A.restart[b] = kids != 0u;   // a child of the last node was rejected
        for (int j = n; j < A.k; ++j) A.path[(size_t)b * A.k + j] = -1;
        const int nl = A.kv_len[b] + 1 + n;
        A.accepted[b] = n;
        A.bonus[b] = g;
        A.kv_len[b] = nl;
        A.kv_len_out[b] = nl;
        A.pending[b] = g;
      }
    }
  } else if (warp == 0) {
    // draft i is accepted while it equals the target's argmax at row i (i < nr - 1)
    const int l = nr - 1;
    const unsigned long long key = lane < nr ? A.row_key[r0 + lane] : 0ull;
    const int tok = (int)argmax_index(key);
    const bool match = lane < l && A.draft[(size_t)b * A.k + lane] == tok;
    const unsigned mism = ~__ballot_sync(0xffffffffu, match);
    const int n = min(__ffs(mism) - 1, l);
    const int g = __shfl_sync(0xffffffffu, tok, n);
    if (lane == 0) {
      s_n = n;
      s_node = n;
      if (blockIdx.x == 0) {
        const int nl = A.kv_len[b] + 1 + n;
        A.accepted[b] = n;
        A.bonus[b] = g;
        A.kv_len[b] = nl;
        A.kv_len_out[b] = nl;
        A.pending[b] = g;
        A.restart[b] = n < l;   // a draft was rejected: the next round restarts
      }
    }
  }
  __syncthreads();
  const int r = r0 + s_node;   // the row that produced the bonus token
  for (int e = tid; e < H * 64; e += blockDim.x) {
    const float v = A.q_anchor[(size_t)r * A.d + e];
    // the tensor-core attention scored bf16(q / 8) against the bf16 keys
    qs[e >> 6][e & 63] = A.kv_bf16 ? bf2f(f2bf(v * 0.125f)) : v;
  }
  if (tid < H) {
    sM[tid] = A.ml[((size_t)r * H + tid) * 2 + 0];
    sL[tid] = A.ml[((size_t)r * H + tid) * 2 + 1];
  }
  __syncthreads();
  if (rows > 0) mbar_wait(&bar, 0, A.status);
  // scores: 8 lanes per (head, frame), each over 8 of the 64 dimensions, so
  // that a warp reads four consecutive key rows of shared memory at once
  const int g = lane >> 3, c = lane & 7;
  const float scale = A.kv_bf16 ? 1.f : ATTN_SCALE;
  for (int base = warp * 4; base < H * FB; base += 32) {   // uniform over the warp
    const int p = base + g;
    const int h = p / FB, fr = p - h * FB;
    const bool ok = p < H * FB && fr < rows;
    float s = 0.f;
    if (ok) {
      const uint8_t* kr = anchor_keys + (h * FB + fr) * C::ROW_BYTES;
      const float* qh = qs[h] + 8 * c;
      if constexpr (sizeof(T) == 2) {
        const uint4 kv = *reinterpret_cast<const uint4*>(kr + 16 * c);
        const __nv_bfloat162* k2 = reinterpret_cast<const __nv_bfloat162*>(&kv);
#pragma unroll
        for (int w = 0; w < 4; ++w) {
          const float2 kf = __bfloat1622float2(k2[w]);
          s = fmaf(qh[2 * w], kf.x, s);
          s = fmaf(qh[2 * w + 1], kf.y, s);
        }
      } else {
        const float4 k0 = *reinterpret_cast<const float4*>(kr + 32 * c);
        const float4 k1 = *reinterpret_cast<const float4*>(kr + 32 * c + 16);
        s = fmaf(qh[0], k0.x, s); s = fmaf(qh[1], k0.y, s); s = fmaf(qh[2], k0.z, s); s = fmaf(qh[3], k0.w, s);
        s = fmaf(qh[4], k1.x, s); s = fmaf(qh[5], k1.y, s); s = fmaf(qh[6], k1.z, s); s = fmaf(qh[7], k1.w, s);
      }
    }
    s += __shfl_xor_sync(0xffffffffu, s, 1);
    s += __shfl_xor_sync(0xffffffffu, s, 2);
    s += __shfl_xor_sync(0xffffffffu, s, 4);
    if (c == 0 && p < H * FB) ph[h][fr] = ok ? expf(s * scale - sM[h]) / sL[h] : 0.f;
  }
  __syncthreads();
  if (warp == 0) {
    float pbar = 0.f;
    const int fr = lane < FB ? lane : 0;
    for (int h = 0; h < H; ++h) pbar += ph[h][fr];
    pbar /= (float)H;
    if (lane < rows) A.profile[(size_t)b * A.t_alloc + f0 + lane] = pbar;
    unsigned long long key = lane < rows ? argmax_key(pbar, (uint32_t)(f0 + lane)) : 0ull;
    key = warp_max_u64(key);
    if (lane == 0) {
      const int n_cta = n_frames > FB ? (n_frames + FB - 1) / FB : 1;   // CTAs of this utterance that take part
      atomicMax(A.frame_key + b, key);
      __threadfence();
      s_last = (atomicAdd(A.tickets + b, 1) == n_cta - 1);
      if (s_last) {
        __threadfence();
        const unsigned long long fk = atomicExch(A.frame_key + b, 0ull);
        A.anchor_out[b] = (int)argmax_index(fk);
        A.tickets[b] = 0;
      }
    }
  }
  tl_mark(A.tl, TL_EXIT);
}

void launch_accept_anchor(const AcceptAnchorArgs& A, cudaStream_t st) {
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(accept_anchor_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         AnchorCfg<__nv_bfloat16>::SMEM);
    cudaFuncSetAttribute(accept_anchor_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         AnchorCfg<float>::SMEM);
  });
  if (A.kv_bf16) {
    using C = AnchorCfg<__nv_bfloat16>;
    dim3 grid((A.t_alloc + C::FB - 1) / C::FB, A.B);
    launch_ex(accept_anchor_kernel<__nv_bfloat16>, grid, dim3(256), (size_t)A.H * C::FB * C::ROW_BYTES, st, A.pdl, 1,
              A);
  } else {
    using C = AnchorCfg<float>;
    dim3 grid((A.t_alloc + C::FB - 1) / C::FB, A.B);
    launch_ex(accept_anchor_kernel<float>, grid, dim3(256), (size_t)A.H * C::FB * C::ROW_BYTES, st, A.pdl, 1, A);
  }
}

// Tree verify commit: one warp per (utterance, layer, head) moves the accepted
// path's K and V rows from the nodes' slots kv_len_old + path[j] to the
// positions kv_len_old + j + 1, in depth order.  Path nodes have increasing
// slots, path[j] >= j + 1, so a slot is overwritten only after the copy that
// reads it (each lane moves the same 4 bytes of every row, in program order).
__global__ void __launch_bounds__(256)
tree_commit_kernel(const int* __restrict__ path, int k, const int* __restrict__ accepted,
                   const int* __restrict__ kv_len, int B, int L, int H, int max_pos, int b_max, uint32_t* kself,
                   uint32_t* vself, int* status) {
  const int w = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
  if (w >= B * L * H) return;
  const int b = w / (L * H), rem = w - b * L * H, l = rem / H, h = rem - l * H;
  const int n = accepted[b];
  if (n <= 0) return;
  const int P = kv_len[b] - 1 - n;
  const size_t head = (((size_t)l * b_max + b) * H + h) * (size_t)max_pos;   // row 0 of (layer, b, head)
  uint32_t* K = kself + head * 32;   // 64 bf16 = 32 words per row
  uint32_t* V = vself + head * 32;
  for (int j = 0; j < n; ++j) {
    const int src = path[(size_t)b * k + j];
    if (bounds_bad(status, P < 0 || src < 1 || P + max(src, j + 1) >= max_pos)) return;
    if (src == j + 1) continue;
    K[(size_t)(P + j + 1) * 32 + lane] = K[(size_t)(P + src) * 32 + lane];
    V[(size_t)(P + j + 1) * 32 + lane] = V[(size_t)(P + src) * 32 + lane];
  }
}

void launch_tree_commit(const int* path, int k, const int* accepted, const int* kv_len, int B, int L, int H,
                        int max_pos, int b_max, void* kself, void* vself, int es, int* status, cudaStream_t st) {
  if (es != 2) return;   // tree verify runs on bf16 caches only (the ABI refuses others)
  const long long threads = 32ll * B * L * H;
  tree_commit_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, st>>>(
      path, k, accepted, kv_len, B, L, H, max_pos, b_max, static_cast<uint32_t*>(kself), static_cast<uint32_t*>(vself),
      status);
}

}  // namespace asrspec
