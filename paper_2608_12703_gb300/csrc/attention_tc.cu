// Tensor-core split-KV attention for bf16 caches (self and cross).
//
// Same computation as the SIMT kernel in attention.cu (Sec. 3 "Speculative
// Loop": all rows of a draft block are scored in one pass; self-attention is
// block-causal, cross-attention covers the utterance's encoder frames), laid
// out for GB300:
//   * one CTA = one (utterance, head, split); it streams every S-th 128-key
//     chunk of the utterance's K and V through a ring of TMA tile loads into
//     128-byte-swizzled shared memory (one mbarrier per slot): 2 deep (three
//     CTAs share an SM) for self-attention and for unsplit cross-attention,
//     3 deep when the encoder keys are split over a cluster;
//   * the utterance's rows (up to 16 per m-tile) are the M side of
//     mma.sync m16n8k16 (bf16 in, fp32 accumulate): S = Q K^T, then an online
//     softmax on the accumulator fragments (quad shuffles), then O = P V with
//     P re-used from the S fragments and V fragments from ldmatrix.trans;
//   * each of the 4 warps takes a quarter of every chunk's keys; the CTA
//     combines its warps, and the S splits of one (utterance, head) form a
//     thread-block cluster: CTA q owns output columns [64q/S, 64(q+1)/S), every
//     split pushes its (max, sum, partial output) of those columns into q's
//     shared memory with st.async (bytes counted on q's mbarrier), and q merges
//     them in split order, so the result does not depend on timing;
//   * the TREE variant (self-attention of a tree verify) makes a cache slot at
//     or past kv_len visible to a row only if it holds one of the row's
//     ancestors (plan.row_mask), the tree attention mask of the tree decoder
//     control.
#include <mutex>

#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_attention_tc)

constexpr int TCA_THREADS = 128;

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void mma_bf16_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                                  uint32_t& r3) {
  asm("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// byte offset of (row, 16-byte chunk) in a 128-byte-swizzled tile of 128-byte rows
__device__ __forceinline__ uint32_t sw128(int row, int chunk16) {
  return (uint32_t)(row * 128 + ((chunk16 ^ (row & 7)) << 4));
}

constexpr int TCA_CH = 128;        // keys per chunk (one TMA tile of K and one of V)
constexpr int TCA_TILE = TCA_CH * 128;

template <int MT, int STAGES, bool PUSH>
struct TcaCfg {
  static constexpr int KW = TCA_CH / 4;       // keys per warp per chunk
  static constexpr int NT = KW / 8;           // n-tiles of keys per warp
  static constexpr int RING = STAGES * 2 * TCA_TILE;
  static constexpr int OW = 4 * MT * 16 * 64 * 4;
  static constexpr int PART = (32 * 64 + 64) * 4;   // this CTA's (max, sum, output) per row
  static constexpr int P_OFF = RING > OW ? RING : OW;
  // split merge by push: the partials of this CTA's output columns from every
  // split, [split][row][4 + 64 / S] floats ((max, sum, -, -), output columns)
  static constexpr int RECV_OFF = P_OFF + PART;
  static constexpr int RECV = PUSH ? MT * 16 * 96 * 4 : 0;
  static constexpr int SMEM = 1024 + RECV_OFF + RECV;
};

// One CTA = one (utterance, head, split).  The CTA streams chunks split,
// split + S, split + 2S, ... of the utterance's keys through a TMA ring,
// keeping a running (max, sum, output) per row (online softmax).  With S > 1
// the S splits of a (utterance, head) form one cluster and merge their
// results by pushing them to the CTA that owns each output column (PUSH).
template <int MT, int TCA_STAGES, bool PUSH, bool TREE>
__global__ void __launch_bounds__(TCA_THREADS)
attn_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, AttnArgs a,
               int* status) {
  using C = TcaCfg<MT, TCA_STAGES, PUSH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  float* Ow = reinterpret_cast<float*>(smem);                  // warp partials, after the ring is drained
  float* Pm = reinterpret_cast<float*>(smem + C::P_OFF);       // [32] max
  float* Pl = Pm + 32;                                          // [32] sum
  float* Po = Pm + 64;                                          // [32][64] output (relative to max)
  __shared__ float mw[4][MT * 16], lw[4][MT * 16];
  __shared__ __align__(8) uint64_t bar[TCA_STAGES];
  __shared__ __align__(8) uint64_t rbar;   // PUSH: the other splits' partials have landed

  const int S = gridDim.x, split = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  tl_mark(a.tl, TL_ENTRY);
  const int nr = a.plan.n_utt_rows[b];
  if (nr == 0) {                             // uniform over the cluster
    pdl_wait();
    return;
  }
  const int row0 = a.plan.row_start[b];
  const int n_keys = a.causal ? a.kv_len[b] + nr : a.enc_len[b];
  if (bounds_bad(status, n_keys > a.t_alloc || nr > a.rows_max)) {   // uniform over the cluster
    pdl_wait();
    return;
  }
  const int nc = (n_keys + TCA_CH - 1) / TCA_CH;
  const int n_iter = split < nc ? (nc - split + S - 1) / S : 0;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  const long long rb = ((long long)b * a.H + h) * a.t_alloc;

  if (tid == 0) {
    for (int st = 0; st < TCA_STAGES; ++st) mbar_init(&bar[st], 1);
    if constexpr (PUSH) {   // (S - 1) messages per row: (max, sum) and 64 / S output columns
      mbar_init(&rbar, 1);
      mbar_arrive_expect_tx(&rbar, (uint32_t)((S - 1) * nr * (8 + 4 * (64 / S))));
    }
    fence_mbar_init();
  }
  __syncthreads();
  // PUSH: announce this CTA's receive barrier; the matching wait comes just
  // before the first remote store, long after every split has arrived
  if constexpr (PUSH) cluster_arrive_relaxed();
  auto issue = [&](int i) {
    const int st = i % TCA_STAGES;
    const int key0 = (split + i * S) * TCA_CH;
    uint8_t* ks = smem + st * 2 * TCA_TILE;
    mbar_arrive_expect_tx(&bar[st], 2 * TCA_TILE);
    tma_load_2d(ks, &kmap, &bar[st], 0, (int)(a.k_row0 + rb + key0));
    tma_load_2d(ks + TCA_TILE, &vmap, &bar[st], 0, (int)(a.v_row0 + rb + key0));
  };
  // The encoder K/V cache is constant during a verify call: its first chunks
  // load while the previous kernel finishes.  Self-attention keys include rows
  // the previous kernel appends, so those loads wait for it.
  if (tid == 0 && !a.causal)
    for (int i = 0; i < n_iter && i < TCA_STAGES; ++i) issue(i);
  pdl_wait();
  tl_mark(a.tl, TL_WORK);
  if (tid == 0 && a.causal)
    for (int i = 0; i < n_iter && i < TCA_STAGES; ++i) issue(i);
  pdl_launch();

  // queries of this utterance and head as A fragments, pre-scaled by 1/sqrt(64)
  uint32_t qa[MT][4][4];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
    const int r_lo = mt * 16 + g, r_hi = r_lo + 8;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int c = h * 64 + kk * 16 + half * 8 + 2 * t;
        float2 lo = make_float2(0.f, 0.f), hi = make_float2(0.f, 0.f);
        if (r_lo < nr) lo = *reinterpret_cast<const float2*>(a.q + (size_t)(row0 + r_lo) * a.d + c);
        if (r_hi < nr) hi = *reinterpret_cast<const float2*>(a.q + (size_t)(row0 + r_hi) * a.d + c);
        qa[mt][kk][half * 2 + 0] = pack_bf16(lo.x * 0.125f, lo.y * 0.125f);
        qa[mt][kk][half * 2 + 1] = pack_bf16(hi.x * 0.125f, hi.y * 0.125f);
      }
    }
  }
  int lim[MT][2];   // visible keys per fragment row (exclusive bound)
  unsigned tmask[MT][2];   // TREE: the row's ancestors among the slots from kv_len on
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int r = mt * 16 + g + 8 * e;
      if constexpr (TREE) {
        lim[mt][e] = n_keys;
        tmask[mt][e] = r < nr ? a.plan.row_mask[row0 + r] : 0u;
      } else {
        lim[mt][e] = (a.causal && r < nr) ? min(n_keys, a.plan.row_pos[row0 + r] + 1) : n_keys;
        tmask[mt][e] = 0u;
      }
    }
  const int p_committed = TREE ? a.kv_len[b] : 0;   // TREE: slots below are the committed cache

  float m_run[MT][2], l_run[MT][2], O[MT][8][4];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      m_run[mt][e] = -INFINITY;
      l_run[mt][e] = 0.f;
    }
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) O[mt][nd][0] = O[mt][nd][1] = O[mt][nd][2] = O[mt][nd][3] = 0.f;
  }
  const int q4 = lane >> 3, rr = lane & 7;

  for (int i = 0; i < n_iter; ++i) {
    const int st = i % TCA_STAGES;
    mbar_wait(&bar[st], (i / TCA_STAGES) & 1, status);
    const uint32_t ks_base = smem_u32(smem + st * 2 * TCA_TILE);
    const uint32_t vs_base = ks_base + TCA_TILE;
    const int kbase = (split + i * S) * TCA_CH + warp * C::KW;

    float Sf[MT][C::NT][4];
#pragma unroll
    for (int nt = 0; nt < C::NT; ++nt) {
      const int krow = warp * C::KW + nt * 8 + g;
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) Sf[mt][nt][0] = Sf[mt][nt][1] = Sf[mt][nt][2] = Sf[mt][nt][3] = 0.f;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk) {
        uint32_t b0, b1;
        asm("ld.shared.b32 %0, [%1];" : "=r"(b0) : "r"(ks_base + sw128(krow, 2 * kk) + 4 * t));
        asm("ld.shared.b32 %0, [%1];" : "=r"(b1) : "r"(ks_base + sw128(krow, 2 * kk + 1) + 4 * t));
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) mma_bf16_16816(Sf[mt][nt], qa[mt][kk], b0, b1);
      }
    }
    // online softmax: new running max, rescale, accumulate
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        float cm = -INFINITY;
#pragma unroll
        for (int nt = 0; nt < C::NT; ++nt)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            float& s = Sf[mt][nt][2 * e + j];
            const int key = kbase + nt * 8 + 2 * t + j;
            if (key >= lim[mt][e]) s = -INFINITY;
            if constexpr (TREE)   // a tree slot is visible to the node's descendants only
              if (key >= p_committed && !((tmask[mt][e] >> (key - p_committed)) & 1u)) s = -INFINITY;
            cm = fmaxf(cm, s);
          }
        cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 1));
        cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 2));
        const float m_new = fmaxf(m_run[mt][e], cm);
        const float mu = (m_new == -INFINITY) ? 0.f : m_new;
        const float alpha = __expf(m_run[mt][e] - mu);
        float l = 0.f;
#pragma unroll
        for (int nt = 0; nt < C::NT; ++nt)
#pragma unroll
          for (int j = 0; j < 2; ++j) {
            float& s = Sf[mt][nt][2 * e + j];
            s = __expf(s - mu);
            l += s;
          }
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);
        l_run[mt][e] = l_run[mt][e] * alpha + l;
        m_run[mt][e] = m_new;
#pragma unroll
        for (int nd = 0; nd < 8; ++nd) {
          O[mt][nd][2 * e + 0] *= alpha;
          O[mt][nd][2 * e + 1] *= alpha;
        }
      }
    }
#pragma unroll
    for (int ks = 0; ks < C::KW / 16; ++ks) {
      uint32_t pa[MT][4];
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) {
        pa[mt][0] = pack_bf16(Sf[mt][2 * ks][0], Sf[mt][2 * ks][1]);
        pa[mt][1] = pack_bf16(Sf[mt][2 * ks][2], Sf[mt][2 * ks][3]);
        pa[mt][2] = pack_bf16(Sf[mt][2 * ks + 1][0], Sf[mt][2 * ks + 1][1]);
        pa[mt][3] = pack_bf16(Sf[mt][2 * ks + 1][2], Sf[mt][2 * ks + 1][3]);
      }
      const int vrow = warp * C::KW + ks * 16 + (q4 & 1) * 8 + rr;
#pragma unroll
      for (int nd2 = 0; nd2 < 4; ++nd2) {
        uint32_t r0, r1, r2, r3;
        ldmatrix_x4_trans(vs_base + sw128(vrow, nd2 * 2 + (q4 >> 1)), r0, r1, r2, r3);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          mma_bf16_16816(O[mt][2 * nd2], pa[mt], r0, r1);
          mma_bf16_16816(O[mt][2 * nd2 + 1], pa[mt], r2, r3);
        }
      }
    }
    __syncthreads();   // every warp is done with stage st
    if (tid == 0 && i + TCA_STAGES < n_iter) issue(i + TCA_STAGES);
  }

  // combine the four warps into this CTA's (max, sum, output) per row
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int r = mt * 16 + g + 8 * e;
      if (t == 0) {
        mw[warp][r] = m_run[mt][e];
        lw[warp][r] = l_run[mt][e];
      }
#pragma unroll
      for (int nd = 0; nd < 8; ++nd) {
        float* o = Ow + ((size_t)(warp * MT * 16 + r) * 64 + nd * 8 + 2 * t);
        o[0] = O[mt][nd][2 * e + 0];
        o[1] = O[mt][nd][2 * e + 1];
      }
    }
  }
  __syncthreads();
  for (int e = tid; e < nr * 64; e += TCA_THREADS) {
    const int r = e >> 6, c = e & 63;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, mw[w][r]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float L = 0.f, o = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float f = __expf(mw[w][r] - Mu);
      L += lw[w][r] * f;
      o += Ow[(size_t)(w * MT * 16 + r) * 64 + c] * f;
    }
    Po[r * 64 + c] = o;
    if (c == 0) {
      Pm[r] = M;
      Pl[r] = L;
    }
  }

  // merge the splits of this (utterance, head) in split order
  tl_mark(a.tl, TL_MID);
  __syncwarp();
  if constexpr (PUSH) {
    __syncthreads();   // this CTA's (max, sum, output) per row are complete
    cluster_wait();    // every split's receive barrier is initialised
    const int cw = 64 / S, rs = 4 + cw;   // columns per owner, floats per received row
    float* recv = reinterpret_cast<float*>(smem + C::RECV_OFF);
    for (int pr = tid; pr < S * nr; pr += TCA_THREADS) {
      const int q = pr / nr, r = pr - q * nr;   // owner rank, row
      float* slot = recv + (split * nr + r) * rs;   // this split's row in q's buffer
      const float* o = Po + r * 64 + q * cw;
      if (q == split) {
        slot[0] = Pm[r];
        slot[1] = Pl[r];
        for (int c = 0; c < cw; c += 4) *reinterpret_cast<float4*>(slot + 4 + c) = *reinterpret_cast<const float4*>(o + c);
      } else {
        const uint32_t dst = dsmem_addr(slot, (uint32_t)q), rb_q = dsmem_addr(&rbar, (uint32_t)q);
        st_async_f2(dst, Pm[r], Pl[r], rb_q);
        for (int c = 0; c < cw; c += 4)
          st_async_f4(dst + (uint32_t)(4 + c) * 4u, *reinterpret_cast<const float4*>(o + c), rb_q);
      }
    }
    __syncthreads();                 // this CTA's own rows
    mbar_wait(&rbar, 0, status);     // the other splits' rows
    for (int e = tid; e < nr * cw; e += TCA_THREADS) {
      const int r = e / cw, c = e - r * cw;
      float M = -INFINITY;
      for (int s2 = 0; s2 < S; ++s2) M = fmaxf(M, recv[(s2 * nr + r) * rs]);
      const float Mu = (M == -INFINITY) ? 0.f : M;
      float L = 0.f, o = 0.f;
      for (int s2 = 0; s2 < S; ++s2) {
        const float* row = recv + (s2 * nr + r) * rs;
        const float f = __expf(row[0] - Mu);
        L += row[1] * f;
        o += row[4 + c] * f;
      }
      reinterpret_cast<__nv_bfloat16*>(a.out)[(size_t)(row0 + r) * a.d + h * 64 + split * cw + c] = f2bf(o / L);
      if (a.ml_out && split == 0 && c == 0) {
        a.ml_out[((size_t)(row0 + r) * a.H + h) * 2 + 0] = M;
        a.ml_out[((size_t)(row0 + r) * a.H + h) * 2 + 1] = L;
      }
    }
  } else {
    __syncthreads();
    for (int e = tid; e < nr * 64; e += TCA_THREADS) {
      const int r = e >> 6, c = e & 63;
      const float M = Pm[r];
      reinterpret_cast<__nv_bfloat16*>(a.out)[(size_t)(row0 + r) * a.d + h * 64 + c] = f2bf(Po[r * 64 + c] / Pl[r]);
      if (a.ml_out && c == 0) {
        a.ml_out[((size_t)(row0 + r) * a.H + h) * 2 + 0] = M;
        a.ml_out[((size_t)(row0 + r) * a.H + h) * 2 + 1] = Pl[r];
      }
    }
  }
  tl_mark(a.tl, TL_EXIT);
}

template <int MT, int ST, bool PUSH, bool TREE = false>
static void configure_one() {
  cudaFuncSetAttribute(attn_tc_kernel<MT, ST, PUSH, TREE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       TcaCfg<MT, ST, PUSH>::SMEM);
  if constexpr (PUSH)
    cudaFuncSetAttribute(attn_tc_kernel<MT, ST, PUSH, TREE>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

void configure_attention_tc() {
  static std::once_flag once;
  std::call_once(once, [] {
    configure_one<1, 1, false>();
    configure_one<2, 1, false>();
    configure_one<1, 2, false>();
    configure_one<2, 2, false>();
    configure_one<1, 2, true>();
    configure_one<2, 2, true>();
    configure_one<1, 3, true>();
    configure_one<2, 3, true>();
    configure_one<1, 2, false, true>();
    configure_one<2, 2, false, true>();
    configure_one<1, 2, true, true>();
    configure_one<2, 2, true, true>();
  });
}

template <int MT, int ST, bool PUSH, bool TREE = false>
static void launch_one(const AttnArgs& a, int splits, int* status, cudaStream_t st) {
  launch_ex(attn_tc_kernel<MT, ST, PUSH, TREE>, dim3(splits, a.H, a.B), dim3(TCA_THREADS), TcaCfg<MT, ST, PUSH>::SMEM,
            st, a.pdl, splits, *a.kmap, *a.vmap, a, status);
}

// a.splits CTAs (1, 2, 4 or 8; one cluster) per (utterance, head);
// rows_max > 16 takes two m-tiles.
void launch_attention_tc(const AttnArgs& a, int* status, cudaStream_t st) {
  configure_attention_tc();
  if (a.tree) {   // self-attention of a tree verify (at most 32 nodes per utterance)
    if (a.splits == 1) {
      if (a.rows_max > 16) launch_one<2, 2, false, true>(a, a.splits, status, st);
      else launch_one<1, 2, false, true>(a, a.splits, status, st);
    } else {
      if (a.rows_max > 16) launch_one<2, 2, true, true>(a, a.splits, status, st);
      else launch_one<1, 2, true, true>(a, a.splits, status, st);
    }
    return;
  }
  if (a.splits == 1 && a.causal) {   // self-attention, one CTA per (utterance, head): a one-chunk ring,
    // five CTAs per SM (a few chunks per utterance; 636 vs 721 us per batch-64 round)
    if (a.rows_max > 16) launch_one<2, 1, false, false>(a, a.splits, status, st);
    else launch_one<1, 1, false, false>(a, a.splits, status, st);
  } else if (a.splits == 1) {   // cross-attention, one CTA per (utterance, head): 2-deep ring, three CTAs per SM
    // (54 vs 56 us at batch 64)
    if (a.rows_max > 16) launch_one<2, 2, false, false>(a, a.splits, status, st);
    else launch_one<1, 2, false, false>(a, a.splits, status, st);
  } else if (a.causal) {   // self-attention keys split over a cluster (at most max_pos keys)
    if (a.rows_max > 16) launch_one<2, 2, true, false>(a, a.splits, status, st);
    else launch_one<1, 2, true, false>(a, a.splits, status, st);
  } else {                 // encoder keys split over a cluster: deeper ring per CTA
    if (a.rows_max > 16) launch_one<2, 3, true, false>(a, a.splits, status, st);
    else launch_one<1, 3, true, false>(a, a.splits, status, st);
  }
}

bool make_tmap_cache(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  return make_tmap_bf16(map, base, rows, 64, box_rows);
}

}  // namespace asrspec
