// Tensor-core split-KV attention for bf16 caches (self and cross).
//
// Same computation as the SIMT kernel in attention.cu (Sec. 3 "Speculative
// Loop": all rows of a draft block are scored in one pass; self-attention is
// block-causal, cross-attention covers the utterance's encoder frames), laid
// out for GB300:
//   * one CTA = one (utterance, head, key chunk); its K and V chunks arrive by
//     two TMA tile loads into 128-byte-swizzled shared memory (one mbarrier);
//   * the utterance's rows (up to 16 per m-tile) are the M side of
//     mma.sync m16n8k16 (bf16 in, fp32 accumulate): S = Q K^T, then the
//     softmax on the accumulator fragments (quad shuffles), then O = P V with
//     P re-used from the S fragments and V fragments from ldmatrix.trans;
//   * each of the 4 warps takes a quarter of the chunk's keys; the CTA
//     combines the warps, writes the chunk's (max, sum, output) and the last
//     CTA of the (utterance, head) merges all chunks in chunk order, so the
//     result does not depend on which CTA finishes last.
#include <mutex>

#include "kernels.h"

namespace asrspec {

constexpr int TCA_THREADS = 128;

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ void mma_bf16_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2,
                                                  uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}

// byte offset of (row, 16-byte chunk) in a 128-byte-swizzled tile of 128-byte rows
__device__ __forceinline__ uint32_t sw128(int row, int chunk16) {
  return (uint32_t)(row * 128 + ((chunk16 ^ (row & 7)) << 4));
}

template <int CHUNK, int MT>
struct TcaCfg {
  static constexpr int KW = CHUNK / 4;        // keys per warp
  static constexpr int NT = KW / 8;           // n-tiles of keys per warp
  static constexpr int TILE = CHUNK * 128;    // bytes of one K or V tile
  static constexpr int OW = 4 * MT * 16 * 64 * 4;
  static constexpr int SMEM = 1024 + (2 * TILE > OW ? 2 * TILE : OW);
};

template <int CHUNK, int MT>
__global__ void __launch_bounds__(TCA_THREADS)
attn_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap, AttnArgs a,
               int* status) {
  using C = TcaCfg<CHUNK, MT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* Ks = smem;
  uint8_t* Vs = smem + C::TILE;
  float* Ow = reinterpret_cast<float*>(smem);   // reused after the K/V tiles are consumed
  __shared__ float mw[4][MT * 16], lw[4][MT * 16];
  __shared__ __align__(8) uint64_t bar;
  __shared__ int s_last;

  const int chunk = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const int nr = a.plan.n_utt_rows[b];
  if (nr == 0) return;
  const int row0 = a.plan.row_start[b];
  const int n_keys = a.causal ? a.kv_len[b] + nr : a.enc_len[b];
  const int key0 = chunk * CHUNK;
  if (key0 >= n_keys) return;
  const int nc = (n_keys + CHUNK - 1) / CHUNK;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;

  if (tid == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (tid == 0) {
    const long long rb = ((long long)b * a.H + h) * a.t_alloc + key0;
    mbar_arrive_expect_tx(&bar, 2 * C::TILE);
    tma_load_2d(Ks, &kmap, &bar, 0, (int)(a.k_row0 + rb));
    tma_load_2d(Vs, &vmap, &bar, 0, (int)(a.v_row0 + rb));
  }

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
  // visible key limit per fragment row (exclusive)
  int lim[MT][2];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int r = mt * 16 + g + 8 * e;
      lim[mt][e] = (a.causal && r < nr) ? min(n_keys, a.plan.row_pos[row0 + r] + 1) : n_keys;
    }

  mbar_wait(&bar, 0, status);

  // S = Q K^T over this warp's keys
  float S[MT][C::NT][4];
  const uint32_t ks_base = smem_u32(Ks), vs_base = smem_u32(Vs);
#pragma unroll
  for (int nt = 0; nt < C::NT; ++nt) {
    const int krow = warp * C::KW + nt * 8 + g;
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) S[mt][nt][0] = S[mt][nt][1] = S[mt][nt][2] = S[mt][nt][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t b0, b1;
      asm volatile("ld.shared.b32 %0, [%1];" : "=r"(b0) : "r"(ks_base + sw128(krow, 2 * kk) + 4 * t));
      asm volatile("ld.shared.b32 %0, [%1];" : "=r"(b1) : "r"(ks_base + sw128(krow, 2 * kk + 1) + 4 * t));
#pragma unroll
      for (int mt = 0; mt < MT; ++mt) mma_bf16_16816(S[mt][nt], qa[mt][kk], b0, b1);
    }
  }

  // masked softmax statistics per row (rows g and g + 8 of each m-tile; a quad shares a row)
  float m_row[MT][2], l_row[MT][2];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      float m = -INFINITY;
#pragma unroll
      for (int nt = 0; nt < C::NT; ++nt)
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          const int key = key0 + warp * C::KW + nt * 8 + 2 * t + j;
          float& s = S[mt][nt][2 * e + j];
          if (key >= lim[mt][e]) s = -INFINITY;
          m = fmaxf(m, s);
        }
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 1));
      m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, 2));
      const float mu = (m == -INFINITY) ? 0.f : m;
      float l = 0.f;
#pragma unroll
      for (int nt = 0; nt < C::NT; ++nt)
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          float& s = S[mt][nt][2 * e + j];
          s = (s == -INFINITY) ? 0.f : __expf(s - mu);
          l += s;
        }
      l += __shfl_xor_sync(0xffffffffu, l, 1);
      l += __shfl_xor_sync(0xffffffffu, l, 2);
      m_row[mt][e] = m;
      l_row[mt][e] = l;
    }
  }

  // O = P V over this warp's keys
  float O[MT][8][4];
#pragma unroll
  for (int mt = 0; mt < MT; ++mt)
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) O[mt][nd][0] = O[mt][nd][1] = O[mt][nd][2] = O[mt][nd][3] = 0.f;
  const int q4 = lane >> 3, rr = lane & 7;
#pragma unroll
  for (int ks = 0; ks < C::KW / 16; ++ks) {
    uint32_t pa[MT][4];
#pragma unroll
    for (int mt = 0; mt < MT; ++mt) {
      pa[mt][0] = pack_bf16(S[mt][2 * ks][0], S[mt][2 * ks][1]);
      pa[mt][1] = pack_bf16(S[mt][2 * ks][2], S[mt][2 * ks][3]);
      pa[mt][2] = pack_bf16(S[mt][2 * ks + 1][0], S[mt][2 * ks + 1][1]);
      pa[mt][3] = pack_bf16(S[mt][2 * ks + 1][2], S[mt][2 * ks + 1][3]);
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

  // combine the four warps of the CTA
  __syncthreads();   // every warp is done with the K/V tiles; Ow reuses them
#pragma unroll
  for (int mt = 0; mt < MT; ++mt) {
#pragma unroll
    for (int e = 0; e < 2; ++e) {
      const int r = mt * 16 + g + 8 * e;
      if (t == 0) {
        mw[warp][r] = m_row[mt][e];
        lw[warp][r] = l_row[mt][e];
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
  float* part = a.part + (((size_t)b * a.H + h) * a.n_chunks + chunk) * a.k1 * 66;
  for (int e = tid; e < nr * 64; e += TCA_THREADS) {
    const int r = e >> 6, c = e & 63;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 4; ++w) M = fmaxf(M, mw[w][r]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float L = 0.f, o = 0.f;
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const float f = (mw[w][r] == -INFINITY) ? 0.f : __expf(mw[w][r] - Mu);
      L += lw[w][r] * f;
      o += Ow[(size_t)(w * MT * 16 + r) * 64 + c] * f;
    }
    part[r * 66 + c] = o;
    if (c == 0) {
      part[r * 66 + 64] = M;
      part[r * 66 + 65] = L;
    }
  }

  // the last CTA of this (utterance, head) merges the chunks in chunk order
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(a.tickets + b * a.H + h, 1) == nc - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // chunk weights first (one thread per (row, chunk), all loads in flight at
  // once), then every output element as one pass over the chunks
  const float* pb = a.part + ((size_t)b * a.H + h) * a.n_chunks * a.k1 * 66;
  const size_t cstride = (size_t)a.k1 * 66;
  float* wgt = Ow;                               // [nr][nc] chunk weights, then [nr] sums
  float* Lsum = Ow + MT * 16 * 32;
  for (int e = tid; e < nr * nc; e += TCA_THREADS) {
    const int r = e / nc, ci = e - r * nc;
    wgt[r * 32 + ci] = __ldcg(pb + ci * cstride + r * 66 + 64);
    Lsum[r * 32 + ci] = __ldcg(pb + ci * cstride + r * 66 + 65);
  }
  __syncthreads();
  if (tid < nr) {
    float M = -INFINITY;
    for (int ci = 0; ci < nc; ++ci) M = fmaxf(M, wgt[tid * 32 + ci]);
    float L = 0.f;
    for (int ci = 0; ci < nc; ++ci) {
      const float mc = wgt[tid * 32 + ci];
      const float f = (mc == -INFINITY) ? 0.f : __expf(mc - M);
      L += Lsum[tid * 32 + ci] * f;
      wgt[tid * 32 + ci] = f;
    }
    for (int ci = 0; ci < nc; ++ci) wgt[tid * 32 + ci] /= L;
    if (a.ml_out) {
      a.ml_out[((size_t)(row0 + tid) * a.H + h) * 2 + 0] = M;
      a.ml_out[((size_t)(row0 + tid) * a.H + h) * 2 + 1] = L;
    }
  }
  __syncthreads();
  for (int e = tid; e < nr * 64; e += TCA_THREADS) {
    const int r = e >> 6, c = e & 63;
    float o = 0.f;
    int ci = 0;
    for (; ci + 4 <= nc; ci += 4) {
      const float p0 = __ldcg(pb + (ci + 0) * cstride + r * 66 + c);
      const float p1 = __ldcg(pb + (ci + 1) * cstride + r * 66 + c);
      const float p2 = __ldcg(pb + (ci + 2) * cstride + r * 66 + c);
      const float p3 = __ldcg(pb + (ci + 3) * cstride + r * 66 + c);
      o += p0 * wgt[r * 32 + ci];
      o += p1 * wgt[r * 32 + ci + 1];
      o += p2 * wgt[r * 32 + ci + 2];
      o += p3 * wgt[r * 32 + ci + 3];
    }
    for (; ci < nc; ++ci) o += __ldcg(pb + ci * cstride + r * 66 + c) * wgt[r * 32 + ci];
    reinterpret_cast<__nv_bfloat16*>(a.out)[(size_t)(row0 + r) * a.d + h * 64 + c] = f2bf(o);
  }
  if (tid == 0) a.tickets[b * a.H + h] = 0;
}

template <int CHUNK, int MT>
static void configure_one() {
  cudaFuncSetAttribute(attn_tc_kernel<CHUNK, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       TcaCfg<CHUNK, MT>::SMEM);
}

void configure_attention_tc() {
  static std::once_flag once;
  std::call_once(once, [] {
    configure_one<128, 1>();
    configure_one<128, 2>();
    configure_one<256, 1>();
    configure_one<256, 2>();
  });
}

template <int CHUNK, int MT>
static void launch_one(const AttnArgs& a, int* status, cudaStream_t st) {
  dim3 grid((a.t_alloc + CHUNK - 1) / CHUNK, a.H, a.B);
  attn_tc_kernel<CHUNK, MT><<<grid, TCA_THREADS, TcaCfg<CHUNK, MT>::SMEM, st>>>(*a.kmap, *a.vmap, a, status);
}

// chunk: 128 or 256 keys; rows_max > 16 takes two m-tiles
void launch_attention_tc(const AttnArgs& a, int* status, cudaStream_t st) {
  configure_attention_tc();
  const bool two = a.rows_max > 16;
  if (a.chunk == 128) {
    if (two) launch_one<128, 2>(a, status, st);
    else launch_one<128, 1>(a, status, st);
  } else {
    if (two) launch_one<256, 2>(a, status, st);
    else launch_one<256, 1>(a, status, st);
  }
}

bool make_tmap_cache(CUtensorMap* map, const void* base, uint64_t rows, uint32_t box_rows) {
  return make_tmap_bf16(map, base, rows, 64, box_rows);
}

}  // namespace asrspec
