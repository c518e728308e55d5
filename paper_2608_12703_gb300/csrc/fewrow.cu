// Few-row verify layers (at most 9 scored rows, e.g. batch 1 with k = 8).
//
// A verification step at batch 1 moves the whole decoder's weights for 9
// rows (Sec. 3 "Speculative Loop": the target scores the draft block in one
// pass), so every projection is matrix-vector-like and the step is a chain of
// dependent exchanges: what a launch costs is its exchange latency, not its
// arithmetic.  Six launches per layer:
//   qkv_self   LayerNorm 1 -> QKV projection of one head per thread-block
//              cluster -> the head's q, k, v gathered in every CTA of the
//              cluster (distributed shared memory) -> self-attention over the
//              head's cache, keys split over the cluster, partials merged in
//              key order by one CTA; the new rows' K/V also go to the cache;
//   out        self-attention output projection + residual (GEMV);
//   q_cross    LayerNorm 2 -> cross query of one head per cluster -> q
//              gathered in the cluster -> cross-attention over the encoder
//              frames split over the cluster, merged in split order;
//   out        cross-attention output projection + residual (GEMV);
//   up         LayerNorm 3 -> MLP up-projection + GELU (GEMV);
//   down       MLP down-projection + residual (GEMV, K split over a cluster
//              of 4 CTAs).
// Every CTA computes whole 8-feature output tiles over its K range (mma.sync
// m16n8k16, the rows padded to 16 as M, 8 weight rows as N; the K range
// split over 8 warps and summed in warp order), so no split-K exchange is
// needed except in the down-projection cluster.  Weights (and the attention
// K/V, constant during a step) are requested before the wait on the previous
// launch, and each launch prefetches into L2 the weights of a later launch
// (the host picks which: three ahead by default).
// The LayerNorm is computed by its consumers from the fp32 residual stream,
// in registers: gain and bias before the wait, the rows straight from L2
// after it.
#include <algorithm>
#include <mutex>

#include "kernels.h"
#include "rowmma.cuh"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_fewrow)

namespace {

constexpr int FR_T = 256;               // threads (8 warps)
constexpr int FR_R = VF_ROWS;           // rows of a step, at most
constexpr int FR_MAXT = 5;              // output tiles of 8 features per CTA, at most
constexpr int FR_KS = 4;                // K split of a GEMV over a cluster, at most
constexpr int FR_CH = 128;              // keys per attention chunk
constexpr int FR_TILE = FR_CH * 128;    // bytes of one chunk of K or V
constexpr int FR_RED = 8 * FR_MAXT * 128 * 4;
constexpr int FR_SCR = (8 * 9 * 64 + 2 * 8 * 16) * 4;   // attention combine scratch
constexpr int FR_PART = FR_R * 66 * 4;                   // one partial (max, sum, out[64]) per row

__host__ __device__ constexpr int fr_pitch(int D) { return 2 * D + 16; }
__host__ __device__ constexpr int align_up(int v, int a) { return (v + a - 1) / a * a; }

__device__ __forceinline__ void fr_stamp(unsigned long long* tr, int phase) {
  if (tr != nullptr && threadIdx.x == 0) tr[(size_t)blockIdx.x * FR_TRACE_PHASES + phase] = global_ns();
}

// LayerNorm of the step's rows in registers.  Lane l of every warp holds the
// gain and bias of columns 4 (l + 32 i) .. + 3 (i < KSW), loaded before the
// kernel waits on its predecessor (they are constants); after the wait, warp
// w reads rows w and w + 8 of the residual stream straight from L2 into
// registers (all FR_R row slots exist; the ones past the live rows are read
// and not used), and writes bf16(LayerNorm(x_r) * g + b), fp32 statistics,
// into the MMA operand rows.
template <int KSW>
struct LnRegs {
  float4 g[KSW], b[KSW];
};
template <int KSW>
__device__ __forceinline__ void fr_ln_params(LnRegs<KSW>& p, const float* g, const float* b) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < KSW; ++i) {
    p.g[i] = __ldg(reinterpret_cast<const float4*>(g) + lane + 32 * i);
    p.b[i] = __ldg(reinterpret_cast<const float4*>(b) + lane + 32 * i);
  }
}
template <int KSW>
__device__ __forceinline__ void fr_ln_fetch(float4 (&v)[2][KSW], const float* x) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int r = warp + 8 * j;
    const float4* xr = reinterpret_cast<const float4*>(x + (size_t)r * KSW * 128);
#pragma unroll
    for (int i = 0; i < KSW; ++i) v[j][i] = r < FR_R ? __ldcg(xr + lane + 32 * i) : make_float4(0.f, 0.f, 0.f, 0.f);
  }
}
template <int KSW>
__device__ __forceinline__ void fr_ln_apply(const float4 (&v)[2][KSW], const LnRegs<KSW>& p, uint8_t* act, int R) {
  constexpr int D = KSW * 128;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float mean[2], rstd[2];
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < KSW; ++i) s += (v[j][i].x + v[j][i].y) + (v[j][i].z + v[j][i].w);
    mean[j] = s;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {   // the two rows' warp sums side by side
    mean[0] += __shfl_xor_sync(0xffffffffu, mean[0], o);
    mean[1] += __shfl_xor_sync(0xffffffffu, mean[1], o);
  }
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    mean[j] = mean[j] / (float)D;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < KSW; ++i) {
      const float a = v[j][i].x - mean[j], b = v[j][i].y - mean[j], c = v[j][i].z - mean[j],
                  e = v[j][i].w - mean[j];
      q += (a * a + b * b) + (c * c + e * e);
    }
    rstd[j] = q;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    rstd[0] += __shfl_xor_sync(0xffffffffu, rstd[0], o);
    rstd[1] += __shfl_xor_sync(0xffffffffu, rstd[1], o);
  }
#pragma unroll
  for (int j = 0; j < 2; ++j) {
    const int r = warp + 8 * j;
    if (r >= R) continue;
    const float rs = rsqrtf(rstd[j] / (float)D + 1e-5f), mu = mean[j];
    uint2* row = reinterpret_cast<uint2*>(act + (size_t)r * fr_pitch(D));
#pragma unroll
    for (int i = 0; i < KSW; ++i) {
      const float4 w = v[j][i], gg = p.g[i], bb = p.b[i];
      uint2 o;
      o.x = bf2_bits((w.x - mu) * rs * gg.x + bb.x, (w.y - mu) * rs * gg.y + bb.y);
      o.y = bf2_bits((w.z - mu) * rs * gg.z + bb.z, (w.w - mu) * rs * gg.w + bb.w);
      row[lane + 32 * i] = o;
    }
  }
}

// Thread 0: this CTA's share of a later launch's weights into L2 (that
// launch's CTAs become resident only as this one's leave).
__device__ __forceinline__ void fr_prefetch(const void* pf, uint32_t pf_bytes) {
  if (pf == nullptr || pf_bytes == 0) return;
  const uint32_t per = ((pf_bytes / gridDim.x) + 15u) & ~15u;
  const uint32_t s0 = blockIdx.x * per;
  if (s0 < pf_bytes) l2_prefetch(static_cast<const char*>(pf) + s0, per < pf_bytes - s0 ? per : pf_bytes - s0);
}

// Weight tiles of the few-row kernels are packed (at create) so that one
// 8-row tile is contiguous and its 16-byte pieces run piece-major: piece c of
// row r (columns 8 c .. 8 c + 7) at byte 16 (8 c + r).  A tile then lands
// with one bulk copy, and the 8 row addresses of an ldmatrix are 128
// consecutive bytes (no bank conflict).
// acc[i] += rows (act panel at a_base) x weight tile i (at w_base + i
// w_tile) over the K columns [8 chunk0, 8 chunk0 + D) of the tiles; warp w
// takes columns [w D / 8, (w + 1) D / 8) of the panel.
template <int KSW>
__device__ __forceinline__ void fr_mma_panel(float (&acc)[FR_MAXT][4], uint32_t a_base, uint32_t w_base,
                                             uint32_t w_tile, int chunk0, int ntile, int R) {
  constexpr int D = KSW * 128, KW = D / 8;
  constexpr uint32_t P = fr_pitch(D);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int ar = min((lane & 7) + 8 * ((lane >> 3) & 1), R - 1);
  const uint32_t a_lane = a_base + (uint32_t)ar * P + 16u * (lane >> 4) + 2u * (uint32_t)(warp * KW);
  const uint32_t b_lane =
      w_base + 16u * (uint32_t)((chunk0 + warp * (KW / 8) + (lane >> 3)) * 8 + (lane & 7));
  uint32_t af[KSW][4];
#pragma unroll
  for (int j = 0; j < KSW; ++j) ldsm_x4(a_lane + 32u * j, af[j]);
#pragma unroll
  for (int i = 0; i < FR_MAXT; ++i) {
    if (i < ntile) {
#pragma unroll
      for (int jj = 0; jj < KSW / 2; ++jj) {
        uint32_t b[4];
        ldsm_x4(b_lane + (uint32_t)i * w_tile + 512u * jj, b);
        mma16816(acc[i], af[2 * jj], b[0], b[1]);
        mma16816(acc[i], af[2 * jj + 1], b[2], b[3]);
      }
    }
  }
}

// The 8 warps' partial tiles into red, then thread o < ntile * 4 * FR_R takes
// output pair (tile i, row r, features 2 n2, 2 n2 + 1), summed in warp order.
struct Pair {
  int i, r, n2;
  float v0, v1;
  bool has;
};
__device__ __forceinline__ Pair fr_reduce(const float (&acc)[FR_MAXT][4], float* red, int ntile, bool live) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  if (live) {
#pragma unroll
    for (int i = 0; i < FR_MAXT; ++i) {
      if (i < ntile) {
        float* o = red + (warp * FR_MAXT + i) * 128;
        *reinterpret_cast<float2*>(o + g * 8 + 2 * t) = make_float2(acc[i][0], acc[i][1]);
        *reinterpret_cast<float2*>(o + (g + 8) * 8 + 2 * t) = make_float2(acc[i][2], acc[i][3]);
      }
    }
  }
  __syncthreads();
  Pair p{0, 0, 0, 0.f, 0.f, false};
  const int o = threadIdx.x;
  if (live && o < ntile * 4 * FR_R) {
    p.has = true;
    p.i = o / (4 * FR_R);
    const int rem = o - p.i * 4 * FR_R;
    p.r = rem >> 2;
    p.n2 = rem & 3;
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      const float2 v = *reinterpret_cast<const float2*>(red + (w * FR_MAXT + p.i) * 128 + p.r * 8 + 2 * p.n2);
      p.v0 += v.x;
      p.v1 += v.y;
    }
  }
  return p;
}

// ---------------------------------------------------------------------------
// GEMV: y[r][m] = sum_k in[r][k] W[m][k].  The grid is G groups of KS CTAs
// (one thread-block cluster per group when KS > 1); group g takes the tiles
// [nt g / G, nt (g + 1) / G) and its CTA of rank q the K range
// [q K / KS, (q + 1) K / KS); rank 0 adds the other ranks' partials after its
// own, in rank order.
// ---------------------------------------------------------------------------
__host__ __device__ inline int gemv_smem_bytes(int D, int tiles_max, int np, int KS) {
  return align_up(tiles_max * 16 * np * D, 128) + np * FR_R * fr_pitch(D) + FR_RED +
         (KS - 1) * FR_MAXT * 4 * FR_R * 8;
}

template <int KSW, int MODE, int KS>
__global__ void __launch_bounds__(FR_T, 1) fr_gemv_kernel(const __grid_constant__ FrGemv A) {
  constexpr int D = KSW * 128;
  constexpr uint32_t P = fr_pitch(D);
  extern __shared__ __align__(128) uint8_t fr_smem[];
  __shared__ __align__(8) uint64_t wbar, abar, rbar;
  const int tid = threadIdx.x;
  const int ks = KS > 1 ? (int)cluster_ctarank() : 0;
  const int Kc = A.K / KS, np = Kc / D;
  const uint32_t wtile = 16u * (uint32_t)Kc;   // one packed 8-row tile of this CTA's K range
  const int nt = (A.N + 7) / 8, G = (int)gridDim.x / KS, grp = (int)blockIdx.x / KS;
  const int t0 = (int)((long long)nt * grp / G), ntile = (int)((long long)nt * (grp + 1) / G) - t0;
  uint8_t* wts = fr_smem;
  uint8_t* act = wts + align_up(A.tiles_max * (int)wtile, 128);
  float* red = reinterpret_cast<float*>(act + np * FR_R * P);
  float2* recv = reinterpret_cast<float2*>(reinterpret_cast<uint8_t*>(red) + FR_RED);
  tl_mark(A.tl, TL_ENTRY);
  fr_stamp(A.trace, 0);
  if (tid == 0) {
    mbar_init(&wbar, 1);
    mbar_init(&abar, 1);
    mbar_init(&rbar, 1);
    fence_mbar_init();
    if (KS > 1 && ks == 0) mbar_arrive_expect_tx(&rbar, (uint32_t)((KS - 1) * ntile * 4 * FR_R * 8));
    mbar_arrive_expect_tx(&wbar, (uint32_t)ntile * wtile);
    for (int i = 0; i < ntile; ++i)
      bulk_load(wts + i * wtile, A.W + ((size_t)(t0 + i) * A.K + (size_t)ks * Kc) * 8, wtile, &wbar);
    fr_prefetch(A.pf, A.pf_bytes);
  }
  LnRegs<KSW> lnr;
  if constexpr (MODE == FR_GELU) fr_ln_params(lnr, A.ln_g, A.ln_b);
  __syncthreads();
  if (KS > 1) cluster_arrive_relaxed();
  pdl_wait();
  tl_mark(A.tl, TL_WORK);
  fr_stamp(A.trace, 1);
  pdl_launch();
  // The input rows (written by the previous launch): all FR_R row slots,
  // requested at once without waiting to read how many are live (rows past
  // them are not used)
  float4 xv[2][KSW];
  if constexpr (MODE == FR_GELU) {
    fr_ln_fetch<KSW>(xv, A.x);
  } else if (tid < 32) {   // panel p, row r: one bulk copy each, issued by the warp's lanes side by side
    if (tid == 0) mbar_arrive_expect_tx(&abar, (uint32_t)(FR_R * np) * 2u * D);
    __syncwarp();
    for (int q = tid; q < FR_R * np; q += 32) {
      const int p = q / FR_R, r = q - p * FR_R;
      bulk_load(act + (p * FR_R + r) * P, A.a + (size_t)r * A.K + (size_t)ks * Kc + (size_t)p * D, 2u * D, &abar);
    }
  }
  const int R = *A.n_rows;   // uniform over the grid
  const bool live = R > 0;
  if constexpr (MODE == FR_GELU) {
    if (live) fr_ln_apply<KSW>(xv, lnr, act, R);
  } else {
    mbar_wait(&abar, 0, A.status);
    fr_stamp(A.trace, 11);
  }
  fr_stamp(A.trace, 2);
  mbar_wait(&wbar, 0, A.status);
  fr_stamp(A.trace, 3);
  __syncthreads();
  float acc[FR_MAXT][4];
#pragma unroll
  for (int i = 0; i < FR_MAXT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
  if (live)
    for (int p = 0; p < np; ++p)
      fr_mma_panel<KSW>(acc, smem_u32(act) + (uint32_t)(p * FR_R) * P, smem_u32(wts), wtile, p * (D / 8), ntile, R);
  Pair pr = fr_reduce(acc, red, ntile, live);
  tl_mark(A.tl, TL_MID);
  fr_stamp(A.trace, 4);
  if constexpr (KS > 1) {
    cluster_wait();   // rank 0's receive barrier exists
    if (live) {
      if (ks > 0) {
        if (pr.has)
          st_async_f2(dsmem_addr(&recv[(ks - 1) * FR_MAXT * 4 * FR_R + tid], 0), pr.v0, pr.v1,
                      dsmem_addr(&rbar, 0));
      } else {
        mbar_wait(&rbar, 0, A.status);
        if (pr.has)
#pragma unroll
          for (int q = 0; q < KS - 1; ++q) {
            const float2 o = recv[q * FR_MAXT * 4 * FR_R + tid];
            pr.v0 += o.x;
            pr.v1 += o.y;
          }
      }
    }
  }
  fr_stamp(A.trace, 5);
  if (ks == 0 && pr.has && pr.r < R) {
    const int m = 8 * (t0 + pr.i) + 2 * pr.n2;
    if (m < A.N) {
      if constexpr (MODE == FR_RESID) {
        float2* xp = reinterpret_cast<float2*>(A.x_out + (size_t)pr.r * A.N + m);
        const float2 old = *xp;
        *xp = make_float2(old.x + (pr.v0 + __ldg(A.bias + m)), old.y + (pr.v1 + __ldg(A.bias + m + 1)));
      } else {
        *reinterpret_cast<__nv_bfloat162*>(A.h_out + (size_t)pr.r * A.N + m) = __floats2bfloat162_rn(
            gelu_erf(pr.v0 + __ldg(A.bias + m)), gelu_erf(pr.v1 + __ldg(A.bias + m + 1)));
      }
    }
  }
  if constexpr (KS > 1) cluster_sync();   // no CTA leaves with its stores to a peer in flight
  fr_stamp(A.trace, 7);
  tl_mark(A.tl, TL_EXIT);
}

// ---------------------------------------------------------------------------
// Per-head cluster kernels: shared memory layout
// ---------------------------------------------------------------------------
struct HeadLayout {
  int wts, act, kv, red, gat, mrg, part, total;
};
// The merge buffer and this CTA's partial alias the reduction buffer: a peer
// sends a partial only after this CTA's gather contribution, which follows
// its reduction.
__host__ __device__ inline HeadLayout head_layout(int D, int tiles_max, int n_slots, int mrg_slots) {
  HeadLayout L;
  int o = 0;
  L.kv = o;                                       // chunk slots: [n_slots][K, V], 1024-aligned
  o += n_slots * 2 * FR_TILE;
  L.wts = o;                                      // packed weight tiles
  o += align_up(tiles_max * 16 * D, 128);
  L.act = o;                                      // LayerNorm rows; later the combine scratch
  o += align_up(FR_R * fr_pitch(D) > FR_SCR ? FR_R * fr_pitch(D) : FR_SCR, 128);
  L.red = o;
  L.mrg = o;                                      // partials received for the merge
  L.part = o + mrg_slots * FR_PART;               // this CTA's partial
  o += align_up(FR_RED > (mrg_slots + 1) * FR_PART ? FR_RED : (mrg_slots + 1) * FR_PART, 128);
  L.gat = o;                                      // gathered q (, k, v) pairs [3][FR_R][32]
  o += 3 * FR_R * 32 * 4;
  L.total = o;
  return L;
}

__device__ __forceinline__ int self_chunks(const RowPlan& plan, const int* kv_len, int b) {
  const int nr = plan.n_utt_rows[b];
  return nr > 0 ? (kv_len[b] + nr + FR_CH - 1) / FR_CH : 0;
}

// A partial (rows [row0, row0 + nr) of `part`, 66 floats each) into the merge
// buffer of CTA `dst` at slot `slot`: asynchronous stores counted on that
// CTA's barrier, or plain stores when dst is this CTA (not counted).
__device__ __forceinline__ void put_partial(const float* part, int nr, int row0, uint8_t* mrg_local, int slot,
                                            uint64_t* bar_local, uint32_t dst, uint32_t self) {
  if (dst == self) {
    float* m = reinterpret_cast<float*>(mrg_local + slot * FR_PART) + row0 * 66;
    for (int e = threadIdx.x; e < nr * 66; e += FR_T) m[e] = part[e];
    return;
  }
  const uint32_t base = dsmem_addr(mrg_local, dst) + (uint32_t)(slot * FR_PART);
  const uint32_t bar = dsmem_addr(bar_local, dst);
  for (int e = threadIdx.x; e < nr * 66; e += FR_T)
    st_async_b32(base + 4u * (uint32_t)((row0 + e / 66) * 66 + e % 66), __float_as_uint(part[e]), bar);
}

// The 16-byte pieces [n][FR_R] of this CTA's gathered values (piece (i, r) at
// word offset off(i) + 32 r of `gat`, already written here) into every other
// CTA of the cluster, counted on their barriers.
template <typename Off>
__device__ __forceinline__ void share_pieces(uint32_t* gat, int n, int C, uint32_t self, uint64_t* bar, Off off) {
  for (int e = threadIdx.x; e < n * FR_R * (C - 1); e += FR_T) {
    const int q = e / (n * FR_R), pc = e - q * n * FR_R, i = pc / FR_R, r = pc - i * FR_R;
    const uint32_t dst = (uint32_t)q + (q >= (int)self ? 1u : 0u);
    const uint32_t w = off(i) + 32u * r;
    const float4 v = *reinterpret_cast<const float4*>(gat + w);
    st_async_f4(dsmem_addr(gat + w, dst), v, dsmem_addr(bar, dst));
  }
}

// ---------------------------------------------------------------------------
// LayerNorm 1 -> QKV of head h -> self-attention of head h, one cluster per head
// ---------------------------------------------------------------------------
template <int KSW>
__global__ void __launch_bounds__(FR_T, 1) fr_self_kernel(const __grid_constant__ CUtensorMap kmap,
                                                       const __grid_constant__ CUtensorMap vmap,
                                                       const __grid_constant__ FrHead A) {
  constexpr int D = KSW * 128;
  extern __shared__ __align__(1024) uint8_t hs_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(hs_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t wbar, gbar, mbar, kvbar;
  __shared__ int s_pos[FR_R];
  const HeadLayout Lo = head_layout(D, A.tiles_max, 1, A.mrg_slots);
  const int tid = threadIdx.x;
  const int C = A.C, c = (int)cluster_ctarank(), hh = (int)blockIdx.x / C;
  const int H = A.H, d = D;
  uint8_t* kvs = sm + Lo.kv;
  uint8_t* wts = sm + Lo.wts;
  uint8_t* act = sm + Lo.act;
  float* red = reinterpret_cast<float*>(sm + Lo.red);
  uint32_t* gat = reinterpret_cast<uint32_t*>(sm + Lo.gat);   // [3][FR_R][32]: q / 8, k, v pairs
  uint8_t* mrg = sm + Lo.mrg;                                 // [chunk][FR_R][66]
  float* part = reinterpret_cast<float*>(sm + Lo.part);
  // this CTA's QKV tiles: local tiles [24 c / C, 24 (c + 1) / C) of the head's
  // 24 (q 0-7, k 8-15, v 16-23)
  const int lt0 = 24 * c / C, lt1 = 24 * (c + 1) / C, ntile = lt1 - lt0;
  auto gtile = [&](int lt) { return (lt >> 3) * (d / 8) + 8 * hh + (lt & 7); };
  const uint32_t wtile = 16u * (uint32_t)D;
  tl_mark(A.tl, TL_ENTRY);
  fr_stamp(A.trace, 0);
  // items: (utterance b, key chunk j) in order; this CTA takes items c, c + C, ...
  // the merge of utterance b happens in the CTA holding item (b, 0)
  if (tid == 0) {
    mbar_init(&wbar, 1);
    mbar_init(&gbar, 1);
    mbar_init(&mbar, 1);
    mbar_init(&kvbar, 1);
    fence_mbar_init();
    // the other CTAs' q, k, v pieces (16 bytes per tile and row)
    mbar_arrive_expect_tx(&gbar, (uint32_t)((24 - ntile) * FR_R * 16));
    uint32_t mrg_bytes = 0;   // partials the other CTAs send for the utterances led here
    int e = 0;
    bool first = true;
    for (int b = 0; b < A.B; ++b) {
      const int nck = self_chunks(A.plan, A.kv_len, b), nr = A.plan.n_utt_rows[b];
      if (nck > 0 && e % C == c)
        for (int j = 0; j < nck; ++j)
          if ((e + j) % C != c) mrg_bytes += (uint32_t)(nr * 66 * 4);
      for (int j = 0; j < nck; ++j, ++e)
        if (e % C == c && first) {   // the first item's K/V: constant during the step
          first = false;
          const long long row = A.row0 + ((long long)b * H + hh) * A.t_alloc + (long long)j * FR_CH;
          mbar_arrive_expect_tx(&kvbar, 2 * FR_TILE);
          tma_load_2d(kvs, &kmap, &kvbar, 0, (int)row);
          tma_load_2d(kvs + FR_TILE, &vmap, &kvbar, 0, (int)row);
        }
    }
    mbar_arrive_expect_tx(&mbar, mrg_bytes);
    mbar_arrive_expect_tx(&wbar, (uint32_t)ntile * wtile);
    for (int i = 0; i < ntile; ++i) bulk_load(wts + i * wtile, A.W + (size_t)gtile(lt0 + i) * 8 * d, wtile, &wbar);
    fr_prefetch(A.pf, A.pf_bytes);
  }
  if (tid < FR_R) s_pos[tid] = A.plan.row_pos[tid];
  LnRegs<KSW> lnr;
  fr_ln_params(lnr, A.ln_g, A.ln_b);
  __syncthreads();
  cluster_arrive_relaxed();
  pdl_wait();
  tl_mark(A.tl, TL_WORK);
  fr_stamp(A.trace, 1);
  pdl_launch();
  // the residual rows: all FR_R slots at once (rows past the live ones are not used)
  float4 xv[2][KSW];
  fr_ln_fetch<KSW>(xv, A.x);
  const int R = *A.plan.n_rows;
  const bool live = R > 0;
  if (live) fr_ln_apply<KSW>(xv, lnr, act, R);
  fr_stamp(A.trace, 2);
  mbar_wait(&wbar, 0, A.status);
  fr_stamp(A.trace, 3);
  __syncthreads();
  float acc[FR_MAXT][4];
#pragma unroll
  for (int i = 0; i < FR_MAXT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
  if (live) fr_mma_panel<KSW>(acc, smem_u32(act), smem_u32(wts), wtile, 0, ntile, R);
  const Pair pr = fr_reduce(acc, red, ntile, live);
  tl_mark(A.tl, TL_MID);
  fr_stamp(A.trace, 4);
  cluster_wait();   // every CTA's barriers exist
  if (pr.has) {
    // q / 8, k, v of (row r, features m, m + 1); k and v also to the cache
    const int lt = lt0 + pr.i, which = lt >> 3, m = 8 * gtile(lt) + 2 * pr.n2;
    const float y0 = pr.v0 + __ldg(A.bias + m), y1 = pr.v1 + __ldg(A.bias + m + 1);
    const uint32_t v = which == 0 ? bf2_bits(y0 * 0.125f, y1 * 0.125f) : bf2_bits(y0, y1);
    if (which > 0 && pr.r < R &&
        !bounds_bad(A.status, A.plan.row_b[pr.r] < 0 || A.plan.row_b[pr.r] >= A.B || s_pos[pr.r] < 0 ||
                                  s_pos[pr.r] >= A.max_pos)) {
      const int f = m - which * d;
      const size_t slot = (((size_t)A.plan.row_b[pr.r] * H + hh) * A.max_pos + s_pos[pr.r]) * 64 + (f & 63);
      *reinterpret_cast<uint32_t*>((which == 1 ? A.ks : A.vs) + slot) = v;
    }
    const int j = ((lt & 7) * 8 + 2 * pr.n2) >> 1;   // pair index within the head
    gat[(which * FR_R + pr.r) * 32 + j] = v;
  }
  __syncthreads();
  if (live)   // this CTA's tiles to the other CTAs of the cluster
    share_pieces(gat, ntile, C, (uint32_t)c, &gbar,
                 [&](int i) { return (uint32_t)(((lt0 + i) >> 3) * FR_R * 32 + ((lt0 + i) & 7) * 4); });
  if (live) mbar_wait(&gbar, 0, A.status);   // a refused step sends nothing
  fr_stamp(A.trace, 5);
  __syncthreads();
  // attention items
  if (live) {
    int e = 0, n_done = 0;
    for (int b = 0; b < A.B; ++b) {
      const int nck = self_chunks(A.plan, A.kv_len, b);
      if (nck == 0) continue;
      const int leader = e % C;
      const int nr = A.plan.n_utt_rows[b], row0 = A.plan.row_start[b], P = A.kv_len[b], n_keys = P + nr;
      for (int j = 0; j < nck; ++j, ++e) {
        if (e % C != c) continue;
        if (n_done > 0) {   // later items reuse the slot (rare: more items than CTAs)
          asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
          __syncthreads();
          if (tid == 0) {
            const long long row = A.row0 + ((long long)b * H + hh) * A.t_alloc + (long long)j * FR_CH;
            mbar_arrive_expect_tx(&kvbar, 2 * FR_TILE);
            tma_load_2d(kvs, &kmap, &kvbar, 0, (int)row);
            tma_load_2d(kvs + FR_TILE, &vmap, &kvbar, 0, (int)row);
          }
        }
        mbar_wait(&kvbar, (uint32_t)(n_done & 1), A.status);
        if (n_done == 0) fr_stamp(A.trace, 8);
        ++n_done;
        // this step's keys and values inside the chunk
        const uint32_t kb = smem_u32(kvs), vb = kb + FR_TILE;
        const int lo = max(P, j * FR_CH), hi = min(n_keys, (j + 1) * FR_CH);
        const int pieces = max(0, hi - lo) * 8;
        for (int q = tid; q < 2 * pieces; q += FR_T) {
          const int wv = q >= pieces, qq = q - wv * pieces;
          const int key = lo + (qq >> 3), c16 = qq & 7, r = row0 + key - P;
          const uint32_t* src = gat + ((1 + wv) * FR_R + r) * 32 + 4 * c16;
          const uint32_t dst = (wv ? vb : kb) + sw128(key - j * FR_CH, c16);
          sts32(dst, src[0]);
          sts32(dst + 4, src[1]);
          sts32(dst + 8, src[2]);
          sts32(dst + 12, src[3]);
        }
        __syncthreads();
        AttnState st;
        attn_init(st, gat + row0 * 32, nr, s_pos + row0, n_keys, true);
        attn_chunk(st, kb, vb, j * FR_CH);
        attn_combine(st, nr, reinterpret_cast<float*>(act), part);
        if (n_done == 1) fr_stamp(A.trace, 9);
        put_partial(part, nr, row0, mrg, j, &mbar, (uint32_t)leader, (uint32_t)c);
      }
    }
    // merge, in key-chunk order, the utterances this CTA leads
    fr_stamp(A.trace, 6);
    mbar_wait(&mbar, 0, A.status);
    fr_stamp(A.trace, 10);
    __syncthreads();
    e = 0;
    for (int b = 0; b < A.B; ++b) {
      const int nck = self_chunks(A.plan, A.kv_len, b);
      if (nck == 0) continue;
      const int leader = e % C;
      e += nck;
      if (leader != c) continue;
      const int nr = A.plan.n_utt_rows[b], row0 = A.plan.row_start[b];
      const float* pm = reinterpret_cast<const float*>(mrg);
      for (int q = tid; q < nr * 32; q += FR_T) {
        const int r = row0 + (q >> 5), jj = q & 31;
        float M = -INFINITY;
        for (int j = 0; j < nck; ++j) M = fmaxf(M, pm[(j * FR_R + r) * 66]);
        const float Mu = (M == -INFINITY) ? 0.f : M;
        float L = 0.f, o0 = 0.f, o1 = 0.f;
        for (int j = 0; j < nck; ++j) {
          const float* row = pm + (j * FR_R + r) * 66;
          const float f = __expf(row[0] - Mu);
          L += row[1] * f;
          o0 += row[2 + 2 * jj] * f;
          o1 += row[3 + 2 * jj] * f;
        }
        *reinterpret_cast<__nv_bfloat162*>(A.att + (size_t)r * d + hh * 64 + 2 * jj) =
            __floats2bfloat162_rn(o0 / L, o1 / L);
      }
    }
  }
  cluster_sync();   // no CTA leaves with its stores to a peer in flight
  fr_stamp(A.trace, 7);
  tl_mark(A.tl, TL_EXIT);
}

// ---------------------------------------------------------------------------
// LayerNorm 2 -> cross query of head h -> cross-attention of head h over the
// encoder frames, one cluster per head; CTA c takes key chunks c, c + C, ...
// ---------------------------------------------------------------------------
template <int KSW>
__global__ void __launch_bounds__(FR_T, 1) fr_cross_kernel(const __grid_constant__ CUtensorMap xmap,
                                                        const __grid_constant__ FrHead A) {
  constexpr int D = KSW * 128;
  extern __shared__ __align__(1024) uint8_t hs_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(hs_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t wbar, gbar, mbar, kvbar[2];
  const HeadLayout Lo = head_layout(D, A.tiles_max, 2, A.mrg_slots);
  const int tid = threadIdx.x;
  const int C = A.C, c = (int)cluster_ctarank(), hh = (int)blockIdx.x / C;
  const int H = A.H, d = D;
  uint8_t* kvs = sm + Lo.kv;
  uint8_t* wts = sm + Lo.wts;
  uint8_t* act = sm + Lo.act;
  float* red = reinterpret_cast<float*>(sm + Lo.red);
  uint32_t* gat = reinterpret_cast<uint32_t*>(sm + Lo.gat);   // [FR_R][32] q / 8 pairs
  uint8_t* mrg = sm + Lo.mrg;                                 // [split][FR_R][66]
  float* part = reinterpret_cast<float*>(sm + Lo.part);
  const int lt0 = 8 * c / C, lt1 = 8 * (c + 1) / C, ntile = lt1 - lt0;
  const uint32_t wtile = 16u * (uint32_t)D;
  const long long vofs = A.vofs;
  auto chunk_row = [&](int b, int j) { return A.row0 + ((long long)b * H + hh) * A.t_alloc + (long long)j * FR_CH; };
  auto n_mine = [&](int b) {   // chunks c, c + C, ... of utterance b
    const int nc = (A.enc_len[b] + FR_CH - 1) / FR_CH;
    return (A.plan.n_utt_rows[b] > 0 && c < nc) ? (nc - c + C - 1) / C : 0;
  };
  tl_mark(A.tl, TL_ENTRY);
  fr_stamp(A.trace, 0);
  if (tid == 0) {
    mbar_init(&wbar, 1);
    mbar_init(&gbar, 1);
    mbar_init(&mbar, 1);
    mbar_init(&kvbar[0], 1);
    mbar_init(&kvbar[1], 1);
    fence_mbar_init();
    // the other CTAs' q pieces (16 bytes per tile and row)
    mbar_arrive_expect_tx(&gbar, (uint32_t)((8 - ntile) * FR_R * 16));
    uint32_t mrg_bytes = 0;   // partials of splits 1 .. sent to split 0
    if (c == 0)
      for (int b = 0; b < A.B; ++b) {
        const int nr = A.plan.n_utt_rows[b], nc = (A.enc_len[b] + FR_CH - 1) / FR_CH;
        if (nr > 0) mrg_bytes += (uint32_t)((min(C, nc) - 1) * nr * 66 * 4);
      }
    mbar_arrive_expect_tx(&mbar, mrg_bytes);
    // the first two chunks of this CTA (the encoder K/V is constant)
    int issued = 0;
    for (int b = 0; b < A.B && issued < 2; ++b)
      for (int i = 0; i < n_mine(b) && issued < 2; ++i, ++issued) {
        const long long row = chunk_row(b, c + i * C);
        uint8_t* dst = kvs + issued * 2 * FR_TILE;
        mbar_arrive_expect_tx(&kvbar[issued], 2 * FR_TILE);
        tma_load_2d(dst, &xmap, &kvbar[issued], 0, (int)row);
        tma_load_2d(dst + FR_TILE, &xmap, &kvbar[issued], 0, (int)(row + vofs));
      }
    mbar_arrive_expect_tx(&wbar, (uint32_t)ntile * wtile);
    for (int i = 0; i < ntile; ++i)
      bulk_load(wts + i * wtile, A.W + (size_t)(8 * hh + lt0 + i) * 8 * d, wtile, &wbar);
    fr_prefetch(A.pf, A.pf_bytes);
  }
  LnRegs<KSW> lnr;
  fr_ln_params(lnr, A.ln_g, A.ln_b);
  __syncthreads();
  cluster_arrive_relaxed();
  pdl_wait();
  tl_mark(A.tl, TL_WORK);
  fr_stamp(A.trace, 1);
  pdl_launch();
  // the residual rows: all FR_R slots at once (rows past the live ones are not used)
  float4 xv[2][KSW];
  fr_ln_fetch<KSW>(xv, A.x);
  const int R = *A.plan.n_rows;
  const bool live = R > 0;
  if (live) fr_ln_apply<KSW>(xv, lnr, act, R);
  fr_stamp(A.trace, 2);
  mbar_wait(&wbar, 0, A.status);
  fr_stamp(A.trace, 3);
  __syncthreads();
  float acc[FR_MAXT][4];
#pragma unroll
  for (int i = 0; i < FR_MAXT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
  if (live) fr_mma_panel<KSW>(acc, smem_u32(act), smem_u32(wts), wtile, 0, ntile, R);
  const Pair pr = fr_reduce(acc, red, ntile, live);
  tl_mark(A.tl, TL_MID);
  fr_stamp(A.trace, 4);
  cluster_wait();
  if (pr.has) {
    const int lt = lt0 + pr.i, m = 64 * hh + 8 * lt + 2 * pr.n2;
    const float y0 = pr.v0 + __ldg(A.bias + m), y1 = pr.v1 + __ldg(A.bias + m + 1);
    if (A.q_anchor != nullptr && pr.r < R)
      *reinterpret_cast<float2*>(A.q_anchor + (size_t)pr.r * d + m) = make_float2(y0, y1);
    gat[pr.r * 32 + ((8 * lt + 2 * pr.n2) >> 1)] = bf2_bits(y0 * 0.125f, y1 * 0.125f);
  }
  __syncthreads();
  if (live)   // this CTA's q tiles to the other CTAs of the cluster
    share_pieces(gat, ntile, C, (uint32_t)c, &gbar, [&](int i) { return (uint32_t)((lt0 + i) * 4); });
  if (live) mbar_wait(&gbar, 0, A.status);   // a refused step sends nothing
  fr_stamp(A.trace, 5);
  __syncthreads();
  if (live) {
    int n = 0;   // chunks consumed by this CTA (slot n % 2, its use n / 2)
    for (int b = 0; b < A.B; ++b) {
      const int mine = n_mine(b);
      if (mine == 0) continue;
      const int nr = A.plan.n_utt_rows[b], row0 = A.plan.row_start[b], T = A.enc_len[b];
      AttnState st;
      attn_init(st, gat + row0 * 32, nr, nullptr, T, false);
      for (int i = 0; i < mine; ++i, ++n) {
        const int s = n & 1;
        mbar_wait(&kvbar[s], (uint32_t)((n >> 1) & 1), A.status);
        if (n == 0) fr_stamp(A.trace, 8);
        const uint32_t kb = smem_u32(kvs + s * 2 * FR_TILE);
        attn_chunk(st, kb, kb + FR_TILE, (c + i * C) * FR_CH);
        // refill this slot with this CTA's chunk n + 2, if any (long encoder memories)
        __syncthreads();
        if (tid == 0) {
          int nb = b, ni = i + 2;
          while (nb < A.B && ni >= n_mine(nb)) {
            ni -= n_mine(nb);
            ++nb;
          }
          if (nb < A.B) {
            const long long row = chunk_row(nb, c + ni * C);
            mbar_arrive_expect_tx(&kvbar[s], 2 * FR_TILE);
            tma_load_2d(kvs + s * 2 * FR_TILE, &xmap, &kvbar[s], 0, (int)row);
            tma_load_2d(kvs + s * 2 * FR_TILE + FR_TILE, &xmap, &kvbar[s], 0, (int)(row + vofs));
          }
        }
      }
      attn_combine(st, nr, reinterpret_cast<float*>(act), part);
      fr_stamp(A.trace, 9);
      put_partial(part, nr, row0, mrg, c, &mbar, 0u, (uint32_t)c);
    }
    fr_stamp(A.trace, 6);
    if (c == 0) {
      mbar_wait(&mbar, 0, A.status);
      fr_stamp(A.trace, 10);
      __syncthreads();
      const float* pm = reinterpret_cast<const float*>(mrg);
      for (int b = 0; b < A.B; ++b) {
        const int nr = A.plan.n_utt_rows[b], nc = (A.enc_len[b] + FR_CH - 1) / FR_CH;
        if (nr == 0) continue;
        const int ns = min(C, nc), row0 = A.plan.row_start[b];
        for (int q = tid; q < nr * 32; q += FR_T) {
          const int r = row0 + (q >> 5), jj = q & 31;
          float M = -INFINITY;
          for (int s = 0; s < ns; ++s) M = fmaxf(M, pm[(s * FR_R + r) * 66]);
          const float Mu = (M == -INFINITY) ? 0.f : M;
          float L = 0.f, o0 = 0.f, o1 = 0.f;
          for (int s = 0; s < ns; ++s) {
            const float* row = pm + (s * FR_R + r) * 66;
            const float f = __expf(row[0] - Mu);
            L += row[1] * f;
            o0 += row[2 + 2 * jj] * f;
            o1 += row[3 + 2 * jj] * f;
          }
          *reinterpret_cast<__nv_bfloat162*>(A.att + (size_t)r * d + hh * 64 + 2 * jj) =
              __floats2bfloat162_rn(o0 / L, o1 / L);
          if (A.ml != nullptr && jj == 0) {
            A.ml[((size_t)r * H + hh) * 2 + 0] = M;
            A.ml[((size_t)r * H + hh) * 2 + 1] = L;
          }
        }
      }
    }
  }
  // every byte sent to a CTA is counted on its gbar / mbar and waited above;
  // the barrier keeps senders until their stores have landed
  cluster_sync();
  fr_stamp(A.trace, 7);
  tl_mark(A.tl, TL_EXIT);
}

template <int KSW>
struct Kern {
  static void* self() { return reinterpret_cast<void*>(&fr_self_kernel<KSW>); }
  static void* cross() { return reinterpret_cast<void*>(&fr_cross_kernel<KSW>); }
  static void* gemv(int mode, int ks) {
    if (mode == FR_RESID) return ks == FR_KS ? reinterpret_cast<void*>(&fr_gemv_kernel<KSW, FR_RESID, FR_KS>)
                                             : reinterpret_cast<void*>(&fr_gemv_kernel<KSW, FR_RESID, 1>);
    return reinterpret_cast<void*>(&fr_gemv_kernel<KSW, FR_GELU, 1>);
  }
};

void* pick(int d, int which, int mode = 0, int ks = 1) {
  switch (d) {
    case 512: return which == 0 ? Kern<4>::self() : which == 1 ? Kern<4>::cross() : Kern<4>::gemv(mode, ks);
    case 768: return which == 0 ? Kern<6>::self() : which == 1 ? Kern<6>::cross() : Kern<6>::gemv(mode, ks);
    case 1024: return which == 0 ? Kern<8>::self() : which == 1 ? Kern<8>::cross() : Kern<8>::gemv(mode, ks);
    case 1280: return which == 0 ? Kern<10>::self() : which == 1 ? Kern<10>::cross() : Kern<10>::gemv(mode, ks);
    default: return nullptr;
  }
}

cudaError_t launch_k(void* k, dim3 grid, size_t smem, cudaStream_t st, bool pdl, int cluster, void** args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(FR_T);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (cluster > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = cluster;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = 1;
    ++n;
  }
  if (pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelExC(&cfg, k, args);
}

// dst = src [N][K] (bf16, N % 8 == 0, K % 8 == 0) packed as the few-row
// kernels read their weights: 8-row tiles, each piece-major (see fr_mma_panel).
__global__ void fr_pack_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int N, int K) {
  const long long n = (long long)N * (K / 8);
  const int kc = K / 8;
  for (long long e = blockIdx.x * (long long)blockDim.x + threadIdx.x; e < n; e += (long long)gridDim.x * blockDim.x) {
    // destination piece e = (tile t, piece c, row r)
    const long long t = e / (8ll * kc);
    const int rem = (int)(e - t * 8ll * kc), c = rem >> 3, r = rem & 7;
    dst[e] = src[(8 * t + r) * kc + c];
  }
}

}  // namespace

cudaError_t launch_fr_pack(const void* src, void* dst, int N, int K, cudaStream_t st) {
  if (N % 8 || K % 8) return cudaErrorInvalidValue;
  fr_pack_kernel<<<1024, 256, 0, st>>>(static_cast<const uint4*>(src), static_cast<uint4*>(dst), N, K);
  return cudaGetLastError();
}

size_t fr_gemv_smem(int d, int K, int tiles_max, int ks) {
  return (size_t)gemv_smem_bytes(d, tiles_max, K / ks / d, ks);
}

size_t fr_head_smem(int d, int tiles_max, bool self_attn, int mrg_slots) {
  return (size_t)head_layout(d, tiles_max, self_attn ? 1 : 2, mrg_slots).total + 1024;
}

int fr_configure(int d, int F, int H, int max_pos, int* C_out, int* sms_out, int* gd_out) {
  if (pick(d, 0) == nullptr || F != FR_KS * d) return 0;
  int dev = 0, max_smem = 0, n_sm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  if (n_sm < 2 * FR_KS) return 0;
  // GEMVs: one wave, at most one CTA per SM; the MLP down-projection's
  // clusters of FR_KS: no more groups than can be resident at once
  const int nt_o = d / 8, nt_f = F / 8;
  const int g_o = std::min(nt_o, n_sm), g_f = std::min(nt_f, n_sm);
  int g_d = std::min(nt_o, n_sm / FR_KS);
  {
    const int t_d = (nt_o + g_d - 1) / g_d;
    void* k = pick(d, 2, FR_RESID, FR_KS);
    const size_t smem = fr_gemv_smem(d, F, FR_MAXT, FR_KS);
    if ((int)smem > max_smem || t_d > FR_MAXT ||
        cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
      return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(g_d * FR_KS);
    cfg.blockDim = dim3(FR_T);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = FR_KS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n_cl = 0;
    if (cudaOccupancyMaxActiveClusters(&n_cl, k, &cfg) != cudaSuccess) n_cl = 0;
    cudaGetLastError();
    g_d = std::min(g_d, n_cl);
    if (g_d < 1 || (nt_o + g_d - 1) / g_d > FR_MAXT) return 0;
  }
  const int gemv[3][4] = {{FR_RESID, 1, d, (nt_o + g_o - 1) / g_o},
                          {FR_GELU, 1, d, (nt_f + g_f - 1) / g_f},
                          {FR_RESID, FR_KS, F, (nt_o + g_d - 1) / g_d}};
  for (auto& g : gemv) {
    const size_t smem = fr_gemv_smem(d, g[2], g[3], g[1]);
    if (g[3] > FR_MAXT || (int)smem > max_smem) return 0;
    void* k = pick(d, 2, g[0], g[1]);
    if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)std::max(smem, g[1] == FR_KS ? fr_gemv_smem(d, F, FR_MAXT, FR_KS) : smem)) !=
        cudaSuccess)
      return 0;
  }
  *gd_out = g_d;
  // cluster size per head: the largest C <= 8 whose H clusters are resident at once
  const int mrg_self = (max_pos + FR_CH - 1) / FR_CH;
  for (int C = 8; C >= 3; --C) {
    if ((24 + C - 1) / C > FR_MAXT) continue;
    const size_t s_self = fr_head_smem(d, (24 + C - 1) / C, true, mrg_self);
    const size_t s_cross = fr_head_smem(d, (8 + C - 1) / C, false, C);
    if ((int)std::max(s_self, s_cross) > max_smem) continue;
    void* ks = pick(d, 0);
    void* kc = pick(d, 1);
    if (cudaFuncSetAttribute(ks, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)s_self) != cudaSuccess ||
        cudaFuncSetAttribute(kc, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)s_cross) != cudaSuccess)
      return 0;
    int ok = 1;
    for (int which = 0; which < 2 && ok; ++which) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(H * C);
      cfg.blockDim = dim3(FR_T);
      cfg.dynamicSmemBytes = which == 0 ? s_self : s_cross;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = C;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n_cl = 0;
      if (cudaOccupancyMaxActiveClusters(&n_cl, which == 0 ? ks : kc, &cfg) != cudaSuccess || n_cl < H) ok = 0;
    }
    cudaGetLastError();
    if (!ok) continue;
    *C_out = C;
    *sms_out = n_sm;
    return 1;
  }
  cudaGetLastError();
  return 0;
}

cudaError_t launch_fr_gemv(const FrGemv& a, int mode, int ks, int groups, int d, cudaStream_t st, bool pdl) {
  void* k = pick(d, 2, mode, ks);
  if (k == nullptr) return cudaErrorInvalidValue;
  void* args[] = {const_cast<FrGemv*>(&a)};
  return launch_k(k, dim3(groups * ks), fr_gemv_smem(d, a.K, a.tiles_max, ks), st, pdl, ks, args);
}

cudaError_t launch_fr_self(const CUtensorMap* kmap, const CUtensorMap* vmap, const FrHead& a, cudaStream_t st,
                           bool pdl) {
  void* k = pick(a.d, 0);
  if (k == nullptr) return cudaErrorInvalidValue;
  void* args[] = {const_cast<CUtensorMap*>(kmap), const_cast<CUtensorMap*>(vmap), const_cast<FrHead*>(&a)};
  return launch_k(k, dim3(a.H * a.C), fr_head_smem(a.d, a.tiles_max, true, a.mrg_slots), st, pdl, a.C, args);
}

cudaError_t launch_fr_cross(const CUtensorMap* xmap, const FrHead& a, cudaStream_t st, bool pdl) {
  void* k = pick(a.d, 1);
  if (k == nullptr) return cudaErrorInvalidValue;
  void* args[] = {const_cast<CUtensorMap*>(xmap), const_cast<FrHead*>(&a)};
  return launch_k(k, dim3(a.H * a.C), fr_head_smem(a.d, a.tiles_max, false, a.mrg_slots), st, pdl, a.C, args);
}

}  // namespace asrspec
