// tcgen05 GEMM for the projections of many verify rows (more than 64): one
// 128 x BN output tile per CTA and about one CTA per SM, so that every SM
// streams with a deep pipeline and the weights are re-read as few times as the
// SM count allows (BN is picked from the rows and the SM count).
//
//   P = WG_PIPES pipelines, each over every P-th k-block with its own ring of
//   (A, B) stages and its own accumulator in tensor memory:
//   warp 2p / lane 0     : TMA producer of pipeline p; pipeline 0 also loads
//                          the tile of the residual stream x that a residual
//                          projection adds to (one TMA box, during the main loop)
//   warp 2p + 1 / lane 0 : issues pipeline p's tcgen05.mma (M = 128, N = BN,
//                          K = 16), 4 per k-block, over its accumulators
//   warps 2 P .. 7  : during the main loop, the tile's per-feature operands
//                     and row data (the folded LayerNorm's row statistics, the
//                     cache slots of the rows)
//   warps 4 - 7     : after the MMAs, the accumulators, summed in a fixed
//                     order, out of tensor memory into shared memory
//   warps 0 - 7     : the epilogue, one row per warp at a time, 4 features per lane
//
// Long K (at least 48 k-blocks) splits in two over a cluster pair: both CTAs
// stage their partial tile, and each sums half of the rows in rank order
// (rank 0 + rank 1, reading the peer's half through distributed shared
// memory), so that results do not depend on timing.
#pragma once

#include "kernels.h"

namespace asrspec {

constexpr int WG_THREADS = 256;
constexpr int WG_DYN_MAX = 220 * 1024;   // dynamic shared memory budget of one CTA
// independent TMA -> MMA pipelines per CTA: a producer/consumer hand-off
// through an mbarrier pair takes a fixed ~380 cycles however deep the ring
// (measured), so one pipeline moves one k-block per ~0.3 us; pipelines run
// side by side
constexpr int WG_PIPES = 3;
static_assert(2 * WG_PIPES <= 6, "warps 0 .. 2 P - 1 hold the pipeline roles; at least two warps stay free");

template <int BN, int MODE>
struct WideCfg {
  static constexpr int A_BYTES = 128 * 64 * 2;
  static constexpr int B_BYTES = BN * 64 * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int XT_BYTES = MODE == EPI_RESID ? BN * 128 * 4 : 0;   // residual tile [BN][128] fp32
  static constexpr int LDS = 128 + 4;                                     // staged tile row stride (floats)
  static constexpr int FIT = (WG_DYN_MAX - 1024 - 256 - XT_BYTES) / STAGE_BYTES;
  static constexpr int STAGES = FIT < 8 ? FIT : 8;
  // dynamic shared memory for s stages per pipeline (the staged tile reuses the ring)
  static constexpr int smem_bytes(int s) { return 1024 + WG_PIPES * s * STAGE_BYTES + XT_BYTES + 256; }
  static constexpr int SMEM = smem_bytes(STAGES / WG_PIPES);
  // accumulators, split over the pipelines (within a pipeline the K = 16
  // steps of a k-block rotate over its share)
  static constexpr int NACC = WG_PIPES;
  static constexpr uint32_t TMEM_COLS = NACC * BN <= 128 ? 128 : NACC * BN <= 256 ? 256 : 512;
  static constexpr int BN_MAX = 512 / WG_PIPES / 32 * 32;
  static_assert(STAGES >= 2 * WG_PIPES, "each pipeline needs two stages");
  static_assert(NACC % WG_PIPES == 0, "accumulators split over the pipelines");
  static_assert(BN * LDS * 4 <= WG_PIPES * STAGE_BYTES, "the staged tile must fit a one-stage ring");
  static_assert(BN % 32 == 0 && BN >= 32 && NACC * BN <= 512, "N tile (the accumulators fill at most 512 columns)");
};

// GELU with erf from Abramowitz & Stegun, formula 7.1.28 (|error| <= 3e-7 in
// erf): for z = |x| / sqrt(2),
// erfc(z) ~= q = 1 / (1 + a1 z + a2 z^2 + ... + a6 z^6)^16, and
// gelu(x) = x / 2 (2 - q) for x >= 0, x / 2 q for x < 0 (no cancellation).
// One reciprocal and no exponential per value (z is clipped at 9, where q
// is below 1e-27, so that the 16th power stays finite).
__device__ __forceinline__ float gelu_as(float x) {
  const float z = fminf(fabsf(x) * 0.70710678118654752f, 9.0f);
  float p = fmaf(z, fmaf(z, fmaf(z, fmaf(z, fmaf(z, fmaf(z, 0.0000430638f, 0.0002765672f), 0.0001520143f),
                                         0.0092705272f), 0.0422820123f), 0.0705230784f), 1.0f);
  p *= p;
  p *= p;
  p *= p;
  p *= p;
  const float q = __fdividef(1.0f, p);
  return 0.5f * x * (x >= 0.f ? 2.0f - q : q);
}

template <int BN, int MODE, int SPLIT>
__global__ void __launch_bounds__(WG_THREADS, 1)
gemm_wide_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB,
                 const __grid_constant__ CUtensorMap mapX, int K, int S, Epi epi, int* status) {
  using C = WideCfg<BN, MODE>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  // layout for S stages per pipeline: A ring, B ring, residual tile, barriers
  const int NS = WG_PIPES * S;
  uint8_t* sA = smem;
  uint8_t* sB = smem + NS * C::A_BYTES;
  float* xt = reinterpret_cast<float*>(smem + NS * C::STAGE_BYTES);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + NS * C::STAGE_BYTES + C::XT_BYTES);
  uint64_t* empty = full + NS;
  uint64_t* done = empty + NS;   // [WG_PIPES]
  uint64_t* xbar = done + WG_PIPES;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(xbar + 1);
  __shared__ float ln_mu[BN], ln_rs[BN];   // folded LayerNorm: statistics of the tile's rows
  __shared__ int s_rb[BN], s_rp[BN];       // QKV: utterance and position of the tile's rows
  __shared__ __align__(16) float s_op[4][128];   // the tile's bias, folded-LayerNorm c1, c2, next gain

  const int split = SPLIT > 1 ? (int)blockIdx.x % SPLIT : 0;
  const int m0 = ((int)blockIdx.x / SPLIT) * 128, n0 = (int)blockIdx.y * BN;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned cta_id = blockIdx.x + gridDim.x * blockIdx.y;
  unsigned long long* tr =
      epi.trace && cta_id < FR_TRACE_CTAS ? epi.trace + (unsigned long long)FR_TRACE_PHASES * cta_id : nullptr;
  if (tr && threadIdx.x == 0) tr[0] = global_ns();
  tl_mark(epi.tl, TL_ENTRY);
  const int n_valid = epi.n_valid ? *epi.n_valid : epi.N;
  const int nkb_total = K / 64;
  const int kb0 = (nkb_total * split) / SPLIT, kb1 = (nkb_total * (split + 1)) / SPLIT;
  const int nkb = kb1 - kb0;
  if (n0 >= n_valid || nkb <= 0) {   // uniform over the CTA and over the pair of a split tile
    pdl_wait();
    return;
  }

  if (warp == 0) {
    __syncwarp();
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  if (threadIdx.x == 32) {
    for (int s = 0; s < NS; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int p = 0; p < WG_PIPES; ++p) mbar_init(&done[p], 1);
    mbar_init(xbar, 1);
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (tr && threadIdx.x == 0) tr[1] = global_ns();

  // pipeline p: k-blocks p, p + WG_PIPES, ...; its stages [p S, (p + 1) S); its
  // accumulators [p APP, (p + 1) APP)
  constexpr int APP = C::NACC / WG_PIPES;
  const int pipe = warp >> 1;
  if (warp < 2 * WG_PIPES && (warp & 1) == 0 && lane == 0) {   // producer of pipeline `pipe`
    const int np = (nkb - pipe + WG_PIPES - 1) / WG_PIPES;
    uint64_t* fb = full + pipe * S;
    uint64_t* eb = empty + pipe * S;
    uint8_t* pa = sA + pipe * S * C::A_BYTES;
    uint8_t* pb = sB + pipe * S * C::B_BYTES;
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    if constexpr (MODE == EPI_RESID) tma_prefetch_desc(&mapX);
    auto kcol = [&](int j) { return (kb0 + pipe + j * WG_PIPES) * 64; };
    // weights first (independent of the previous kernel), activations after its completion
    const int first = np < S ? np : S;
    for (int j = 0; j < first; ++j) {
      mbar_arrive_expect_tx(&fb[j], C::STAGE_BYTES);
      tma_load_2d(pa + j * C::A_BYTES, &mapA, &fb[j], kcol(j), m0);
    }
    pdl_wait();
    tl_mark(epi.tl, TL_WORK);
    if (tr && pipe == 0) tr[8] = global_ns();
    for (int j = 0; j < first; ++j) tma_load_2d(pb + j * C::B_BYTES, &mapB, &fb[j], kcol(j), n0);
    if constexpr (MODE == EPI_RESID) {   // x rows n0 .. n0 + BN, features m0 .. m0 + 128 (zero past the buffer)
      if (pipe == 0) {
        mbar_arrive_expect_tx(xbar, C::XT_BYTES);
        tma_load_2d(xt, &mapX, xbar, m0, n0);
      }
    }
    pdl_launch();
    int issued = first;
    for (int j = first; j < np; ++j) {
      const int s = j % S;
      if (!mbar_wait(&eb[s], ((j / S) & 1) ^ 1, status)) break;
      mbar_arrive_expect_tx(&fb[s], C::STAGE_BYTES);
      tma_load_2d(pa + s * C::A_BYTES, &mapA, &fb[s], kcol(j), m0);
      tma_load_2d(pb + s * C::B_BYTES, &mapB, &fb[s], kcol(j), n0);
      issued = j + 1;
    }
    if (tr && pipe == 0) tr[9] = global_ns();
    for (int j = issued - S > 0 ? issued - S : 0; j < issued; ++j)   // drain
      mbar_wait(&fb[j % S], (j / S) & 1, status);
  } else if (warp < 2 * WG_PIPES && lane == 0) {   // MMA issuer of pipeline `pipe`
    const int np = (nkb - pipe + WG_PIPES - 1) / WG_PIPES;
    uint64_t* fb = full + pipe * S;
    uint64_t* eb = empty + pipe * S;
    const uint32_t acc0 = tmem + (uint32_t)(pipe * APP * BN);
    constexpr uint32_t idesc = umma_idesc_bf16(128, BN);
    for (int j = 0; j < np; ++j) {
      const int s = j % S;
      if (!mbar_wait(&fb[s], (j / S) & 1, status)) break;
      if (tr && pipe == 0 && j == 0) tr[2] = global_ns();
      tc_fence_after();
      const uint32_t a_addr = smem_u32(sA + (pipe * S + s) * C::A_BYTES);
      const uint32_t b_addr = smem_u32(sB + (pipe * S + s) * C::B_BYTES);
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        umma_bf16(acc0 + (uint32_t)((kk % APP) * BN), umma_desc_sw128(a_addr + kk * 32),
                  umma_desc_sw128(b_addr + kk * 32), idesc, (j > 0 || kk >= APP) ? 1u : 0u);
      umma_commit(&eb[s]);
    }
    umma_commit(&done[pipe]);
  } else {
    pdl_wait();
    pdl_launch();
    if (warp >= 2 * WG_PIPES) {   // the warps without a pipeline role
      constexpr int NT = WG_THREADS - 64 * WG_PIPES;
      const int t = threadIdx.x - 64 * WG_PIPES;
      // the epilogue's per-feature operands of this tile
      for (int f = t; f < 128; f += NT) {
        s_op[0][f] = __ldg(epi.bias + m0 + f);
        if (epi.ln_part != nullptr && MODE != EPI_RESID) {
          s_op[1][f] = __ldg(epi.ln_c1 + m0 + f);
          s_op[2][f] = __ldg(epi.ln_c2 + m0 + f);
        }
        if (MODE == EPI_RESID && epi.xg != nullptr) s_op[3][f] = __ldg(epi.xg_gain + m0 + f);
      }
      // Folded LayerNorm: row statistics combined from the producer's equal
      // slices, one pass shifted by the first slice's mean:
      // mean = shift + E / S, M2 = sum M2_s + c (sum e_s^2 - E^2 / S)
      if (epi.ln_part != nullptr) {
        const int S = epi.ln_S;
        for (int rl = t; rl < BN; rl += NT) {
          const int n = n0 + rl;
          const bool ok = n < n_valid;
          const float2* pr = epi.ln_part + (ok ? n : 0);
          const float shift = ok ? pr[0].x : 0.f;
          float e1 = 0.f, e2 = 0.f, m2 = 0.f;
          if (ok)
            for (int j = 0; j < S; ++j) {
              const float2 p = pr[(size_t)j * epi.ln_stride];
              const float es = p.x - shift;
              e1 += es;
              e2 += es * es;
              m2 += p.y;
            }
          const float mean = shift + e1 / (float)S;
          const float q = m2 + (float)epi.ln_c * fmaxf(e2 - e1 * e1 / (float)S, 0.f);
          ln_mu[rl] = ok ? mean : 0.f;
          ln_rs[rl] = ok ? rsqrtf(q / (float)(S * epi.ln_c) + 1e-5f) : 0.f;
        }
      }
      if constexpr (MODE == EPI_QKV)
        for (int rl = t; rl < BN; rl += NT) {
          const int n = n0 + rl;
          s_rb[rl] = n < n_valid ? epi.row_b[n] : 0;
          s_rp[rl] = n < n_valid ? epi.row_pos[n] : 0;
        }
    }
  }

  // epilogue operands, loaded while the MMAs run: lane l covers features
  // mq .. mq + 3 of the tile (M % 128 == 0, so every lane's features exist);
  // warp w the rows r_lo + w, + 8, ...
  const int mq = m0 + 4 * lane;
  const bool fold = epi.ln_part != nullptr && MODE != EPI_RESID;
  int kind = 0, head = 0, col = 0;   // QKV: 0 query, 1 key, 2 value
  if constexpr (MODE == EPI_QKV) {
    if (mq >= epi.d) {
      const int f = mq - epi.d;
      kind = f >= epi.d ? 2 : 1;
      const int g = f - (kind - 1) * epi.d;
      head = g >> 6;
      col = g & 63;
    }
  }

  // every thread: the accumulators are final
  __syncwarp();
  const int pipes = nkb < WG_PIPES ? nkb : WG_PIPES;   // pipelines that ran k-blocks
  for (int p = 0; p < WG_PIPES; ++p) mbar_wait(&done[p], 0, status);
  if (tr && threadIdx.x == 0) tr[3] = global_ns();
  tl_mark(epi.tl, TL_MID);
  __syncwarp();
  tc_fence_after();
  // warps 4-7: tensor memory (lane = feature m, column = row n) -> stg[n][m]
  float* stg = reinterpret_cast<float*>(smem);
  if (warp >= 4) {
    const int wq = warp - 4, ml = wq * 32 + lane;
    const uint32_t t_lane = tmem + ((uint32_t)(wq * 32) << 16);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16], w[16];
      tmem_ld16(t_lane + c0, v);
#pragma unroll
      for (int a = 1; a < C::NACC; ++a) {   // the accumulators summed in a fixed order
        if (a / APP >= pipes) break;        // a pipeline without k-blocks wrote nothing
        tmem_ld16(t_lane + (uint32_t)(a * BN) + c0, w);
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] += w[i];
      }
#pragma unroll
      for (int i = 0; i < 16; ++i) stg[(c0 + i) * C::LDS + ml] = v[i];
    }
  }
  if (tr && threadIdx.x == 0) tr[5] = global_ns();
  __syncthreads();
  if constexpr (SPLIT > 1) cluster_sync();   // the peer's partial tile is staged too
  if (tr && threadIdx.x == 0) tr[6] = global_ns();

  if constexpr (MODE == EPI_RESID) mbar_wait(xbar, 0, status);   // the residual tile has landed
  const float4 bias = *reinterpret_cast<const float4*>(&s_op[0][4 * lane]);
  const float4 c1 = fold ? *reinterpret_cast<const float4*>(&s_op[1][4 * lane]) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float4 c2 = fold ? *reinterpret_cast<const float4*>(&s_op[2][4 * lane]) : make_float4(0.f, 0.f, 0.f, 0.f);
  const float4 gain = (MODE == EPI_RESID && epi.xg) ? *reinterpret_cast<const float4*>(&s_op[3][4 * lane])
                                                    : make_float4(0.f, 0.f, 0.f, 0.f);
  if (tr && threadIdx.x == 0) tr[10] = global_ns();
  const int r_lo = SPLIT > 1 ? split * (BN / 2) : 0;
  const int r_end = min(SPLIT > 1 ? r_lo + BN / 2 : BN, n_valid - n0);
  const uint32_t peer = (uint32_t)(split ^ 1);
  constexpr int RB = 4;   // rows per batch per warp, loads in flight together
  for (int j0 = r_lo + warp; j0 < r_end; j0 += 8 * RB) {
    if (tr && threadIdx.x == 0 && j0 == r_lo + 8 * RB) tr[11] = global_ns();
    float4 a[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int nl = j0 + 8 * r;
      a[r] = nl < r_end ? *reinterpret_cast<const float4*>(stg + nl * C::LDS + 4 * lane)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (SPLIT > 1) {   // rank 0's partial + rank 1's, in that order
        if (nl < r_end) {
          const float4 p = ld_dsmem_f4(dsmem_addr(stg + nl * C::LDS + 4 * lane, peer));
          a[r] = split == 0 ? make_float4(a[r].x + p.x, a[r].y + p.y, a[r].z + p.z, a[r].w + p.w)
                            : make_float4(p.x + a[r].x, p.y + a[r].y, p.z + a[r].z, p.w + a[r].w);
        }
      }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int nl = j0 + 8 * r;
      if (nl >= r_end) break;   // uniform over the warp
      const int n = n0 + nl;
      float4 v = a[r];
      if (fold) {   // y = rstd (acc - mu c1) + c2
        const float mu = ln_mu[nl], rs = ln_rs[nl];
        v = make_float4(rs * (v.x - mu * c1.x) + c2.x, rs * (v.y - mu * c1.y) + c2.y, rs * (v.z - mu * c1.z) + c2.z,
                        rs * (v.w - mu * c1.w) + c2.w);
      }
      v.x += bias.x;
      v.y += bias.y;
      v.z += bias.z;
      v.w += bias.w;
      if constexpr (MODE == EPI_Q) {
        *reinterpret_cast<float4*>(epi.out_f32 + (size_t)n * epi.d + mq) = v;
      } else if constexpr (MODE == EPI_GELU) {
        v = make_float4(gelu_as(v.x), gelu_as(v.y), gelu_as(v.z), gelu_as(v.w));
        __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
        *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(epi.act) + (size_t)n * epi.M + mq) =
            make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
      } else if constexpr (MODE == EPI_RESID) {
        const float4 o = *reinterpret_cast<const float4*>(xt + nl * 128 + 4 * lane);
        const float4 xn = make_float4(o.x + v.x, o.y + v.y, o.z + v.z, o.w + v.w);
        *reinterpret_cast<float4*>(epi.x + (size_t)n * epi.d + mq) = xn;
        if (epi.xg) {   // the next LayerNorm's operand and the statistics of this 128-feature slice
          __nv_bfloat162 lo = __floats2bfloat162_rn(gain.x * xn.x, gain.y * xn.y);
          __nv_bfloat162 hi = __floats2bfloat162_rn(gain.z * xn.z, gain.w * xn.w);
          *reinterpret_cast<uint2*>(epi.xg + (size_t)n * epi.d + mq) =
              make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
          const float mean = warp_sum((xn.x + xn.y) + (xn.z + xn.w)) * (1.f / 128.f);
          const float dx = xn.x - mean, dy = xn.y - mean, dz = xn.z - mean, dw = xn.w - mean;
          const float m2 = warp_sum((dx * dx + dy * dy) + (dz * dz + dw * dw));
          if (lane == 0) epi.st_part[(size_t)(m0 / 128) * epi.st_stride + n] = make_float2(mean, m2);
        }
      } else if constexpr (MODE == EPI_QKV) {
        if (kind == 0) {
          *reinterpret_cast<float4*>(epi.out_f32 + (size_t)n * epi.d + mq) = v;
        } else if (!qkv_slot_bad(epi, s_rb[nl], s_rp[nl])) {
          const size_t idx = (((size_t)s_rb[nl] * epi.n_heads + head) * epi.max_pos + s_rp[nl]) * 64 + col;
          __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
          *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(kind == 1 ? epi.kcache : epi.vcache) + idx) =
              make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
        }
      }
    }
  }
  if (tr && threadIdx.x == 0) tr[7] = global_ns();
  if constexpr (SPLIT > 1) cluster_sync();   // the peer has read this CTA's partial
  if (tr && threadIdx.x == 0) tr[4] = global_ns();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  tl_mark(epi.tl, TL_EXIT);
}

}  // namespace asrspec
