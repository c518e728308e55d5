// tcgen05 tensor-core GEMM for the decoder projections, the LM head and the
// per-utterance cross-attention K/V build.
//
// C[m][n] = sum_k A[m][k] B[n][k], A and B bf16 and K-major, fp32 accumulators
// in tensor memory.  One CTA computes one 128 x BN output tile (optionally one
// split of its K range):
//   warp 0 / lane 0 : TMA producer, STAGES-deep ring of (A, B) k-blocks
//   warp 1 / lane 0 : issues tcgen05.mma (M=128, N=BN, K=16) x 4 per k-block
//   warps 0..3      : epilogue, each reading its 32 TMEM lanes (= 32 values of m)
// Split K, two ways, both summing the partials in split order so that results
// do not depend on CTA timing:
//   * cluster split (CLU): the splits of a tile form one thread-block cluster
//     and CTA r of the cluster owns rows [r * 128 / splits, (r + 1) * 128 /
//     splits) of the tile.  Narrow tiles (BN <= 64) push: every CTA writes
//     each row of its partial straight into the owner's receive buffer with
//     st.async, which counts the bytes on the owner's mbarrier, so an owner
//     waits for exactly its own data and no cluster-wide barrier sits on the
//     critical path.  Wide tiles pull: each CTA stages its partial, and after
//     a cluster barrier the owners read the slices through distributed shared
//     memory.  Either way the owner sums its rows over the splits and runs
//     the epilogue on them;
//   * workspace split: partials go to a global workspace and the last CTA of
//     the tile (atomic ticket) sums them.
#include <cstdio>
#include <mutex>

#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_gemm_tc)

constexpr int TC_BM = 128;
constexpr int TC_BK = 64;

template <int BN, bool PUSH = false>
struct TcCfg {
  // 4-deep ring for narrow tiles; 3-deep for 128-wide tiles, and for 64-wide
  // tiles with a receive buffer, so that two CTAs share an SM (one CTA's
  // epilogue overlaps the other's main loop)
  static constexpr int STAGES = (BN == 128 || (PUSH && BN == 64)) ? 3 : 4;
  static constexpr int A_BYTES = TC_BM * TC_BK * 2;
  static constexpr int B_BYTES = BN * TC_BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int BAR_OFF = STAGES * STAGE_BYTES;
  // push split: receive buffer [split][row of the owner's slice][RECV_LD]
  // (= 128 rows), padded by 16 bytes per row against bank conflicts
  static constexpr int RECV_LD = BN + 4;
  static constexpr int RECV_OFF = BAR_OFF + 256;
  static constexpr int RECV_BYTES = PUSH ? TC_BM * RECV_LD * 4 : 0;
  static constexpr int SMEM = 1024 + BAR_OFF + 256 + RECV_BYTES;
  // tcgen05.alloc takes a power of two of at least 32 columns
  static constexpr uint32_t TMEM_COLS = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "N tile of one tcgen05.mma (M = 128)");
  static_assert(B_BYTES % 1024 == 0, "B tile must keep 1024-byte alignment");
};


template <int BN, int MODE, bool CLU>
__global__ void __launch_bounds__(128, 1)
gemm_tc_kernel(const __grid_constant__ CUtensorMap mapA, const __grid_constant__ CUtensorMap mapB, int K, int splits,
               float* __restrict__ ws, int* __restrict__ tickets, Epi epi, int* status) {
  constexpr bool PUSH = CLU && BN <= 64;
  using C = TcCfg<BN, PUSH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + C::STAGES * C::A_BYTES;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
  uint64_t* empty = full + C::STAGES;
  uint64_t* done = empty + C::STAGES;
  uint64_t* recv_bar = done + 1;   // push split: the peers' partial rows have landed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 2);
  float* recv = reinterpret_cast<float*>(smem + C::RECV_OFF);
  __shared__ unsigned long long red[4][BN];
  __shared__ int s_last;
  __shared__ float ln_mu[BN], ln_rs[BN];   // folded LayerNorm: statistics of the tile's rows

  // Grid: cluster split: (M tiles x splits, N tiles), the splits of a tile
  // consecutive along x (one cluster); otherwise (N tiles, M tiles, splits), so
  // that the CTAs sharing a weight tile run together and read it from HBM once.
  int tile_m = CLU ? (int)blockIdx.x / splits : (int)blockIdx.y;
  const int split = CLU ? (int)blockIdx.x % splits : (int)blockIdx.z;
  int tile_n = CLU ? (int)blockIdx.y : (int)blockIdx.x;
  if (!CLU && epi.group_m > 0) {   // grouped order: a band of group_m M tiles sweeps the N tiles
    const int mt = (epi.M + TC_BM - 1) / TC_BM, nt = (epi.N + BN - 1) / BN;
    const int band = (int)blockIdx.x / (epi.group_m * nt);
    const int r = (int)blockIdx.x - band * epi.group_m * nt;
    const int gm = min(epi.group_m, mt - band * epi.group_m);
    tile_m = band * epi.group_m + r % gm;
    tile_n = r / gm;
  }
  const int m0 = tile_m * TC_BM, n0 = tile_n * BN;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const unsigned cta_id = blockIdx.x + gridDim.x * (blockIdx.y + gridDim.y * blockIdx.z);
  unsigned long long* tr =
      epi.trace && cta_id < FR_TRACE_CTAS ? epi.trace + (unsigned long long)FR_TRACE_PHASES * cta_id : nullptr;
  if (tr && threadIdx.x == 0) tr[0] = global_ns();
  tl_mark(epi.tl, TL_ENTRY);
  const int n_valid = epi.n_valid ? *epi.n_valid : epi.N;
  const int nkb_total = K / TC_BK;
  const int kb0 = (nkb_total * split) / splits;
  const int kb1 = (nkb_total * (split + 1)) / splits;
  const int nkb = kb1 - kb0;
  bool dead = false;   // encoder-cache build: every frame of the tile is padding
  if constexpr (MODE == EPI_CROSSKV) {
    dead = true;
    for (int mr = m0; mr < m0 + TC_BM && mr < epi.M;) {   // one segment per utterance in the tile
      const int b = mr / epi.t_max, t = mr - b * epi.t_max;
      if (t < epi.enc_len[b]) {
        dead = false;
        break;
      }
      mr = (b + 1) * epi.t_max;
    }
  }
  if (n0 >= n_valid || nkb <= 0 || dead) {   // uniform over the CTA and over all splits of a tile
    pdl_wait();
    return;
  }

  if (warp == 0) {
    __syncwarp();   // warp-aligned allocation
    tmem_alloc(tmem_slot, C::TMEM_COLS);
    tmem_relinquish();
  }
  if (threadIdx.x == 32) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(done, 1);
    if constexpr (PUSH) {
      // the other splits each send this CTA's slice of their partial tile
      mbar_init(recv_bar, 1);
      mbar_arrive_expect_tx(recv_bar, (uint32_t)((splits - 1) * (TC_BM / splits) * BN * 4));
    }
    fence_mbar_init();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // push split: announce this CTA's receive barrier; the matching wait comes
  // just before the first remote store, long after every peer has arrived
  if constexpr (PUSH) cluster_arrive_relaxed();
  const uint32_t tmem = *tmem_slot;
  if (tr && threadIdx.x == 0) tr[1] = global_ns();

  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&mapA);
    tma_prefetch_desc(&mapB);
    // The weights (A) do not depend on the previous kernel: fill the ring with
    // them first, then wait for the predecessor before loading activations (B).
    constexpr uint32_t TX = C::STAGE_BYTES;
    const int first = nkb < C::STAGES ? nkb : C::STAGES;
    for (int i = 0; i < first; ++i) {
      mbar_arrive_expect_tx(&full[i], TX);
      tma_load_2d(sA + i * C::A_BYTES, &mapA, &full[i], (kb0 + i) * TC_BK, m0);
    }
    pdl_wait();
    tl_mark(epi.tl, TL_WORK);
    if (tr) tr[8] = global_ns();
    for (int i = 0; i < first; ++i) tma_load_2d(sB + i * C::B_BYTES, &mapB, &full[i], (kb0 + i) * TC_BK, n0);
    pdl_launch();
    int issued = first;
    for (int i = first; i < nkb; ++i) {
      const int s = i % C::STAGES;
      const uint32_t ph = (i / C::STAGES) & 1;
      if (!mbar_wait(&empty[s], ph ^ 1, status)) break;
      mbar_arrive_expect_tx(&full[s], TX);
      tma_load_2d(sA + s * C::A_BYTES, &mapA, &full[s], (kb0 + i) * TC_BK, m0);
      tma_load_2d(sB + s * C::B_BYTES, &mapB, &full[s], (kb0 + i) * TC_BK, n0);
      issued = i + 1;
    }
    if (tr) tr[9] = global_ns();
    // Drain: every issued copy has landed before this CTA can exit.
    for (int i = issued - C::STAGES > 0 ? issued - C::STAGES : 0; i < issued; ++i)
      mbar_wait(&full[i % C::STAGES], (i / C::STAGES) & 1, status);
  } else if (warp == 1 && lane == 0) {
    constexpr uint32_t idesc = umma_idesc_bf16(TC_BM, BN);
    for (int i = 0; i < nkb; ++i) {
      const int s = i % C::STAGES;
      const uint32_t ph = (i / C::STAGES) & 1;
      if (!mbar_wait(&full[s], ph, status)) break;
      if (tr && i == 0) tr[2] = global_ns();
      tc_fence_after();
      const uint32_t a_addr = smem_u32(sA + s * C::A_BYTES);
      const uint32_t b_addr = smem_u32(sB + s * C::B_BYTES);
#pragma unroll
      for (int kk = 0; kk < TC_BK / 16; ++kk)
        umma_bf16(tmem, umma_desc_sw128(a_addr + kk * 32), umma_desc_sw128(b_addr + kk * 32), idesc,
                  (i | kk) != 0);
      umma_commit(&empty[s]);
    }
    umma_commit(done);
  }
  if (!(warp == 0 && lane == 0)) {
    pdl_wait();
    pdl_launch();
  }
  // Folded LayerNorm: warps 2-3 (idle during the main loop) combine the row
  // statistics of the tile's rows from the producer's slices (equal slice
  // sizes: mean = average of slice means, M2 = sum of slice M2 + c * sum of
  // squared deviations of the slice means), 64 / BN threads per row.
  if (epi.ln_part != nullptr && warp >= 2) {
    const int t = threadIdx.x - 64;
    constexpr int TPR = BN >= 64 ? 1 : 64 / BN;   // threads per row (a power of two)
    const int S = epi.ln_S;
    for (int rl = t / TPR; rl < BN; rl += 64 / TPR) {
      const int n = n0 + rl;
      const int sub = t % TPR;
      const bool ok = n < n_valid;
      const float2* pr = epi.ln_part + (ok ? n : 0);
      // one pass, shifted by the first slice's mean (well conditioned when the
      // slice means are close to the row mean): with e_s = mean_s - shift,
      // mean = shift + E/S and M2 = sum M2_s + c (sum e_s^2 - E^2 / S)
      const float shift = ok ? pr[0].x : 0.f;
      float e1 = 0.f, e2 = 0.f, m2 = 0.f;
      if (ok)
#pragma unroll 8
        for (int j = sub; j < S; j += TPR) {
          const float2 p = pr[(size_t)j * epi.ln_stride];
          const float es = p.x - shift;
          e1 += es;
          e2 += es * es;
          m2 += p.y;
        }
#pragma unroll
      for (int o = TPR / 2; o > 0; o >>= 1) {
        e1 += __shfl_xor_sync(0xffffffffu, e1, o);
        e2 += __shfl_xor_sync(0xffffffffu, e2, o);
        m2 += __shfl_xor_sync(0xffffffffu, m2, o);
      }
      const float mean = shift + e1 / (float)S;
      const float q = m2 + (float)epi.ln_c * fmaxf(e2 - e1 * e1 / (float)S, 0.f);
      if (sub == 0) {
        ln_mu[rl] = ok ? mean : 0.f;
        ln_rs[rl] = ok ? rsqrtf(q / (float)(S * epi.ln_c) + 1e-5f) : 0.f;
      }
    }
  }
  // Push split: this thread's first-pass outputs of the owner's slice, and
  // their other operands (bias, residual, row metadata) loaded now, while the
  // MMAs run.  Item it = (row r of the slice, 4 columns c4).
  constexpr int EM = MODE == EPI_ARGMAX ? EPI_F32 : MODE;
  constexpr int IU = 4;
  const int rows_per = TC_BM / splits;
  const int r_first = split * rows_per;
  const int items = rows_per * (BN / 4);
  auto item_coords = [&](int base, int* mm, int* nn, bool* ok) {
#pragma unroll
    for (int u = 0; u < IU; ++u) {
      const int it = base + u * (int)blockDim.x;
      const int r = it % rows_per, c4 = it / rows_per;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        mm[4 * u + i] = m0 + r_first + r;
        nn[4 * u + i] = n0 + 4 * c4 + i;
        ok[4 * u + i] = it < items && m0 + r_first + r < epi.M && n0 + 4 * c4 + i < n_valid;
      }
    }
  };
  int pm[4 * IU], pn[4 * IU];
  bool pok[4 * IU];
  EpiPre<EM, 4 * IU> pre;
  if constexpr (PUSH) {
    item_coords(threadIdx.x, pm, pn, pok);
    epi_load<EM, 4 * IU>(epi, pm, pn, pok, pre);
  }
  __syncwarp();
  mbar_wait(done, 0, status);
  if (tr && threadIdx.x == 0) tr[3] = global_ns();
  tl_mark(epi.tl, TL_MID);
  __syncwarp();   // the warp leaves the wait together: the TMEM loads below are warp-aligned
  tc_fence_after();

  const int m = m0 + warp * 32 + lane;
  const uint32_t t_lane = tmem + ((uint32_t)(warp * 32) << 16);

  if (rowwise_mode<MODE>() && splits == 1) {
    // Stage the tile as [n][m] in the pipeline buffers (every copy has landed
    // and every MMA retired), then write whole rows.
    constexpr int LDS = TC_BM + 4;
    float* stg = reinterpret_cast<float*>(smem);
    const int ml = warp * 32 + lane;
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(t_lane + c0, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) stg[(c0 + i) * LDS + ml] = v[i];
    }
    if (tr && threadIdx.x == 0) tr[5] = global_ns();
    __syncthreads();
    if (tr && threadIdx.x == 0) tr[6] = global_ns();
    const int rows = n_valid - n0 < BN ? n_valid - n0 : BN;
    epi_rows<MODE>(epi, stg, LDS, m0 + 4 * lane, 4 * lane, n0, warp, rows, ln_mu, ln_rs);
    if (tr && threadIdx.x == 0) tr[7] = global_ns();
  } else if (splits == 1) {
    // encoder-cache build: this thread's frame (utterance fb, frame ft) and whether it is real
    const int fb = MODE == EPI_CROSSKV ? m / epi.t_max : 0, ft = MODE == EPI_CROSSKV ? m - fb * epi.t_max : 0;
    const bool frame_ok = MODE == EPI_CROSSKV && m < epi.M && ft < epi.enc_len[fb];
    const bool fold = epi.ln_part != nullptr && MODE != EPI_CROSSKV;
    float c1m = 0.f, c2m = 0.f;
    if (fold) {
      __syncthreads();   // the row statistics of warps 2-3
      if (m < epi.M) {
        c1m = __ldg(epi.ln_c1 + m);
        c2m = __ldg(epi.ln_c2 + m);
      }
    }
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(t_lane + c0, v);
      if (fold) {   // y = rstd (acc - mu c1) + c2
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = ln_rs[c0 + i] * (v[i] - ln_mu[c0 + i] * c1m) + c2m;
      }
      if constexpr (MODE == EPI_ARGMAX) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int n = n0 + c0 + i;
          unsigned long long key = (m < epi.M && n < n_valid) ? argmax_key(v[i], (uint32_t)m) : 0ull;
          key = warp_max_u64(key);
          if (lane == 0) red[warp][c0 + i] = key;
        }
      } else if constexpr (MODE == EPI_CROSSKV) {
        // 16 consecutive features of one frame lie in one head: one index, two
        // 16-byte stores (bf16) per thread
        if (frame_ok && n0 + c0 < n_valid) {
          const int n = n0 + c0, two_d = 2 * epi.d;
          const int l = n / two_d, r = n - l * two_d;
          const int which = r / epi.d, f = r - which * epi.d;
          const size_t idx =
              (((((size_t)l * 2 + which) * epi.b_max + fb) * epi.n_heads + (f >> 6)) * epi.max_enc + ft) * 64 + (f & 63);
          float w[16];
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const float4 bq = __ldg(reinterpret_cast<const float4*>(epi.bias + n) + q);
            w[4 * q + 0] = v[4 * q + 0] + bq.x;
            w[4 * q + 1] = v[4 * q + 1] + bq.y;
            w[4 * q + 2] = v[4 * q + 2] + bq.z;
            w[4 * q + 3] = v[4 * q + 3] + bq.w;
          }
          if (epi.kv_bf16) {
            uint32_t pk[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              __nv_bfloat162 t2 = __floats2bfloat162_rn(w[2 * q], w[2 * q + 1]);
              pk[q] = *reinterpret_cast<uint32_t*>(&t2);
            }
            uint4* dst = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(epi.kcache) + idx);
            dst[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            dst[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
          } else {
            float4* dst = reinterpret_cast<float4*>(static_cast<float*>(epi.kcache) + idx);
#pragma unroll
            for (int q = 0; q < 4; ++q) dst[q] = make_float4(w[4 * q], w[4 * q + 1], w[4 * q + 2], w[4 * q + 3]);
          }
        }
      } else {
        int mm[16], nn[16];
        bool ok[16];
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          mm[i] = m;
          nn[i] = n0 + c0 + i;
          ok[i] = m < epi.M && nn[i] < n_valid;
        }
        epi_batch<MODE, 16>(epi, mm, nn, v, ok);
      }
    }
    if constexpr (MODE == EPI_ARGMAX) {
      __syncthreads();
      for (int c = threadIdx.x; c < BN; c += blockDim.x) {
        const int n = n0 + c;
        unsigned long long k = red[0][c];
#pragma unroll
        for (int w = 1; w < 4; ++w) k = red[w][c] > k ? red[w][c] : k;
        if (n < n_valid) atomicMax(epi.row_key + n, k);
      }
    }
  } else if constexpr (PUSH) {
    cluster_wait();   // every peer's receive barrier is initialised
    const int ml = warp * 32 + lane;
    const uint32_t owner = (uint32_t)(ml / rows_per);
    // this split's copy of row ml sits at the same offset in the owner's buffer
    float* slot = recv + (split * rows_per + ml % rows_per) * C::RECV_LD;
    const bool mine = owner == (uint32_t)split;
    const uint32_t dst = dsmem_addr(slot, owner);
    const uint32_t bar = dsmem_addr(recv_bar, owner);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(t_lane + c0, v);   // whole warp (tcgen05.ld is warp-aligned); only the stores branch
#pragma unroll
      for (int i = 0; i < 16; i += 4) {
        const float4 q = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
        if (mine) *reinterpret_cast<float4*>(slot + c0 + i) = q;
        else st_async_f4(dst + (uint32_t)(c0 + i) * 4u, q, bar);
      }
    }
    if (tr && threadIdx.x == 0) tr[5] = global_ns();
    __syncthreads();                    // own slice written by this CTA's threads
    mbar_wait(recv_bar, 0, status);     // the peers' slices
    if (tr && threadIdx.x == 0) tr[6] = global_ns();
    // sum rows [split * rows_per, (split + 1) * rows_per) over the splits, in split order
    for (int base = threadIdx.x; base < items; base += IU * blockDim.x) {
      int mm[4 * IU], nn[4 * IU];
      bool ok[4 * IU];
      float vals[4 * IU];
      item_coords(base, mm, nn, ok);
#pragma unroll
      for (int u = 0; u < IU; ++u) {
        const int it = base + u * blockDim.x;
        const int r = it % rows_per, c4 = it / rows_per;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        if (it < items) {
          const float* src = recv + r * C::RECV_LD + 4 * c4;
#pragma unroll 4
          for (int s2 = 0; s2 < splits; ++s2) {
            const float4 p = *reinterpret_cast<const float4*>(src + s2 * rows_per * C::RECV_LD);
            acc.x += p.x; acc.y += p.y; acc.z += p.z; acc.w += p.w;
          }
        }
        vals[4 * u + 0] = acc.x;
        vals[4 * u + 1] = acc.y;
        vals[4 * u + 2] = acc.z;
        vals[4 * u + 3] = acc.w;
      }
      // the first pass's operands were loaded during the main loop; later passes load theirs now
      if (base != (int)threadIdx.x) epi_load<EM, 4 * IU>(epi, mm, nn, ok, pre);
      const EpiPre<EM, 4 * IU>& op = pre;
      if constexpr (EM != EPI_RESID) {
        if (epi.ln_part != nullptr) {   // folded LayerNorm: y = rstd (acc - mu c1) + c2
#pragma unroll
          for (int k = 0; k < 4 * IU; ++k) {
            if (!ok[k]) continue;
            const int nl = nn[k] - n0;
            vals[k] = ln_rs[nl] * (vals[k] - ln_mu[nl] * op.c1[k]) + op.c2[k];
          }
        }
      }
      epi_store<EM, 4 * IU>(epi, mm, nn, vals, ok, op);
      if constexpr (EM == EPI_RESID) {
        if (epi.xg != nullptr) {
          // the next LayerNorm's operand bf16(g * x), and x staged as [feature
          // of the slice][row] in the pipeline buffers (free since the MMAs
          // retired) for the slice statistics below
          float* xt = reinterpret_cast<float*>(smem);
#pragma unroll
          for (int k = 0; k < 4 * IU; ++k) {
            if (!ok[k]) continue;
            const float xn = op.old[k] + (vals[k] + op.bias[k]);   // the value just stored
            epi.xg[(size_t)nn[k] * epi.d + mm[k]] = __float2bfloat16_rn(op.gain[k] * xn);
            xt[(mm[k] - m0 - r_first) * (BN + 4) + (nn[k] - n0)] = xn;
          }
        }
      }
    }
    if constexpr (EM == EPI_RESID) {
      if (epi.xg != nullptr) {
        // Statistics of this owner's slice (rows_per features) of every row:
        // one thread per row sums its column of the staged tile.
        const float* xt = reinterpret_cast<const float*>(smem);
        __syncthreads();
        for (int c = threadIdx.x; c < BN; c += blockDim.x) {
          const int n = n0 + c;
          if (n >= n_valid) continue;
          float sm = 0.f;
          for (int r = 0; r < rows_per; ++r) sm += xt[r * (BN + 4) + c];
          const float mean = sm / (float)rows_per;
          float q = 0.f;
          for (int r = 0; r < rows_per; ++r) {
            const float dv = xt[r * (BN + 4) + c] - mean;
            q += dv * dv;
          }
          epi.st_part[(size_t)((m0 + r_first) / rows_per) * epi.st_stride + n] = make_float2(mean, q);
        }
      }
    }
    if (tr && threadIdx.x == 0) tr[7] = global_ns();
  } else if constexpr (CLU) {
    // stage this split's tile in shared memory (the pipeline buffers are free now)
    constexpr int LD = BN + 4;
    float* red = reinterpret_cast<float*>(smem);
    const int ml = warp * 32 + lane;
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(t_lane + c0, v);
#pragma unroll
      for (int i = 0; i < 16; i += 4)
        *reinterpret_cast<float4*>(red + ml * LD + c0 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
    if (tr && threadIdx.x == 0) tr[5] = global_ns();
    cluster_sync();
    if (tr && threadIdx.x == 0) tr[6] = global_ns();
    // this CTA sums rows [rank * 128 / splits, (rank + 1) * 128 / splits) over all
    // splits, IU float4 loads from every split in flight per pass
    for (int base = threadIdx.x; base < items; base += IU * blockDim.x) {
      float4 acc[IU];
      const float* local[IU];
      int mm[4 * IU], nn[4 * IU];
      bool ok[4 * IU];
#pragma unroll
      for (int u = 0; u < IU; ++u) {
        const int it = base + u * blockDim.x;
        const int row = r_first + (it % rows_per), c4 = it / rows_per;
        local[u] = red + row * LD + 4 * (c4 < BN / 4 ? c4 : 0);
        acc[u] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          mm[4 * u + i] = m0 + row;
          nn[4 * u + i] = n0 + 4 * c4 + i;
          ok[4 * u + i] = it < items && m0 + row < epi.M && n0 + 4 * c4 + i < n_valid;
        }
      }
      for (int s = 0; s < splits; ++s) {
        float4 p[IU];
#pragma unroll
        for (int u = 0; u < IU; ++u) p[u] = ld_dsmem_f4(dsmem_addr(local[u], (uint32_t)s));
#pragma unroll
        for (int u = 0; u < IU; ++u) {
          acc[u].x += p[u].x; acc[u].y += p[u].y; acc[u].z += p[u].z; acc[u].w += p[u].w;
        }
      }
      float vals[4 * IU];
#pragma unroll
      for (int u = 0; u < IU; ++u) {
        vals[4 * u + 0] = acc[u].x;
        vals[4 * u + 1] = acc[u].y;
        vals[4 * u + 2] = acc[u].z;
        vals[4 * u + 3] = acc[u].w;
      }
      epi_batch<MODE == EPI_ARGMAX ? EPI_F32 : MODE, 4 * IU>(epi, mm, nn, vals, ok);
    }
    if (tr && threadIdx.x == 0) tr[7] = global_ns();
    cluster_sync();   // no CTA leaves while another may still read its shared memory
  } else {
    const int tile = tile_n * ((epi.M + TC_BM - 1) / TC_BM) + tile_m;
    float* my = ws + ((size_t)(tile * splits + split) * TC_BM + warp * 32 + lane) * BN;
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 16) {
      float v[16];
      tmem_ld16(t_lane + c0, v);
#pragma unroll
      for (int i = 0; i < 16; i += 4)
        *reinterpret_cast<float4*>(my + c0 + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = (atomicAdd(tickets + tile, 1) == splits - 1);
    __syncthreads();
    if (s_last) {
      __threadfence();
      const float* base = ws + ((size_t)tile * splits * TC_BM + warp * 32 + lane) * BN;
      const int c_end = min(BN, ((n_valid - n0) + 3) & ~3);   // columns past the valid rows are not read
#pragma unroll 1
      for (int c0 = 0; c0 < c_end; c0 += 16) {
        // 16 columns x all splits in flight before the (split-ordered) sums
        float4 acc[4];
#pragma unroll
        for (int q = 0; q < 4; ++q) acc[q] = __ldcg(reinterpret_cast<const float4*>(base + c0 + 4 * q));
        int s = 1;
        for (; s + 2 <= splits; s += 2) {   // two splits' loads in flight, summed in split order
          float4 p[2][4];
#pragma unroll
          for (int u = 0; u < 2; ++u) {
            const float* ps = base + (size_t)(s + u) * TC_BM * BN + c0;
#pragma unroll
            for (int q = 0; q < 4; ++q) p[u][q] = __ldcg(reinterpret_cast<const float4*>(ps + 4 * q));
          }
#pragma unroll
          for (int u = 0; u < 2; ++u)
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              acc[q].x += p[u][q].x; acc[q].y += p[u][q].y; acc[q].z += p[u][q].z; acc[q].w += p[u][q].w;
            }
        }
        for (; s < splits; ++s) {
          float4 p[4];
          const float* ps = base + (size_t)s * TC_BM * BN + c0;
#pragma unroll
          for (int q = 0; q < 4; ++q) p[q] = __ldcg(reinterpret_cast<const float4*>(ps + 4 * q));
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            acc[q].x += p[q].x; acc[q].y += p[q].y; acc[q].z += p[q].z; acc[q].w += p[q].w;
          }
        }
        int mm[16], nn[16];
        bool ok[16];
        float vals[16];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          vals[4 * q + 0] = acc[q].x;
          vals[4 * q + 1] = acc[q].y;
          vals[4 * q + 2] = acc[q].z;
          vals[4 * q + 3] = acc[q].w;
        }
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          mm[i] = m;
          nn[i] = n0 + c0 + i;
          ok[i] = m < epi.M && nn[i] < n_valid;
        }
        epi_batch<MODE == EPI_ARGMAX ? EPI_F32 : MODE, 16>(epi, mm, nn, vals, ok);
      }
      if (threadIdx.x == 0) tickets[tile] = 0;
    }
  }

  if (tr && threadIdx.x == 0) tr[4] = global_ns();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
  tl_mark(epi.tl, TL_EXIT);
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------
using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPoint("cuTensorMapEncodeTiled", &p, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

bool make_tmap_bf16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (cols * 2) % 16) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool make_tmap_f32(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols, uint32_t box_cols,
                   uint32_t box_rows) {
  EncodeTiledFn fn = get_encode_fn();
  if (!fn) return false;
  if ((reinterpret_cast<uintptr_t>(base) & 15) || (cols * 4) % 16 || (box_cols * 4) % 16) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 4};
  cuuint32_t box[2] = {box_cols, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

int tc_pick_bn(int n_max) {
  if (n_max <= 16) return 16;
  if (n_max <= 32) return 32;
  if (n_max <= 64) return 64;
  if (n_max <= 128) return 128;
  return 256;
}

size_t tc_smem_bytes(int bn) {
  switch (bn) {
    case 16: return TcCfg<16>::SMEM;
    case 32: return TcCfg<32>::SMEM;
    case 64: return TcCfg<64>::SMEM;
    case 128: return TcCfg<128>::SMEM;
    case 192: return TcCfg<192>::SMEM;
    case 224: return TcCfg<224>::SMEM;
    default: return TcCfg<256>::SMEM;
  }
}

// N tile for many rows: fewest tiles first, then the least padding.
int tc_pick_bn_wide(int n) {
  const int cand[4] = {128, 192, 224, 256};
  int best = 256, best_nt = 1 << 30, best_pad = 1 << 30;
  for (int c : cand) {
    const int nt = (n + c - 1) / c, pad = nt * c - n;
    if (nt < best_nt || (nt == best_nt && pad < best_pad)) {
      best = c;
      best_nt = nt;
      best_pad = pad;
    }
  }
  return best;
}

template <int BN, int MODE>
static void launch_tc_t(const TcGemm& g, const Epi& epi, int* status, cudaStream_t st) {
  const int mt = (g.M + TC_BM - 1) / TC_BM, nt = (g.N + BN - 1) / BN;
  if (g.cluster && g.splits > 1) {
    launch_ex(gemm_tc_kernel<BN, MODE, true>, dim3(mt * g.splits, nt, 1), dim3(128),
              TcCfg<BN, (BN <= 64)>::SMEM, st, g.pdl, g.splits, g.mapA, g.mapB, g.K, g.splits, g.ws, g.tickets, epi,
              status);
    return;
  }
  const dim3 grid = epi.group_m > 0 ? dim3(nt * mt, 1, g.splits) : dim3(nt, mt, g.splits);
  launch_ex(gemm_tc_kernel<BN, MODE, false>, grid, dim3(128), TcCfg<BN>::SMEM, st, g.pdl, 1, g.mapA, g.mapB,
            g.K, g.splits, g.ws, g.tickets, epi, status);
}

template <int MODE>
static void launch_tc_mode(const TcGemm& g, const Epi& epi, int* status, cudaStream_t st) {
  switch (g.bn) {
    case 16: launch_tc_t<16, MODE>(g, epi, status, st); break;
    case 32: launch_tc_t<32, MODE>(g, epi, status, st); break;
    case 64: launch_tc_t<64, MODE>(g, epi, status, st); break;
    case 128: launch_tc_t<128, MODE>(g, epi, status, st); break;
    case 192: launch_tc_t<192, MODE>(g, epi, status, st); break;
    case 224: launch_tc_t<224, MODE>(g, epi, status, st); break;
    default: launch_tc_t<256, MODE>(g, epi, status, st); break;
  }
}

template <int BN, int MODE>
static void configure_one() {
  cudaFuncSetAttribute(gemm_tc_kernel<BN, MODE, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       TcCfg<BN>::SMEM);
  cudaFuncSetAttribute(gemm_tc_kernel<BN, MODE, true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                       TcCfg<BN, (BN <= 64)>::SMEM);
  cudaFuncSetAttribute(gemm_tc_kernel<BN, MODE, true>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
}

template <int MODE>
static void configure_mode() {
  configure_one<16, MODE>();
  configure_one<32, MODE>();
  configure_one<64, MODE>();
  configure_one<128, MODE>();
  configure_one<192, MODE>();
  configure_one<224, MODE>();
  configure_one<256, MODE>();
}

// Opt every instance into its dynamic shared memory once, before any launch or
// stream capture.
void configure_gemm_tc() {
  static std::once_flag once;
  std::call_once(once, [] {
    configure_mode<EPI_F32>();
    configure_mode<EPI_F32_MN>();
    configure_mode<EPI_QKV>();
    configure_mode<EPI_RESID>();
    configure_mode<EPI_Q>();
    configure_mode<EPI_GELU>();
    configure_mode<EPI_CROSSKV>();
    configure_mode<EPI_ARGMAX>();
  });
}

void launch_gemm_tc(const TcGemm& g, int mode, const Epi& epi, int* status, cudaStream_t st) {
  configure_gemm_tc();
  switch (mode) {
    case EPI_F32: launch_tc_mode<EPI_F32>(g, epi, status, st); break;
    case EPI_F32_MN: launch_tc_mode<EPI_F32_MN>(g, epi, status, st); break;
    case EPI_QKV: launch_tc_mode<EPI_QKV>(g, epi, status, st); break;
    case EPI_RESID: launch_tc_mode<EPI_RESID>(g, epi, status, st); break;
    case EPI_Q: launch_tc_mode<EPI_Q>(g, epi, status, st); break;
    case EPI_GELU: launch_tc_mode<EPI_GELU>(g, epi, status, st); break;
    case EPI_CROSSKV: launch_tc_mode<EPI_CROSSKV>(g, epi, status, st); break;
    case EPI_ARGMAX: launch_tc_mode<EPI_ARGMAX>(g, epi, status, st); break;
  }
}

}  // namespace asrspec
