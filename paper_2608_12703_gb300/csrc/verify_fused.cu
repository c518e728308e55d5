// Fused verify for few rows: one persistent cooperative kernel for the decoder
// layers and the LM head of a verify step (Sec. 3 "Speculative Loop": the
// target scores the whole draft block in one pass).
//
// With at most VF_ROWS verify rows (batch 1 with up to 8 drafts) every
// projection is a matrix-vector-like product whose cost is its weight bytes,
// and a chain of ~8 dependent launches per layer spends most of its time in
// per-launch fixed costs.  Here one CTA per SM stays resident for the whole
// step:
//   * warp 8 (the producer) walks the step's projections in order and streams
//     this CTA's slice of each weight matrix (a contiguous run of 8-row tiles)
//     into a ring of shared-memory slots with 1-D bulk copies, one row per
//     copy into a padded row pitch (conflict-free ldmatrix); it runs ahead of
//     the compute warps across stage boundaries, so the weights of the next
//     projections are in flight while the current stage waits on the grid;
//   * warps 0-7 run the stages: input preparation (LayerNorm of the fp32
//     residual, or a copy of a bf16 activation) into shared memory, then
//     mma.sync m16n8k16 with the verify rows as the 16-row M side and 8 weight
//     rows as N, the K range of every chunk split over the 8 warps and the
//     partial tiles summed in warp order (deterministic), then the epilogue;
//     attention stages work per (utterance, head) (self) or per (utterance,
//     head, split of the encoder frames) (cross, TMA loads of 128-key chunks,
//     splits merged in split order by the last split to finish);
//   * a grid-wide barrier (release add, acquire poll, bounded) separates
//     dependent stages: 8 per layer.
// Numerics follow the multi-kernel chain: bf16 operands, fp32 accumulation,
// fp32 residual stream, LayerNorm statistics in fp32 from registers.
#include <mutex>

#include "kernels.h"

namespace asrspec {

namespace {

constexpr int VF_CT = 256;               // compute threads (warps 0-7)
constexpr int VF_THREADS = VF_CT + 32;   // + the producer warp
constexpr int VF_NSLOT = 5;              // weight ring slots (8 rows x d each)
constexpr int VF_GT = 4;                 // 8-row tiles reduced together
constexpr int VF_CH = 128;               // keys per attention chunk
constexpr int VF_TILE = VF_CH * 128;     // bytes of one chunk of K or V
constexpr int VF_RED = 8 * VF_GT * 128 * 4;

__device__ __forceinline__ void cbar() { asm volatile("bar.sync 1, 256;" ::: "memory"); }

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ uint32_t lds32(uint32_t addr) {
  uint32_t v;
  asm volatile("ld.shared.b32 %0, [%1];" : "=r"(v) : "r"(addr));
  return v;
}
__device__ __forceinline__ void mma16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t bf2_bits(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}
// byte offset of (row, 16-byte chunk) in a 128-byte-swizzled tile of 128-byte rows
__device__ __forceinline__ uint32_t sw128(int row, int c16) { return (uint32_t)(row * 128 + ((c16 ^ (row & 7)) << 4)); }

__device__ __forceinline__ void tile_range(int nt, int G, int c, int& t0, int& t1) {
  t0 = (int)((long long)nt * c / G);
  t1 = (int)((long long)nt * (c + 1) / G);
}

// Grid-wide barrier of the compute warps (the producer warp never joins).
// Returns false when a bounded wait anywhere in the grid has given up.
__device__ __forceinline__ bool grid_sync(unsigned* ctr, unsigned target, int* status, volatile int* s_flag) {
  cbar();
  if (threadIdx.x == 0) {
    int ok = 1;
    asm volatile("fence.acq_rel.gpu;" ::: "memory");
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
    const long long t0 = clock64();
    int spins = 0;
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if ((int)(v - target) >= 0) break;
      if ((++spins & 1023) == 0) {
        if (*reinterpret_cast<volatile int*>(status) & ST_WAIT_TIMEOUT) { ok = 0; break; }
        if (clock64() - t0 > (1ll << 31)) {
          set_status(status, ST_WAIT_TIMEOUT);
          ok = 0;
          break;
        }
      }
    }
    *s_flag = ok;
  }
  cbar();
  return *s_flag != 0;
}

struct Smem {
  uint8_t* act;    // activation rows / attention chunks
  uint8_t* ring;   // weight slots
  float* red;      // cross-warp partial tiles; attention (max, sum, output) per row
  uint64_t* full;
  uint64_t* empty;
  uint64_t* abar;
  uint64_t* lbar;  // LayerNorm gain and bias staged in `red` before the barrier
  unsigned long long* rkey;
  // copied from global memory at kernel start (shared memory is not affected
  // by the L1 invalidation of every grid barrier's acquire): the layer table,
  // per utterance (rows, first row, committed length, encoder frames) and per
  // row (utterance, position, token)
  const VfLayer* layers;
  const int *u_nr, *u_row0, *u_kv, *u_enc;
  const int *r_b, *r_pos, *r_tok;
  volatile int* flag;
  int slot;        // slot bytes
};

// ---- producer -----------------------------------------------------------------
// The chunk order must match gemm_stage: per group of VF_GT tiles, per K panel
// of d columns, per tile.
__device__ bool produce(const Smem& S, const __nv_bfloat16* W, int K, int N, int d, int G, int cta, uint32_t& pc,
                        int* status) {
  const int nt = (N + 7) >> 3;
  int t0, t1;
  tile_range(nt, G, cta, t0, t1);
  const int np = K / d;
  const uint32_t row_bytes = (uint32_t)d * 2u, pitch = row_bytes + 16u;
  for (int g0 = t0; g0 < t1; g0 += VF_GT) {
    const int g1 = min(g0 + VF_GT, t1);
    for (int p = 0; p < np; ++p)
      for (int t = g0; t < g1; ++t) {
        const int s = (int)(pc % VF_NSLOT);
        if (pc >= (uint32_t)VF_NSLOT && !mbar_wait(&S.empty[s], ((pc / VF_NSLOT) - 1) & 1, status)) return false;
        const int rows = min(8, N - 8 * t);
        uint8_t* dst = S.ring + (size_t)s * S.slot;
        mbar_arrive_expect_tx(&S.full[s], (uint32_t)rows * row_bytes);
        const __nv_bfloat16* src = W + (size_t)8 * t * K + (size_t)p * d;
        for (int r = 0; r < rows; ++r) bulk_load(dst + r * pitch, src + (size_t)r * K, row_bytes, &S.full[s]);
        ++pc;
      }
  }
  return true;
}

__device__ void producer_main(const VfArgs& A, const Smem& S, int G, int cta) {
  uint32_t pc = 0;
  const int d = A.d, F = A.F;
  bool ok = true;
  for (int l = 0; l < A.L && ok; ++l) {
    const VfLayer& w = S.layers[l];
    ok = produce(S, w.wqkv, d, 3 * d, d, G, cta, pc, A.status) && produce(S, w.wo, d, d, d, G, cta, pc, A.status) &&
         produce(S, w.wcq, d, d, d, G, cta, pc, A.status) && produce(S, w.wco, d, d, d, G, cta, pc, A.status) &&
         produce(S, w.w1, d, F, d, G, cta, pc, A.status) && produce(S, w.w2, F, d, d, G, cta, pc, A.status);
  }
  if (ok) ok = produce(S, A.tok_emb, d, A.V, d, G, cta, pc, A.status);
  // After a time-out the compute warps stop consuming: wait (bounded) for the
  // copies still in flight before the CTA exits.
  if (!ok) {
    const uint32_t first = pc > (uint32_t)VF_NSLOT ? pc - VF_NSLOT : 0u;
    for (uint32_t i = first; i < pc; ++i) {
      const long long t0 = clock64();
      while (!mbar_try_wait(&S.full[i % VF_NSLOT], (i / VF_NSLOT) & 1))
        if (clock64() - t0 > (1ll << 31)) break;
    }
  }
}

// ---- input preparation ------------------------------------------------------------
// Thread 0: the next LayerNorm's gain and bias (constants) into S.red, while
// the grid barrier before its stage is pending.  S.red must be free: called
// after the current stage's last CTA barrier.
__device__ __forceinline__ void ln_issue(const Smem& S, const float* g, const float* bta, int d) {
  if (threadIdx.x == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    mbar_arrive_expect_tx(S.lbar, (uint32_t)(8 * d));
    bulk_load(S.red, g, (uint32_t)(4 * d), S.lbar);
    bulk_load(S.red + d, bta, (uint32_t)(4 * d), S.lbar);
  }
}

// act[r][0..d) = bf16(LayerNorm(x_r) * g + b) for r < R: the rows of x are
// first copied into shared memory (past the bf16 rows) with 16-byte
// asynchronous copies, all in flight at once; then one warp per row (warp 0
// also row 8) reduces from shared memory.  g and b come from S.red (ln_issue,
// phase ln_n).  The first layer takes x_r = tok_emb[tok] + pos_emb[pos] and
// CTA 0 stores it.
template <int KSW>
__device__ void prep_ln(const VfArgs& A, const Smem& S, uint32_t ln_n, bool embed, bool write_xf, int R, int cta) {
  constexpr int D = KSW * 128;
  constexpr int XOFF = (VF_ROWS * (2 * D + 16) + 1023) & ~1023;   // fp32 rows after the bf16 rows
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const float4* xs = reinterpret_cast<const float4*>(S.act + XOFF);
  if (!embed) {
    const uint8_t* src = reinterpret_cast<const uint8_t*>(A.x);
    const uint32_t dst = smem_u32(S.act + XOFF);
    for (int i = threadIdx.x; i < R * D / 4; i += VF_CT)
      asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst + 16u * i), "l"(src + 16 * (size_t)i)
                   : "memory");
    asm volatile("cp.async.wait_all;" ::: "memory");
    cbar();
  }
  mbar_wait(S.lbar, ln_n & 1, A.status);
  const float4* g4 = reinterpret_cast<const float4*>(S.red);
  const float4* b4 = reinterpret_cast<const float4*>(S.red + D);
  for (int r = warp; r < R; r += 8) {
    float4 v[KSW];
    if (embed) {
      const int tok = S.r_tok[r], pos = S.r_pos[r];
      const uint2* te = reinterpret_cast<const uint2*>(A.tok_emb + (size_t)tok * D);
      const uint2* pe = reinterpret_cast<const uint2*>(A.pos_emb + (size_t)pos * D);
#pragma unroll
      for (int i = 0; i < KSW; ++i) {
        const uint2 a = __ldg(te + lane + 32 * i), b = __ldg(pe + lane + 32 * i);
        const __nv_bfloat162* ah = reinterpret_cast<const __nv_bfloat162*>(&a);
        const __nv_bfloat162* bh = reinterpret_cast<const __nv_bfloat162*>(&b);
        const float2 a0 = __bfloat1622float2(ah[0]), a1 = __bfloat1622float2(ah[1]);
        const float2 b0 = __bfloat1622float2(bh[0]), b1 = __bfloat1622float2(bh[1]);
        v[i] = make_float4(a0.x + b0.x, a0.y + b0.y, a1.x + b1.x, a1.y + b1.y);
        if (cta == 0) reinterpret_cast<float4*>(A.x + (size_t)r * D)[lane + 32 * i] = v[i];
      }
    } else {
#pragma unroll
      for (int i = 0; i < KSW; ++i) v[i] = xs[r * (D / 4) + lane + 32 * i];
    }
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < KSW; ++i) s += (v[i].x + v[i].y) + (v[i].z + v[i].w);
    const float mean = warp_sum(s) / (float)D;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < KSW; ++i) {
      const float a = v[i].x - mean, b = v[i].y - mean, c = v[i].z - mean, e = v[i].w - mean;
      q += (a * a + b * b) + (c * c + e * e);
    }
    const float rstd = rsqrtf(warp_sum(q) / (float)D + 1e-5f);
    uint8_t* arow = S.act + (size_t)r * (2 * D + 16);
#pragma unroll
    for (int i = 0; i < KSW; ++i) {
      const int c4 = lane + 32 * i;
      const float4 gg = g4[c4], bb = b4[c4];
      uint2 o;
      o.x = bf2_bits((v[i].x - mean) * rstd * gg.x + bb.x, (v[i].y - mean) * rstd * gg.y + bb.y);
      o.y = bf2_bits((v[i].z - mean) * rstd * gg.z + bb.z, (v[i].w - mean) * rstd * gg.w + bb.w);
      *reinterpret_cast<uint2*>(arow + 8 * c4) = o;
      if (write_xf && cta == 0) reinterpret_cast<uint2*>(A.xf + (size_t)r * D)[c4] = o;
    }
  }
}

// act[r][0..K) = src[r][0..K) (bf16) for r < R: 16-byte asynchronous copies
// through L2 (cp.async.cg), all in flight at once.
__device__ void prep_copy(const Smem& S, const __nv_bfloat16* src, int K, int R) {
  const int per_row = K >> 3;   // 16-byte pieces
  const int total = R * per_row;
  const uint8_t* s8 = reinterpret_cast<const uint8_t*>(src);
  const uint32_t dst0 = smem_u32(S.act);
  for (int i = threadIdx.x; i < total; i += VF_CT) {
    const int r = i / per_row, c = i - r * per_row;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst0 + (uint32_t)(r * (2 * K + 16) + 16 * c)),
                 "l"(s8 + 16 * (size_t)i)
                 : "memory");
  }
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// ---- projections ------------------------------------------------------------------
enum VfMode : int { VF_QKV = 0, VF_RESID = 1, VF_Q = 2, VF_GELU = 3, VF_ARGMAX = 4 };

struct VfEpi {
  int mode;
  const float* bias;
  float* out;                  // VF_Q
  __nv_bfloat16 *ks, *vs;      // VF_QKV cache append
};

// What one output (row r, feature m) needs besides its accumulator, loaded
// before the stage's MMAs: the bias, and the residual (VF_RESID) or the
// row's cache slot (VF_QKV).
struct VfPre {
  float bias, old;
  size_t slot;
};
__device__ __forceinline__ VfPre vf_load(const VfArgs& A, const Smem& S, const VfEpi& e, int r, int m) {
  VfPre p{0.f, 0.f, 0};
  const int d = A.d;
  if (e.mode != VF_ARGMAX) p.bias = __ldg(e.bias + m);
  if (e.mode == VF_RESID) p.old = __ldcg(A.x + (size_t)r * d + m);
  if (e.mode == VF_QKV && m >= d) {
    const int f = (m - d) % d;
    p.slot = (((size_t)S.r_b[r] * A.H + (f >> 6)) * A.max_pos + S.r_pos[r]) * 64 +
             (f & 63);
  }
  return p;
}

__device__ __forceinline__ void vf_apply(const VfArgs& A, const VfEpi& e, const Smem& S, int r, int m, float v,
                                         const VfPre& p) {
  const int d = A.d;
  switch (e.mode) {
    case VF_QKV: {
      const float y = v + p.bias;
      if (m < d) A.q[(size_t)r * d + m] = y;
      else ((m - d) < d ? e.ks : e.vs)[p.slot] = f2bf(y);
      break;
    }
    case VF_RESID: A.x[(size_t)r * d + m] = p.old + (v + p.bias); break;
    case VF_Q: e.out[(size_t)r * d + m] = v + p.bias; break;
    case VF_GELU: A.hbuf[(size_t)r * A.F + m] = f2bf(gelu_erf(v + p.bias)); break;
    default: atomicMax(&S.rkey[r], argmax_key(v, (uint32_t)m)); break;
  }
}

// C[r][m] = sum_k act[r][k] W[m][k] over this CTA's 8-row tiles of W, in
// groups of VF_GT tiles; act holds the R rows (stride K + 8) in shared memory.
template <int KSW>
__device__ void gemm_stage(const VfArgs& A, const Smem& S, int K, int N, const VfEpi& e, int R, int G, int cta,
                           uint32_t& cc) {
  constexpr int D = KSW * 128;
  constexpr int KW = D / 8;   // K columns per warp per panel
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int nt = (N + 7) >> 3;
  int t0, t1;
  tile_range(nt, G, cta, t0, t1);
  const int np = K / D;
  const uint32_t act_base = smem_u32(S.act), ring_base = smem_u32(S.ring);
  const int a_pitch = 2 * K + 16;
  // ldmatrix row addresses: A = rows (clamped to the valid ones), B = weight rows
  const int ar = min((lane & 7) + 8 * ((lane >> 3) & 1), R - 1);
  const uint32_t a_lane = act_base + (uint32_t)(ar * a_pitch) + 16u * (lane >> 4);
  const uint32_t b_lane = (uint32_t)((lane & 7) * (2 * D + 16) + 16 * (lane >> 3));

  for (int g0 = t0; g0 < t1; g0 += VF_GT) {
    const int ng = min(VF_GT, t1 - g0);
    const int n_out = ng * 8 * R;   // <= 2 * VF_CT
    VfPre pre[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int o = threadIdx.x + j * VF_CT;
      if (o < n_out) {
        const int i = o / (8 * R), rem = o - i * 8 * R;
        const int m = 8 * (g0 + i) + (rem & 7);
        if (m < N) pre[j] = vf_load(A, S, e, rem >> 3, m);
      }
    }
    float acc[VF_GT][4];
#pragma unroll
    for (int i = 0; i < VF_GT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
    for (int p = 0; p < np; ++p) {
      const int k0 = p * D + warp * KW;
      uint32_t af[KSW][4];
#pragma unroll
      for (int j = 0; j < KSW; ++j) ldsm_x4(a_lane + 2u * (uint32_t)(k0 + 16 * j), af[j]);
#pragma unroll
      for (int i = 0; i < VF_GT; ++i) {
        if (i < ng) {
          const int s = (int)(cc % VF_NSLOT);
          mbar_wait(&S.full[s], (cc / VF_NSLOT) & 1, A.status);
          __syncwarp();
          const uint32_t sb = ring_base + (uint32_t)(s * S.slot) + b_lane + 2u * (uint32_t)(warp * KW);
#pragma unroll
          for (int jj = 0; jj < KSW / 2; ++jj) {
            uint32_t b[4];
            ldsm_x4(sb + 64u * jj, b);
            mma16816(acc[i], af[2 * jj], b[0], b[1]);
            mma16816(acc[i], af[2 * jj + 1], b[2], b[3]);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&S.empty[s]);
          ++cc;
        }
      }
    }
    // partial tiles of the 8 warps, summed in warp order
#pragma unroll
    for (int i = 0; i < VF_GT; ++i) {
      if (i < ng) {
        float* o = S.red + (warp * VF_GT + i) * 128;
        *reinterpret_cast<float2*>(o + g * 8 + 2 * t) = make_float2(acc[i][0], acc[i][1]);
        *reinterpret_cast<float2*>(o + (g + 8) * 8 + 2 * t) = make_float2(acc[i][2], acc[i][3]);
      }
    }
    cbar();
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int o = threadIdx.x + j * VF_CT;
      if (o < n_out) {
        const int i = o / (8 * R), rem = o - i * 8 * R;
        const int r = rem >> 3, n = rem & 7;
        float v = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) v += S.red[(w * VF_GT + i) * 128 + r * 8 + n];
        const int m = 8 * (g0 + i) + n;
        if (m < N) vf_apply(A, e, S, r, m, v, pre[j]);
      }
    }
    cbar();
  }
}

// ---- attention -------------------------------------------------------------------
// Running (max, sum, output) of one warp's keys for up to 16 rows of one head.
struct AttnState {
  uint32_t qa[4][4];
  int lim[2];
  float m_run[2], l_run[2], O[8][4];
};

__device__ __forceinline__ void attn_init(AttnState& st, const float* q, int row0, int nr, int d, int hh,
                                          const int* row_pos, int n_keys, bool causal) {
  const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
  for (int kk = 0; kk < 4; ++kk)
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int c = hh * 64 + kk * 16 + half * 8 + 2 * t;
      float2 lo = make_float2(0.f, 0.f), hi = make_float2(0.f, 0.f);
      if (g < nr) lo = __ldcg(reinterpret_cast<const float2*>(q + (size_t)(row0 + g) * d + c));
      if (g + 8 < nr) hi = __ldcg(reinterpret_cast<const float2*>(q + (size_t)(row0 + g + 8) * d + c));
      st.qa[kk][half * 2 + 0] = bf2_bits(lo.x * 0.125f, lo.y * 0.125f);
      st.qa[kk][half * 2 + 1] = bf2_bits(hi.x * 0.125f, hi.y * 0.125f);
    }
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int r = g + 8 * e;
    st.lim[e] = (causal && r < nr) ? min(n_keys, row_pos[row0 + r] + 1) : n_keys;
    st.m_run[e] = -INFINITY;
    st.l_run[e] = 0.f;
  }
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) st.O[nd][0] = st.O[nd][1] = st.O[nd][2] = st.O[nd][3] = 0.f;
}

// One 128-key chunk (K at ks, V at vs, 128-byte swizzled); this warp takes
// keys [16 warp, 16 warp + 16) of it; key0 = index of the chunk's first key.
__device__ __forceinline__ void attn_chunk(AttnState& st, uint32_t ks, uint32_t vs, int key0) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  float Sf[2][4];
#pragma unroll
  for (int nt = 0; nt < 2; ++nt) {
    const int krow = warp * 16 + nt * 8 + g;
    Sf[nt][0] = Sf[nt][1] = Sf[nt][2] = Sf[nt][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      const uint32_t b0 = lds32(ks + sw128(krow, 2 * kk) + 4 * t);
      const uint32_t b1 = lds32(ks + sw128(krow, 2 * kk + 1) + 4 * t);
      mma16816(Sf[nt], st.qa[kk], b0, b1);
    }
  }
  const int kbase = key0 + warp * 16;
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    float cm = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        float& s = Sf[nt][2 * e + j];
        if (kbase + nt * 8 + 2 * t + j >= st.lim[e]) s = -INFINITY;
        cm = fmaxf(cm, s);
      }
    cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 1));
    cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, 2));
    const float m_new = fmaxf(st.m_run[e], cm);
    const float mu = (m_new == -INFINITY) ? 0.f : m_new;
    const float alpha = __expf(st.m_run[e] - mu);
    float l = 0.f;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        float& s = Sf[nt][2 * e + j];
        s = __expf(s - mu);
        l += s;
      }
    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    st.l_run[e] = st.l_run[e] * alpha + l;
    st.m_run[e] = m_new;
#pragma unroll
    for (int nd = 0; nd < 8; ++nd) {
      st.O[nd][2 * e + 0] *= alpha;
      st.O[nd][2 * e + 1] *= alpha;
    }
  }
  uint32_t pa[4];
  pa[0] = bf2_bits(Sf[0][0], Sf[0][1]);
  pa[1] = bf2_bits(Sf[0][2], Sf[0][3]);
  pa[2] = bf2_bits(Sf[1][0], Sf[1][1]);
  pa[3] = bf2_bits(Sf[1][2], Sf[1][3]);
  const int q4 = lane >> 3, rr = lane & 7;
  const int vrow = warp * 16 + (q4 & 1) * 8 + rr;
#pragma unroll
  for (int nd2 = 0; nd2 < 4; ++nd2) {
    uint32_t r[4];
    ldsm_x4_t(vs + sw128(vrow, nd2 * 2 + (q4 >> 1)), r);
    mma16816(st.O[2 * nd2], pa, r[0], r[1]);
    mma16816(st.O[2 * nd2 + 1], pa, r[2], r[3]);
  }
}

// Combine the 8 warps into (Pm, Pl, Po) per row (in S.red); uses S.act as
// scratch, so every chunk load into S.act must be complete.
__device__ __forceinline__ void attn_combine(const AttnState& st, const Smem& S, int nr, float* mw, float* lw) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  float* Ow = reinterpret_cast<float*>(S.act);   // [8][16][64]
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int r = g + 8 * e;
    if (t == 0) {
      mw[warp * 16 + r] = st.m_run[e];
      lw[warp * 16 + r] = st.l_run[e];
    }
#pragma unroll
    for (int nd = 0; nd < 8; ++nd)
      *reinterpret_cast<float2*>(Ow + (warp * 16 + r) * 64 + nd * 8 + 2 * t) =
          make_float2(st.O[nd][2 * e], st.O[nd][2 * e + 1]);
  }
  cbar();
  float* Pm = S.red;
  float* Pl = S.red + 16;
  float* Po = S.red + 32;
  for (int e = threadIdx.x; e < nr * 64; e += VF_CT) {
    const int r = e >> 6, c = e & 63;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < 8; ++w) M = fmaxf(M, mw[w * 16 + r]);
    const float Mu = (M == -INFINITY) ? 0.f : M;
    float L = 0.f, o = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) {
      const float f = __expf(mw[w * 16 + r] - Mu);
      L += lw[w * 16 + r] * f;
      o += Ow[(w * 16 + r) * 64 + c] * f;
    }
    Po[r * 64 + c] = o;
    if (c == 0) {
      Pm[r] = M;
      Pl[r] = L;
    }
  }
  cbar();
}

// Self-attention: one CTA per (utterance, head); keys 0..kv_len + rows - 1 of
// the layer's cache (this step's rows were appended by the QKV stage), two
// 128-key chunks at a time, loaded through registers into swizzled tiles.
__device__ void self_stage(const VfArgs& A, const Smem& S, const VfLayer& w, int G, int cta, float* mw, float* lw) {
  const int H = A.H, d = A.d;
  for (int item = cta; item < A.B * H; item += G) {
    const int b = item / H, hh = item - b * H;
    const int nr = S.u_nr[b];
    if (nr == 0) continue;
    const int row0 = S.u_row0[b];
    const int n_keys = S.u_kv[b] + nr;
    const int nc = (n_keys + VF_CH - 1) / VF_CH;
    const size_t head0 = ((size_t)b * H + hh) * A.max_pos * 64;
    const uint4* kg = reinterpret_cast<const uint4*>(w.ks + head0);
    const uint4* vg = reinterpret_cast<const uint4*>(w.vs + head0);
    AttnState st;
    attn_init(st, A.q, row0, nr, d, hh, S.r_pos, n_keys, true);
    const uint32_t base = smem_u32(S.act);
    for (int j0 = 0; j0 < nc; j0 += 2) {
      uint4 kr[8], vr[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {   // (chunk j0 + u / 4, 128-byte key row, 16-byte piece)
        const int e = threadIdx.x + VF_CT * (u & 3);
        const int key = (j0 + (u >> 2)) * VF_CH + (e >> 3);
        if (key < n_keys) {
          kr[u] = __ldcg(kg + (size_t)key * 8 + (e & 7));
          vr[u] = __ldcg(vg + (size_t)key * 8 + (e & 7));
        } else {
          kr[u] = vr[u] = make_uint4(0u, 0u, 0u, 0u);
        }
      }
      cbar();   // the previous chunks are consumed
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int e = threadIdx.x + VF_CT * (u & 3);
        uint8_t* buf = S.act + (u >> 2) * 2 * VF_TILE;
        *reinterpret_cast<uint4*>(buf + sw128(e >> 3, e & 7)) = kr[u];
        *reinterpret_cast<uint4*>(buf + VF_TILE + sw128(e >> 3, e & 7)) = vr[u];
      }
      cbar();
      for (int u = 0; u < 2 && j0 + u < nc; ++u)
        attn_chunk(st, base + u * 2 * VF_TILE, base + u * 2 * VF_TILE + VF_TILE, (j0 + u) * VF_CH);
    }
    cbar();
    attn_combine(st, S, nr, mw, lw);
    const float* Pl = S.red + 16;
    const float* Po = S.red + 32;
    for (int e = threadIdx.x; e < nr * 64; e += VF_CT) {
      const int r = e >> 6, c = e & 63;
      A.att[(size_t)(row0 + r) * d + hh * 64 + c] = f2bf(Po[r * 64 + c] / Pl[r]);
    }
    cbar();
  }
}

struct CrossItem {
  int b, hh, split, nr, row0, T, nc, n_iter;
};
__device__ __forceinline__ CrossItem cross_item(const VfArgs& A, const Smem& S, int item) {
  CrossItem c;
  const int bh = item / A.S;
  c.split = item - bh * A.S;
  c.b = bh / A.H;
  c.hh = bh - c.b * A.H;
  c.nr = S.u_nr[c.b];
  c.row0 = S.u_row0[c.b];
  c.T = S.u_enc[c.b];
  c.nc = (c.T + VF_CH - 1) / VF_CH;
  c.n_iter = (c.nr > 0 && c.split < c.nc) ? (c.nc - c.split + A.S - 1) / A.S : 0;
  return c;
}

// Thread 0: chunk i of an item's split into attention buffer (n % 2).
__device__ __forceinline__ void cross_issue(const VfArgs& A, const Smem& S, const CUtensorMap* xmap, int l,
                                            const CrossItem& c, int i, uint32_t n) {
  const int buf = (int)(n & 1);
  const long long per_half = (long long)A.b_max * A.H * A.t_alloc;
  const long long krow = (long long)l * 2 * per_half + ((long long)c.b * A.H + c.hh) * A.t_alloc +
                         (long long)(c.split + i * A.S) * VF_CH;
  uint8_t* dst = S.act + buf * 2 * VF_TILE;
  mbar_arrive_expect_tx(&S.abar[buf], 2 * VF_TILE);
  tma_load_2d(dst, xmap, &S.abar[buf], 0, (int)krow);
  tma_load_2d(dst + VF_TILE, xmap, &S.abar[buf], 0, (int)(krow + per_half));
}

// Thread 0, after this CTA's query projection: the first chunks of its first
// cross-attention item (the encoder cache is constant during the step).
__device__ __forceinline__ int cross_prefetch(const VfArgs& A, const Smem& S, const CUtensorMap* xmap, int l, int cta,
                                              uint32_t an) {
  if (cta >= A.B * A.H * A.S) return 0;
  const CrossItem c = cross_item(A, S, cta);
  const int n = min(2, c.n_iter);
  if (threadIdx.x == 0) {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
    for (int i = 0; i < n; ++i) cross_issue(A, S, xmap, l, c, i, an + i);
  }
  return n;
}

// Cross-attention: one CTA per (utterance, head, split); split s takes chunks
// s, s + S, ... of the utterance's encoder frames; the last split to finish
// merges the splits' (max, sum, output) in split order.  At the anchor layer
// the full softmax (max, sum) per (row, head) is kept for the anchor readout.
__device__ void cross_stage(const VfArgs& A, const Smem& S, const CUtensorMap* xmap, int l, int G, int cta,
                            uint32_t& an, int prefetched, float* mw, float* lw) {
  const int d = A.d, H = A.H;
  const float* qc = (l == A.anchor) ? A.q_anchor : A.q;
  float* ml = (l == A.anchor) ? A.ml : nullptr;
  bool first = true;
  for (int item = cta; item < A.B * H * A.S; item += G) {
    const CrossItem c = cross_item(A, S, item);
    const int issued = first ? prefetched : 0;
    first = false;
    if (c.n_iter == 0) continue;
    const uint32_t base = an - (uint32_t)issued;   // counter of this item's chunk 0
    if (threadIdx.x == 0) {
      if (issued == 0) asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      for (int i = issued; i < min(2, c.n_iter); ++i) cross_issue(A, S, xmap, l, c, i, base + i);
    }
    AttnState st;
    attn_init(st, qc, c.row0, c.nr, d, c.hh, S.r_pos, c.T, false);
    const uint32_t sbase = smem_u32(S.act);
    for (int i = 0; i < c.n_iter; ++i) {
      const uint32_t n = base + i;
      const int buf = (int)(n & 1);
      mbar_wait(&S.abar[buf], (n >> 1) & 1, A.status);
      __syncwarp();
      attn_chunk(st, sbase + buf * 2 * VF_TILE, sbase + buf * 2 * VF_TILE + VF_TILE, (c.split + i * A.S) * VF_CH);
      cbar();   // every warp is done with this buffer
      if (threadIdx.x == 0 && i + 2 < c.n_iter) cross_issue(A, S, xmap, l, c, i + 2, n + 2);
    }
    an = base + (uint32_t)c.n_iter;
    attn_combine(st, S, c.nr, mw, lw);
    const float* Pm = S.red;
    const float* Pl = S.red + 16;
    const float* Po = S.red + 32;
    const int s_eff = min(A.S, c.nc);
    const int bh = c.b * H + c.hh;
    if (s_eff == 1) {
      for (int e = threadIdx.x; e < c.nr * 64; e += VF_CT) {
        const int r = e >> 6, cc = e & 63;
        A.att[(size_t)(c.row0 + r) * d + c.hh * 64 + cc] = f2bf(Po[r * 64 + cc] / Pl[r]);
        if (ml && cc == 0) {
          ml[((size_t)(c.row0 + r) * H + c.hh) * 2 + 0] = Pm[r];
          ml[((size_t)(c.row0 + r) * H + c.hh) * 2 + 1] = Pl[r];
        }
      }
    } else {
      float* mine = A.part + ((size_t)bh * A.S + c.split) * VF_ROWS * 66;
      for (int e = threadIdx.x; e < c.nr * 66; e += VF_CT) {
        const int r = e / 66, k = e - r * 66;
        mine[r * 66 + k] = k == 0 ? Pm[r] : (k == 1 ? Pl[r] : Po[r * 64 + k - 2]);
      }
      cbar();
      if (threadIdx.x == 0) {   // release this split's rows, acquire the others' when last
        int old;
        asm volatile("fence.acq_rel.gpu;" ::: "memory");
        asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(A.tickets + bh) : "memory");
        *S.flag = (old == s_eff - 1);
      }
      cbar();
      if (*S.flag) {
        // every split's rows into shared memory at once (float2 pieces), then merge
        const float2* all = reinterpret_cast<const float2*>(A.part + (size_t)bh * A.S * VF_ROWS * 66);
        float2* sp = reinterpret_cast<float2*>(S.act);   // [s_eff][VF_ROWS][33]
        const int per_split = c.nr * 33, n2 = s_eff * per_split;
        for (int base = threadIdx.x; base < n2; base += VF_CT * 8) {
          float2 v[8];
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int i = base + u * VF_CT;
            if (i < n2) {
              const int s2 = i / per_split;
              v[u] = __ldcg(all + s2 * VF_ROWS * 33 + (i - s2 * per_split));
            }
          }
#pragma unroll
          for (int u = 0; u < 8; ++u) {
            const int i = base + u * VF_CT;
            if (i < n2) {
              const int s2 = i / per_split;
              sp[s2 * VF_ROWS * 33 + (i - s2 * per_split)] = v[u];
            }
          }
        }
        cbar();
        const float* pf = reinterpret_cast<const float*>(S.act);
        for (int e = threadIdx.x; e < c.nr * 64; e += VF_CT) {
          const int r = e >> 6, cc = e & 63;
          float M = -INFINITY;
          for (int s2 = 0; s2 < s_eff; ++s2) M = fmaxf(M, pf[(s2 * VF_ROWS + r) * 66]);
          const float Mu = (M == -INFINITY) ? 0.f : M;
          float L = 0.f, o = 0.f;
          for (int s2 = 0; s2 < s_eff; ++s2) {
            const float* row = pf + (s2 * VF_ROWS + r) * 66;
            const float f = __expf(row[0] - Mu);
            L += row[1] * f;
            o += row[2 + cc] * f;
          }
          A.att[(size_t)(c.row0 + r) * d + c.hh * 64 + cc] = f2bf(o / L);
          if (ml && cc == 0) {
            ml[((size_t)(c.row0 + r) * H + c.hh) * 2 + 0] = M;
            ml[((size_t)(c.row0 + r) * H + c.hh) * 2 + 1] = L;
          }
        }
        if (threadIdx.x == 0) A.tickets[bh] = 0;
      }
    }
    cbar();
  }
}

// ---- the kernel -------------------------------------------------------------------
template <int KSW>
__global__ void __launch_bounds__(VF_THREADS, 1)
verify_fused_kernel(const __grid_constant__ CUtensorMap xmap, const __grid_constant__ VfArgs A) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[VF_NSLOT], empty[VF_NSLOT], abar[2], lbar;
  __shared__ unsigned long long rkey[VF_ROWS];
  __shared__ float mw[8 * 16], lw[8 * 16];
  __shared__ int flag;
  constexpr int D = KSW * 128;
  Smem S;
  S.act = sm;
  S.ring = sm + A.a_bytes;
  S.red = reinterpret_cast<float*>(S.ring + (size_t)VF_NSLOT * A.slot_bytes);
  S.full = full;
  S.empty = empty;
  S.abar = abar;
  S.lbar = &lbar;
  S.rkey = rkey;
  S.flag = &flag;
  S.slot = A.slot_bytes;
  uint8_t* tab = reinterpret_cast<uint8_t*>(S.red) + VF_RED;
  VfLayer* lt = reinterpret_cast<VfLayer*>(tab);
  int* it = reinterpret_cast<int*>(tab + (size_t)A.L * sizeof(VfLayer));
  S.layers = lt;
  S.u_nr = it;
  S.u_row0 = it + VF_ROWS;
  S.u_kv = it + 2 * VF_ROWS;
  S.u_enc = it + 3 * VF_ROWS;
  S.r_b = it + 4 * VF_ROWS;
  S.r_pos = it + 5 * VF_ROWS;
  S.r_tok = it + 6 * VF_ROWS;
  const int G = gridDim.x, cta = blockIdx.x, tid = threadIdx.x;
  tl_mark(A.tl, TL_ENTRY);
  const int R = *A.plan.n_rows;   // written by the row plan (an earlier launch)
  if (R <= 0 || R > VF_ROWS) return;   // a refused step: nothing to score
  if (tid == 0) {
    for (int s = 0; s < VF_NSLOT; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 8);
    }
    mbar_init(&abar[0], 1);
    mbar_init(&abar[1], 1);
    mbar_init(&lbar, 1);
    fence_mbar_init();
  }
  if (tid < VF_ROWS) rkey[tid] = 0ull;
  {
    const unsigned long long* src = reinterpret_cast<const unsigned long long*>(A.layers);
    unsigned long long* dst = reinterpret_cast<unsigned long long*>(lt);
    for (int i = tid; i < A.L * (int)(sizeof(VfLayer) / 8); i += VF_THREADS) dst[i] = src[i];
    if (tid < VF_ROWS) {
      const bool ub = tid < A.B;
      it[tid] = ub ? A.plan.n_utt_rows[tid] : 0;
      it[VF_ROWS + tid] = ub ? A.plan.row_start[tid] : 0;
      it[2 * VF_ROWS + tid] = ub ? A.kv_len[tid] : 0;
      it[3 * VF_ROWS + tid] = ub ? A.enc_len[tid] : 0;
      const bool ur = tid < R;
      it[4 * VF_ROWS + tid] = ur ? A.plan.row_b[tid] : 0;
      it[5 * VF_ROWS + tid] = ur ? A.plan.row_pos[tid] : 0;
      it[6 * VF_ROWS + tid] = ur ? A.plan.row_tok[tid] : 0;
    }
  }
  __syncthreads();
  tl_mark(A.tl, TL_WORK);
  if (tid >= VF_CT) {
    if (tid == VF_CT) producer_main(A, S, G, cta);
    return;
  }

  uint32_t cc = 0, an = 0, target = 0, ln_n = 0;
  const int d = D, F = A.F;
  unsigned long long* trace = A.trace ? A.trace + (size_t)cta * vf_trace_points(A.L) : nullptr;
  auto stamp = [&](int i) {
    if (trace != nullptr && tid == 0) trace[i] = global_ns();
  };
  auto sync = [&]() {
    target += (unsigned)G;
    return grid_sync(A.bar_ctr, target, A.status, &flag);
  };
  ln_issue(S, S.layers[0].ln1g, S.layers[0].ln1b, d);
  for (int l = 0; l < A.L; ++l) {
    const VfLayer& w = S.layers[l];
    const int t0 = 16 * l;
    stamp(t0);
    // self-attention block
    prep_ln<KSW>(A, S, ln_n++, l == 0, false, R, cta);
    cbar();
    gemm_stage<KSW>(A, S, d, 3 * d, VfEpi{VF_QKV, w.bqkv, nullptr, w.ks, w.vs}, R, G, cta, cc);
    stamp(t0 + 1);
    if (!sync()) return;
    stamp(t0 + 2);
    self_stage(A, S, w, G, cta, mw, lw);
    stamp(t0 + 3);
    if (!sync()) return;
    stamp(t0 + 4);
    prep_copy(S, A.att, d, R);
    cbar();
    gemm_stage<KSW>(A, S, d, d, VfEpi{VF_RESID, w.bo, nullptr, nullptr, nullptr}, R, G, cta, cc);
    ln_issue(S, w.ln2g, w.ln2b, d);
    stamp(t0 + 5);
    if (!sync()) return;
    stamp(t0 + 6);
    // cross-attention block
    prep_ln<KSW>(A, S, ln_n++, false, false, R, cta);
    cbar();
    gemm_stage<KSW>(A, S, d, d, VfEpi{VF_Q, w.bcq, l == A.anchor ? A.q_anchor : A.q, nullptr, nullptr}, R, G, cta,
                    cc);
    const int pf = cross_prefetch(A, S, &xmap, l, cta, an);
    an += (uint32_t)pf;
    stamp(t0 + 7);
    if (!sync()) return;
    stamp(t0 + 8);
    cross_stage(A, S, &xmap, l, G, cta, an, pf, mw, lw);
    stamp(t0 + 9);
    if (!sync()) return;
    stamp(t0 + 10);
    prep_copy(S, A.att, d, R);
    cbar();
    gemm_stage<KSW>(A, S, d, d, VfEpi{VF_RESID, w.bco, nullptr, nullptr, nullptr}, R, G, cta, cc);
    ln_issue(S, w.ln3g, w.ln3b, d);
    stamp(t0 + 11);
    if (!sync()) return;
    stamp(t0 + 12);
    // MLP block
    prep_ln<KSW>(A, S, ln_n++, false, false, R, cta);
    cbar();
    gemm_stage<KSW>(A, S, d, F, VfEpi{VF_GELU, w.b1, nullptr, nullptr, nullptr}, R, G, cta, cc);
    stamp(t0 + 13);
    if (!sync()) return;
    stamp(t0 + 14);
    prep_copy(S, A.hbuf, F, R);
    cbar();
    gemm_stage<KSW>(A, S, F, d, VfEpi{VF_RESID, w.b2, nullptr, nullptr, nullptr}, R, G, cta, cc);
    if (l + 1 < A.L) ln_issue(S, S.layers[l + 1].ln1g, S.layers[l + 1].ln1b, d);
    else ln_issue(S, A.lnf_g, A.lnf_b, d);
    stamp(t0 + 15);
    if (!sync()) return;
  }
  tl_mark(A.tl, TL_MID);
  stamp(16 * A.L);
  // final LayerNorm, LM head with argmax (no logits stored)
  prep_ln<KSW>(A, S, ln_n++, false, true, R, cta);
  cbar();
  gemm_stage<KSW>(A, S, d, A.V, VfEpi{VF_ARGMAX, nullptr, nullptr, nullptr, nullptr}, R, G, cta, cc);
  if (tid < R && rkey[tid] != 0ull) atomicMax(A.row_key + tid, rkey[tid]);
  stamp(16 * A.L + 1);
  tl_mark(A.tl, TL_EXIT);
}

template <int KSW>
void* vf_kernel() {
  return reinterpret_cast<void*>(&verify_fused_kernel<KSW>);
}

void* vf_pick(int d) {
  switch (d) {
    case 512: return vf_kernel<4>();
    case 768: return vf_kernel<6>();
    case 1024: return vf_kernel<8>();
    case 1280: return vf_kernel<10>();
    default: return nullptr;
  }
}

}  // namespace

void vf_layout(int d, int F, int L, int* a_bytes, int* slot_bytes, int* total) {
  const int act = VF_ROWS * (2 * std::max(d, F) + 16);
  const int att = 2 * 2 * VF_TILE;   // two chunks of K and V; also the 8 warps' [16][64] fp32 partials
  int a = std::max(act, att);
  a = (a + 1023) & ~1023;
  const int slot = 8 * (2 * d + 16);
  *a_bytes = a;
  *slot_bytes = slot;
  *total = 1024 + a + VF_NSLOT * slot + VF_RED + L * (int)sizeof(VfLayer) + 7 * VF_ROWS * 4;
}

int vf_grid(int d, int F, int L) {
  void* k = vf_pick(d);
  if (k == nullptr || F % d != 0) return 0;
  int a, s, total;
  vf_layout(d, F, L, &a, &s, &total);
  int dev = 0, n_sm = 0, coop = 0, max_smem = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 0;
  cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
  cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
  cudaDeviceGetAttribute(&max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev);
  if (!coop || total + 2048 > max_smem) return 0;
  if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, total) != cudaSuccess) return 0;
  int per_sm = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, VF_THREADS, total) != cudaSuccess || per_sm < 1)
    return 0;
  return n_sm;
}

cudaError_t launch_verify_fused(const CUtensorMap* xmap, const VfArgs& a, int grid, cudaStream_t st) {
  void* k = vf_pick(a.d);
  if (k == nullptr) return cudaErrorInvalidValue;
  int ab, sb, total;
  vf_layout(a.d, a.F, a.L, &ab, &sb, &total);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(VF_THREADS);
  cfg.dynamicSmemBytes = total;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {const_cast<CUtensorMap*>(xmap), const_cast<VfArgs*>(&a)};
  return cudaLaunchKernelExC(&cfg, k, args);
}

}  // namespace asrspec
