// Warp-level building blocks of the few-row kernels: ldmatrix / mma.sync
// wrappers, bf16 packing, the 128-byte swizzle of TMA tiles, and a
// flash-attention step over one 128-key chunk for up to 16 query rows of one
// head (rows as the MMA's M side; running max, sum and output per warp).
#pragma once

#include "common.cuh"

namespace asrspec {

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
__device__ __forceinline__ void sts32(uint32_t addr, uint32_t v) {
  asm volatile("st.shared.b32 [%0], %1;" ::"r"(addr), "r"(v) : "memory");
}
// D (16 x 8 fp32) += A (16 x 16 bf16, row-major) x B (16 x 8 bf16, column-major)
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
__device__ __forceinline__ float2 bits_bf2(uint32_t u) {
  __nv_bfloat162 v = *reinterpret_cast<__nv_bfloat162*>(&u);
  return __bfloat1622float2(v);
}
// byte offset of (row, 16-byte piece) in a 128-byte-swizzled tile of 128-byte rows
__device__ __forceinline__ uint32_t sw128(int row, int c16) { return (uint32_t)(row * 128 + ((c16 ^ (row & 7)) << 4)); }

// 4-byte asynchronous store into another CTA's shared memory, counted on its mbarrier
__device__ __forceinline__ void st_async_b32(uint32_t addr, uint32_t v, uint32_t remote_bar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(addr), "r"(v),
               "r"(remote_bar)
               : "memory");
}
// Fire-and-forget prefetch of global memory into L2 (16-byte aligned, bytes % 16 == 0).
__device__ __forceinline__ void l2_prefetch(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(reinterpret_cast<uint64_t>(p)), "r"(bytes)
               : "memory");
}

// Running (max, sum, output) of one warp's keys for up to 16 query rows of one head.
struct AttnState {
  uint32_t qa[4][4];
  int lim[2];
  float m_run[2], l_run[2], O[8][4];
};

// q: [rows][32] bf16 pairs of q / 8 (shared memory, row stride 32 words);
// rows >= nr are zero.  lim: the keys row r sees, min(n_keys, pos_r + 1) when
// causal (pos_r = row_pos[r]), else n_keys.
__device__ __forceinline__ void attn_init(AttnState& st, const uint32_t* q, int nr, const int* row_pos, int n_keys,
                                          bool causal) {
  const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
  for (int kk = 0; kk < 4; ++kk)
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int pr = kk * 8 + half * 4 + t;
      st.qa[kk][half * 2 + 0] = g < nr ? q[g * 32 + pr] : 0u;
      st.qa[kk][half * 2 + 1] = g + 8 < nr ? q[(g + 8) * 32 + pr] : 0u;
    }
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int r = g + 8 * e;
    st.lim[e] = (causal && r < nr) ? min(n_keys, row_pos[r] + 1) : n_keys;
    st.m_run[e] = -INFINITY;
    st.l_run[e] = 0.f;
  }
#pragma unroll
  for (int nd = 0; nd < 8; ++nd) st.O[nd][0] = st.O[nd][1] = st.O[nd][2] = st.O[nd][3] = 0.f;
}

// One 128-key chunk (K at ks, V at vs: shared addresses of 128-byte-swizzled
// tiles); warp w takes keys [16 w, 16 w + 16) of it; key0 = the chunk's first key.
// Probabilities are rounded to bf16 for the P.V product; accumulation in fp32.
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

// Combine the 8 warps' states for rows < nr (<= 9) into out[r][66] = (max,
// sum, output[64]) of the rows (fixed warp order).  scratch: [8][9][64] fp32
// plus [2][8][16]; every thread of the CTA's 8 warps calls it.
__device__ __forceinline__ void attn_combine(const AttnState& st, int nr, float* scratch, float* out) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
  float* Ow = scratch;                 // [8][9][64]
  float* mw = scratch + 8 * 9 * 64;    // [8][16]
  float* lw = mw + 8 * 16;
#pragma unroll
  for (int e = 0; e < 2; ++e) {
    const int r = g + 8 * e;
    if (r < nr) {
      if (t == 0) {
        mw[warp * 16 + r] = st.m_run[e];
        lw[warp * 16 + r] = st.l_run[e];
      }
#pragma unroll
      for (int nd = 0; nd < 8; ++nd)
        *reinterpret_cast<float2*>(Ow + (warp * 9 + r) * 64 + nd * 8 + 2 * t) =
            make_float2(st.O[nd][2 * e], st.O[nd][2 * e + 1]);
    }
  }
  __syncthreads();
  for (int e = threadIdx.x; e < nr * 64; e += blockDim.x) {
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
      o += Ow[(w * 9 + r) * 64 + c] * f;
    }
    out[r * 66 + 2 + c] = o;
    if (c == 0) {
      out[r * 66 + 0] = M;
      out[r * 66 + 1] = L;
    }
  }
  __syncthreads();
}

}  // namespace asrspec
