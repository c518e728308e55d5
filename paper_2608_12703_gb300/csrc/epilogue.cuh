// GEMM epilogues of the verify step.
//
// Every projection of the decoder (Sec. 3 "Models and Protocol": the
// Whisper-style target decoder) is one GEMM C[m][n] = sum_k A[m][k] B[n][k].
// Over the verify rows the weights are the A operand (m = output feature) and
// the rows are the B operand (n = row), so that the many weight rows fill the
// 128-lane MMA side and the few verify rows the narrow N side.  The epilogue
// adds the bias and routes each value to where the next step reads it.
#pragma once

#include "common.cuh"

namespace asrspec {

enum EpiMode : int {
  EPI_F32 = 0,       // out_f32[n * ld + m] = acc                                  (tests, debug logits)
  EPI_QKV = 1,       // q -> q_out[n][m]; k, v -> self cache at (row_b[n], head, row_pos[n])
  EPI_RESID = 2,     // x[n][m] += acc + bias[m]                                   (residual, fp32)
  EPI_Q = 3,         // q_out[n][m] = acc + bias[m]                                (cross-attention query)
  EPI_GELU = 4,      // act[n][m] = gelu(acc + bias[m])                            (MLP hidden, storage type)
  EPI_CROSSKV = 5,   // m = frame (b, t), n = (layer, k|v, head, c) -> cross cache (encode_cache)
  EPI_ARGMAX = 6,    // m = vocab id, n = row: per-row argmax key, atomicMax        (LM head)
  EPI_F32_MN = 7,    // out_f32[m * ld + n] = acc                                  (tests)
};

struct Epi {
  const float* bias = nullptr;
  const int* n_valid = nullptr;   // device count of valid n (verify rows); null = all
  int M = 0, N = 0;
  int d = 0;                      // d_model
  int ld = 0;                     // leading dimension of the plain outputs
  float* out_f32 = nullptr;       // EPI_F32 / EPI_Q / EPI_QKV (q part)
  float* x = nullptr;             // EPI_RESID
  void* act = nullptr;            // EPI_GELU (bf16 or fp32 by `act_bf16`)
  int act_bf16 = 0;
  // self-attention cache append (EPI_QKV): cache layout [B_max][H][max_pos][64]
  const int* row_b = nullptr;
  const int* row_pos = nullptr;
  void* kcache = nullptr;
  void* vcache = nullptr;
  int kv_bf16 = 0;
  int max_pos = 0;
  int n_heads = 0;
  // cross cache (EPI_CROSSKV): layout [L][2][B_max][H][max_enc][64]
  const int* enc_len = nullptr;
  int t_max = 0;
  int max_enc = 0;
  int b_max = 0;
  // LM head argmax
  unsigned long long* row_key = nullptr;
  // device status word, for the bounds-check mode (ST_BOUNDS), or null
  int* status = nullptr;
  // LayerNorm folded into the GEMM (consumer).  The B operand is bf16(g * x)
  // and y = rstd_n (acc - mu_n c1_m) + c2_m (+ bias), with c1 = W g, c2 = W b
  // and the row statistics combined from ln_S slices of ln_c features each:
  // ln_part[s * ln_stride + n] = (slice mean, slice sum of squared deviations).
  const float2* ln_part = nullptr;
  int ln_S = 0, ln_c = 0, ln_stride = 0;
  const float* ln_c1 = nullptr;
  const float* ln_c2 = nullptr;
  // Producer of the next folded LayerNorm (EPI_RESID): writes xg = bf16(g * x)
  // [n][d] and its slice statistics st_part[slice * st_stride + n].
  __nv_bfloat16* xg = nullptr;
  const float* xg_gain = nullptr;
  float2* st_part = nullptr;
  int st_stride = 0;
  // launch timeline slot (see tl_mark), or null
  unsigned long long* tl = nullptr;
  // > 0: one-dimensional grid walked in bands of group_m M tiles, each band
  // sweeping every N tile (L2 reuse when both operands exceed the L2)
  int group_m = 0;
  // optional phase timestamps (ns, %globaltimer) per CTA: [CTA][FR_TRACE_PHASES]
  // for the first FR_TRACE_CTAS CTAs (0 entry, 1 set-up done, 2 first stage
  // full, 3 MMAs done, 4 end; cluster split: 5 partials staged, 6 exchange
  // landed, 7 reduction done)
  unsigned long long* trace = nullptr;
};

// Bounds-check mode: a self-cache slot (utterance rb, position rp) outside the cache.
__device__ __forceinline__ bool qkv_slot_bad(const Epi& e, int rb, int rp) {
  return bounds_bad(e.status, rp < 0 || rp >= e.max_pos || rb < 0 || (e.b_max > 0 && rb >= e.b_max));
}

template <typename T>
__device__ __forceinline__ void store_as(void* base, size_t idx, float v) {
  reinterpret_cast<T*>(base)[idx] = from_f<T>(v);
}

// One output element (all modes but EPI_ARGMAX).  Caller guarantees m < M and n < n_valid.
template <int MODE>
__device__ __forceinline__ void epi_apply(const Epi& e, int m, int n, float acc) {
  if constexpr (MODE == EPI_F32) {
    e.out_f32[(size_t)n * e.ld + m] = acc;
  } else if constexpr (MODE == EPI_F32_MN) {
    e.out_f32[(size_t)m * e.ld + n] = acc;
  } else if constexpr (MODE == EPI_RESID) {
    float* p = e.x + (size_t)n * e.d + m;
    *p = *p + (acc + e.bias[m]);
  } else if constexpr (MODE == EPI_Q) {
    e.out_f32[(size_t)n * e.d + m] = acc + e.bias[m];
  } else if constexpr (MODE == EPI_GELU) {
    float v = gelu_erf(acc + e.bias[m]);
    size_t idx = (size_t)n * e.M + m;
    if (e.act_bf16) store_as<__nv_bfloat16>(e.act, idx, v);
    else store_as<float>(e.act, idx, v);
  } else if constexpr (MODE == EPI_QKV) {
    float v = acc + e.bias[m];
    if (m < e.d) {
      e.out_f32[(size_t)n * e.d + m] = v;
    } else {
      int which = (m - e.d) / e.d;            // 0 = k, 1 = v
      int f = (m - e.d) - which * e.d;
      int h = f >> 6, c = f & 63;
      if (qkv_slot_bad(e, e.row_b[n], e.row_pos[n])) return;
      size_t idx = (((size_t)e.row_b[n] * e.n_heads + h) * e.max_pos + e.row_pos[n]) * 64 + c;
      void* base = which == 0 ? e.kcache : e.vcache;
      if (e.kv_bf16) store_as<__nv_bfloat16>(base, idx, v);
      else store_as<float>(base, idx, v);
    }
  } else if constexpr (MODE == EPI_CROSSKV) {
    int b = m / e.t_max, t = m - b * e.t_max;
    if (bounds_bad(e.status, b >= e.b_max || t >= e.max_enc)) return;
    if (t >= e.enc_len[b]) return;
    int two_d = 2 * e.d;
    int l = n / two_d;
    int r = n - l * two_d;
    int which = r / e.d;
    int f = r - which * e.d;
    int h = f >> 6, c = f & 63;
    size_t idx = (((((size_t)l * 2 + which) * e.b_max + b) * e.n_heads + h) * e.max_enc + t) * 64 + c;
    float v = acc + e.bias[n];
    if (e.kv_bf16) store_as<__nv_bfloat16>(e.kcache, idx, v);
    else store_as<float>(e.kcache, idx, v);
  }
}

// U output elements at once, in two halves so that a caller can issue the
// loads early (before the accumulators are ready) and keep them in registers:
// epi_load fetches what the outputs depend on besides the accumulators (bias,
// residual, row metadata), epi_store combines and writes.  The elements are
// distinct, so no store can feed a later load.
template <int MODE, int U>
struct EpiPre {
  float bias[U];
  float old[U];   // EPI_RESID: x before the update
  int rb[U], rp[U];   // EPI_QKV: utterance and position of the row
  bool bad[U];        // EPI_QKV: the slot failed the bounds-check mode
  float c1[U], c2[U];   // folded LayerNorm (consumer)
  float gain[U];        // next LayerNorm's gain (EPI_RESID producer)
};

template <int MODE, int U>
__device__ __forceinline__ void epi_load(const Epi& e, const int* m, const int* n, const bool* ok,
                                         EpiPre<MODE, U>& p) {
#pragma unroll
  for (int u = 0; u < U; ++u) {
    if constexpr (MODE == EPI_RESID || MODE == EPI_QKV || MODE == EPI_Q || MODE == EPI_GELU)
      p.bias[u] = ok[u] ? __ldg(e.bias + m[u]) : 0.f;
    if constexpr (MODE == EPI_RESID) p.old[u] = ok[u] ? e.x[(size_t)n[u] * e.d + m[u]] : 0.f;
    if constexpr (MODE == EPI_QKV) {
      p.rb[u] = ok[u] && m[u] >= e.d ? e.row_b[n[u]] : 0;
      p.rp[u] = ok[u] && m[u] >= e.d ? e.row_pos[n[u]] : 0;
      p.bad[u] = ok[u] && m[u] >= e.d && qkv_slot_bad(e, p.rb[u], p.rp[u]);
    }
    if constexpr (MODE != EPI_RESID && MODE != EPI_CROSSKV) {
      p.c1[u] = ok[u] && e.ln_part ? __ldg(e.ln_c1 + m[u]) : 0.f;
      p.c2[u] = ok[u] && e.ln_part ? __ldg(e.ln_c2 + m[u]) : 0.f;
    }
    if constexpr (MODE == EPI_RESID) p.gain[u] = ok[u] && e.xg ? __ldg(e.xg_gain + m[u]) : 0.f;
  }
}

template <int MODE, int U>
__device__ __forceinline__ void epi_store(const Epi& e, const int* m, const int* n, const float* v, const bool* ok,
                                          const EpiPre<MODE, U>& p) {
#pragma unroll
  for (int u = 0; u < U; ++u) {
    if (!ok[u]) continue;
    if constexpr (MODE == EPI_RESID) {
      e.x[(size_t)n[u] * e.d + m[u]] = p.old[u] + (v[u] + p.bias[u]);
    } else if constexpr (MODE == EPI_QKV) {
      const float val = v[u] + p.bias[u];
      if (m[u] < e.d) {
        e.out_f32[(size_t)n[u] * e.d + m[u]] = val;
      } else if (!p.bad[u]) {
        const int which = (m[u] - e.d) / e.d;
        const int f = (m[u] - e.d) - which * e.d;
        const size_t idx = (((size_t)p.rb[u] * e.n_heads + (f >> 6)) * e.max_pos + p.rp[u]) * 64 + (f & 63);
        void* base = which == 0 ? e.kcache : e.vcache;
        if (e.kv_bf16) store_as<__nv_bfloat16>(base, idx, val);
        else store_as<float>(base, idx, val);
      }
    } else if constexpr (MODE == EPI_Q) {
      e.out_f32[(size_t)n[u] * e.d + m[u]] = v[u] + p.bias[u];
    } else if constexpr (MODE == EPI_GELU) {
      const float g = gelu_erf(v[u] + p.bias[u]);
      const size_t idx = (size_t)n[u] * e.M + m[u];
      if (e.act_bf16) store_as<__nv_bfloat16>(e.act, idx, g);
      else store_as<float>(e.act, idx, g);
    } else {
      epi_apply<MODE>(e, m[u], n[u], v[u]);
    }
  }
}

template <int MODE, int U>
__device__ __forceinline__ void epi_batch(const Epi& e, const int* m, const int* n, const float* v,
                                          const bool* ok) {
  EpiPre<MODE, U> p;
  epi_load<MODE, U>(e, m, n, ok, p);
  epi_store<MODE, U>(e, m, n, v, ok, p);
}

// Row-wise epilogue over a tile staged in shared memory as stg[n_local][m_local]
// (leading dimension lds): lane l of warp w covers features m = mq .. mq + 3
// (mq = tile m0 + 4 l) of rows n_local = w, w + 4, ...  Each row is written
// with one 16-byte (fp32) or 8-byte (bf16) store per lane, so a warp writes
// whole 512- or 256-byte runs; bias and the feature's role are per lane, the
// row metadata per row.  Modes: F32 (any M), Q, RESID, GELU, QKV (M, d, and
// the leading dimensions multiples of 4).
template <int MODE>
__host__ __device__ constexpr bool rowwise_mode() {
  return MODE == EPI_F32 || MODE == EPI_Q || MODE == EPI_RESID || MODE == EPI_GELU || MODE == EPI_QKV;
}

// ln_mu / ln_rs: the folded LayerNorm's row statistics of the tile's rows
// (shared memory, indexed by local row), used when e.ln_part is set.  A
// residual producer (e.xg set) also writes bf16(g * x) and the statistics of
// the warp's 128 features (slice m0 / 128) of each row.
template <int MODE>
__device__ __forceinline__ void epi_rows(const Epi& e, const float* stg, int lds, int mq, int m_local, int n0,
                                         int warp, int rows, const float* ln_mu, const float* ln_rs) {
  const bool mok = mq < e.M;
  float4 bias = make_float4(0.f, 0.f, 0.f, 0.f);
  if constexpr (MODE != EPI_F32)
    if (mok) bias = __ldg(reinterpret_cast<const float4*>(e.bias + mq));
  const bool fold = e.ln_part != nullptr && MODE != EPI_RESID;
  float4 c1 = make_float4(0.f, 0.f, 0.f, 0.f), c2 = c1, gain = c1;
  if (fold && mok) {
    c1 = __ldg(reinterpret_cast<const float4*>(e.ln_c1 + mq));
    c2 = __ldg(reinterpret_cast<const float4*>(e.ln_c2 + mq));
  }
  if constexpr (MODE == EPI_RESID)
    if (e.xg && mok) gain = __ldg(reinterpret_cast<const float4*>(e.xg_gain + mq));
  int kind = 0, head = 0, c = 0;   // EPI_QKV: 0 query, 1 key, 2 value
  if constexpr (MODE == EPI_QKV) {
    if (mq >= e.d) {
      const int f = mq - e.d;
      kind = f >= e.d ? 2 : 1;
      const int g = f - (kind - 1) * e.d;
      head = g >> 6;
      c = g & 63;
    }
  }
  constexpr int RB = 4;   // rows per batch, their loads in flight together
  for (int j0 = warp; j0 < rows; j0 += 4 * RB) {
    float4 a[RB], old[RB];
    int rb[RB], rp[RB];
    bool ok[RB];
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      const int nl = j0 + 4 * r;
      ok[r] = nl < rows && mok;
      const int n = n0 + (nl < rows ? nl : 0);
      a[r] = ok[r] ? *reinterpret_cast<const float4*>(stg + nl * lds + m_local) : make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (MODE == EPI_RESID)
        old[r] = ok[r] ? *reinterpret_cast<const float4*>(e.x + (size_t)n * e.d + mq) : make_float4(0.f, 0.f, 0.f, 0.f);
      if constexpr (MODE == EPI_QKV) {
        rb[r] = ok[r] && kind ? e.row_b[n] : 0;
        rp[r] = ok[r] && kind ? e.row_pos[n] : 0;
        if (ok[r] && kind && qkv_slot_bad(e, rb[r], rp[r])) ok[r] = false;
      }
    }
#pragma unroll
    for (int r = 0; r < RB; ++r) {
      if (!ok[r]) continue;
      const int n = n0 + j0 + 4 * r;
      float4 v = a[r];
      if (fold) {   // y = rstd (acc - mu c1) + c2
        const float mu = ln_mu[j0 + 4 * r], rs = ln_rs[j0 + 4 * r];
        v = make_float4(rs * (v.x - mu * c1.x) + c2.x, rs * (v.y - mu * c1.y) + c2.y, rs * (v.z - mu * c1.z) + c2.z,
                        rs * (v.w - mu * c1.w) + c2.w);
      }
      if constexpr (MODE == EPI_F32) {
        float* o = e.out_f32 + (size_t)n * e.ld;
        if (mq + 0 < e.M) o[mq + 0] = v.x;
        if (mq + 1 < e.M) o[mq + 1] = v.y;
        if (mq + 2 < e.M) o[mq + 2] = v.z;
        if (mq + 3 < e.M) o[mq + 3] = v.w;
        continue;
      }
      v.x += bias.x; v.y += bias.y; v.z += bias.z; v.w += bias.w;
      if constexpr (MODE == EPI_Q) {
        *reinterpret_cast<float4*>(e.out_f32 + (size_t)n * e.d + mq) = v;
      } else if constexpr (MODE == EPI_RESID) {
        const float4 o = old[r];
        const float4 xn = make_float4(o.x + v.x, o.y + v.y, o.z + v.z, o.w + v.w);
        *reinterpret_cast<float4*>(e.x + (size_t)n * e.d + mq) = xn;
        if (e.xg) {   // the next LayerNorm's operand and this slice's statistics (uniform over the warp)
          __nv_bfloat162 lo = __floats2bfloat162_rn(gain.x * xn.x, gain.y * xn.y);
          __nv_bfloat162 hi = __floats2bfloat162_rn(gain.z * xn.z, gain.w * xn.w);
          *reinterpret_cast<uint2*>(e.xg + (size_t)n * e.d + mq) =
              make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
          const float mean = warp_sum((xn.x + xn.y) + (xn.z + xn.w)) * (1.f / 128.f);
          const float dx = xn.x - mean, dy = xn.y - mean, dz = xn.z - mean, dw = xn.w - mean;
          const float m2 = warp_sum((dx * dx + dy * dy) + (dz * dz + dw * dw));
          if ((threadIdx.x & 31) == 0) e.st_part[(size_t)(mq / 128) * e.st_stride + n] = make_float2(mean, m2);
        }
      } else if constexpr (MODE == EPI_GELU) {
        v = make_float4(gelu_erf(v.x), gelu_erf(v.y), gelu_erf(v.z), gelu_erf(v.w));
        const size_t idx = (size_t)n * e.M + mq;
        if (e.act_bf16) {
          __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
          *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(e.act) + idx) =
              make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
        } else {
          *reinterpret_cast<float4*>(static_cast<float*>(e.act) + idx) = v;
        }
      } else if constexpr (MODE == EPI_QKV) {
        if (kind == 0) {
          *reinterpret_cast<float4*>(e.out_f32 + (size_t)n * e.d + mq) = v;
        } else {
          const size_t idx = (((size_t)rb[r] * e.n_heads + head) * e.max_pos + rp[r]) * 64 + c;
          void* base = kind == 1 ? e.kcache : e.vcache;
          if (e.kv_bf16) {
            __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
            *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(base) + idx) =
                make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
          } else {
            *reinterpret_cast<float4*>(static_cast<float*>(base) + idx) = v;
          }
        }
      }
    }
  }
}

}  // namespace asrspec
