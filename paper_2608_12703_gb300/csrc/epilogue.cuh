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
  // B operand = LayerNorm(ln_x) (few-row GEMMs): fp32 rows [N][K], gain and bias [K]
  const float* ln_x = nullptr;
  const float* ln_g = nullptr;
  const float* ln_b = nullptr;
  // optional phase timestamps (ns, %globaltimer) per CTA: [CTA][8]
  // (entry, set-up done, first stage full, MMAs done, end; cluster split:
  // partials staged, first cluster barrier passed, reduction done)
  unsigned long long* trace = nullptr;
};

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
      size_t idx = (((size_t)e.row_b[n] * e.n_heads + h) * e.max_pos + e.row_pos[n]) * 64 + c;
      void* base = which == 0 ? e.kcache : e.vcache;
      if (e.kv_bf16) store_as<__nv_bfloat16>(base, idx, v);
      else store_as<float>(base, idx, v);
    }
  } else if constexpr (MODE == EPI_CROSSKV) {
    int b = m / e.t_max, t = m - b * e.t_max;
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

// U output elements at once.  The residual update loads every x value before
// it stores any (the elements are distinct, so no store can feed a later
// load), which keeps U loads in flight instead of U dependent round trips.
template <int MODE, int U>
__device__ __forceinline__ void epi_batch(const Epi& e, const int* m, const int* n, const float* v,
                                          const bool* ok) {
  if constexpr (MODE == EPI_RESID) {
    float old[U], bias[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      old[u] = ok[u] ? e.x[(size_t)n[u] * e.d + m[u]] : 0.f;
      bias[u] = ok[u] ? e.bias[m[u]] : 0.f;
    }
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (ok[u]) e.x[(size_t)n[u] * e.d + m[u]] = old[u] + (v[u] + bias[u]);
  } else if constexpr (MODE == EPI_QKV) {
    // row metadata and biases first, then the stores
    float bias[U];
    int rb[U], rp[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      bias[u] = ok[u] ? e.bias[m[u]] : 0.f;
      rb[u] = ok[u] && m[u] >= e.d ? e.row_b[n[u]] : 0;
      rp[u] = ok[u] && m[u] >= e.d ? e.row_pos[n[u]] : 0;
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const float val = v[u] + bias[u];
      if (m[u] < e.d) {
        e.out_f32[(size_t)n[u] * e.d + m[u]] = val;
      } else {
        const int which = (m[u] - e.d) / e.d;
        const int f = (m[u] - e.d) - which * e.d;
        const size_t idx = (((size_t)rb[u] * e.n_heads + (f >> 6)) * e.max_pos + rp[u]) * 64 + (f & 63);
        void* base = which == 0 ? e.kcache : e.vcache;
        if (e.kv_bf16) store_as<__nv_bfloat16>(base, idx, val);
        else store_as<float>(base, idx, val);
      }
    }
  } else if constexpr (MODE == EPI_Q) {
    float bias[U];
#pragma unroll
    for (int u = 0; u < U; ++u) bias[u] = ok[u] ? e.bias[m[u]] : 0.f;
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (ok[u]) e.out_f32[(size_t)n[u] * e.d + m[u]] = v[u] + bias[u];
  } else if constexpr (MODE == EPI_GELU) {
    float bias[U];
#pragma unroll
    for (int u = 0; u < U; ++u) bias[u] = ok[u] ? e.bias[m[u]] : 0.f;
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (!ok[u]) continue;
      const float g = gelu_erf(v[u] + bias[u]);
      const size_t idx = (size_t)n[u] * e.M + m[u];
      if (e.act_bf16) store_as<__nv_bfloat16>(e.act, idx, g);
      else store_as<float>(e.act, idx, g);
    }
  } else {
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (ok[u]) epi_apply<MODE>(e, m[u], n[u], v[u]);
  }
}

}  // namespace asrspec
