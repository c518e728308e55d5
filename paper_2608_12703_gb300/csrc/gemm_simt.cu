// SIMT GEMM with the same epilogues as the tensor-core path.
//
// Used for fp32 models (no TF32 anywhere: every product and sum in fp32 FFMA)
// and as an independent cross-check of the tcgen05 GEMM in the kernel tests.
// C[m][n] = sum_k A[m][k] B[n][k]; 64 x 64 tiles, 16-deep k slices staged in
// shared memory, 4 x 4 outputs per thread.
#include "kernels.h"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_gemm_simt)

constexpr int SG_BM = 64, SG_BN = 64, SG_BK = 16;

template <typename TA, typename TB, int MODE>
__global__ void __launch_bounds__(256)
gemm_simt_kernel(const TA* __restrict__ A, const TB* __restrict__ B, int M, int N, int K, Epi epi) {
  __shared__ float As[SG_BK][SG_BM + 4];
  __shared__ float Bs[SG_BK][SG_BN + 4];
  const int n_valid = epi.n_valid ? min(*epi.n_valid, N) : N;
  const int m0 = blockIdx.x * SG_BM, n0 = blockIdx.y * SG_BN;
  if (n0 >= n_valid) return;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += SG_BK) {
    // 64 x 16 elements of each operand; 256 threads x 4 elements
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const int idx = tid + e * 256;
      const int r = idx >> 4, c = idx & 15;
      const int gm = m0 + r, gn = n0 + r, gk = k0 + c;
      As[c][r] = (gm < M && gk < K) ? to_f<TA>(A[(size_t)gm * K + gk]) : 0.f;
      Bs[c][r] = (gn < n_valid && gk < K) ? to_f<TB>(B[(size_t)gn * K + gk]) : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < SG_BK; ++kk) {
      float a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][tx + 16 * i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][ty + 16 * j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  if constexpr (MODE == EPI_ARGMAX) {
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int n = n0 + ty + 16 * j;
      unsigned long long key = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int m = m0 + tx + 16 * i;
        if (m < M) {
          unsigned long long kk = argmax_key(acc[i][j], (uint32_t)m);
          key = kk > key ? kk : key;
        }
      }
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) {
        unsigned long long w = __shfl_xor_sync(0xffffffffu, key, o);
        key = w > key ? w : key;
      }
      if (tx == 0 && n < n_valid) atomicMax(epi.row_key + n, key);
    }
  } else {
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int m = m0 + tx + 16 * i, n = n0 + ty + 16 * j;
        if (m < M && n < n_valid) epi_apply<MODE>(epi, m, n, acc[i][j]);
      }
  }
}

template <typename TA, typename TB, int MODE>
static void launch_t(const void* A, const void* B, int M, int N, int K, const Epi& epi, cudaStream_t st) {
  dim3 grid((M + SG_BM - 1) / SG_BM, (N + SG_BN - 1) / SG_BN);
  gemm_simt_kernel<TA, TB, MODE><<<grid, 256, 0, st>>>(static_cast<const TA*>(A), static_cast<const TB*>(B), M, N,
                                                       K, epi);
}

template <int MODE>
static void launch_mode(const void* A, int a_bf16, const void* B, int b_bf16, int M, int N, int K, const Epi& epi,
                        cudaStream_t st) {
  using bf = __nv_bfloat16;
  if (a_bf16 && b_bf16) launch_t<bf, bf, MODE>(A, B, M, N, K, epi, st);
  else if (a_bf16) launch_t<bf, float, MODE>(A, B, M, N, K, epi, st);
  else if (b_bf16) launch_t<float, bf, MODE>(A, B, M, N, K, epi, st);
  else launch_t<float, float, MODE>(A, B, M, N, K, epi, st);
}

void launch_gemm_simt(const void* A, int a_bf16, const void* B, int b_bf16, int M, int N, int K, int mode,
                      const Epi& epi, cudaStream_t st) {
  switch (mode) {
    case EPI_F32: launch_mode<EPI_F32>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_F32_MN: launch_mode<EPI_F32_MN>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_QKV: launch_mode<EPI_QKV>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_RESID: launch_mode<EPI_RESID>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_Q: launch_mode<EPI_Q>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_GELU: launch_mode<EPI_GELU>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_CROSSKV: launch_mode<EPI_CROSSKV>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
    case EPI_ARGMAX: launch_mode<EPI_ARGMAX>(A, a_bf16, B, b_bf16, M, N, K, epi, st); break;
  }
}

}  // namespace asrspec
