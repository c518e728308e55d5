// Host side of the many-row projection GEMM (gemm_wide.cuh): tile choice,
// instantiations, launch.
#include <mutex>

#include "gemm_wide.cuh"

namespace asrspec {

ASRSPEC_CHECK_SETTER(set_check_gemm_wide)

namespace {

template <int BN, int MODE, int SPLIT>
void launch_w(const WideGemm& g, const Epi& epi, int* status, cudaStream_t st) {
  using C = WideCfg<BN, MODE>;
  static std::once_flag once;
  std::call_once(once, [] {
    cudaFuncSetAttribute(gemm_wide_kernel<BN, MODE, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  });
  const dim3 grid((unsigned)(g.M / 128 * SPLIT), (unsigned)((g.N + BN - 1) / BN));
  constexpr int S_MAX = C::STAGES / WG_PIPES;   // stages per pipeline
  const int S = g.stages >= 1 && g.stages < S_MAX ? g.stages : S_MAX;
  launch_ex(gemm_wide_kernel<BN, MODE, SPLIT>, grid, dim3(WG_THREADS), (size_t)C::smem_bytes(S), st, g.pdl, SPLIT,
            g.mapA, g.mapB, g.mapX, g.K, S, epi, status);
}

template <int MODE, int SPLIT>
void launch_bn(const WideGemm& g, const Epi& epi, int* status, cudaStream_t st) {
  switch (g.bn) {
    case 32: launch_w<32, MODE, SPLIT>(g, epi, status, st); break;
    case 64: launch_w<64, MODE, SPLIT>(g, epi, status, st); break;
    case 96: launch_w<96, MODE, SPLIT>(g, epi, status, st); break;
    default:
      if constexpr (MODE != EPI_RESID) launch_w<128, MODE, SPLIT>(g, epi, status, st);
      break;
  }
}

template <int MODE>
void launch_bn_wide(const WideGemm& g, const Epi& epi, int* status, cudaStream_t st) {
  switch (g.bn) {
    case 160: launch_w<160, MODE, 1>(g, epi, status, st); break;
    default: launch_bn<MODE, 1>(g, epi, status, st); break;
  }
}

}  // namespace

// N tiles: as many as the SMs left per M tile allow (a tile per SM), rounded
// up to a tile width of the set; long K (>= 48 k-blocks) split over a pair.
bool wide_pick(int M, int N, int K, int mode, int sms, int* bn, int* split) {
  if (M % 128 || K % 64 || N < 1 || sms < 1) return false;
  if (mode != EPI_QKV && mode != EPI_Q && mode != EPI_GELU && mode != EPI_RESID) return false;
  const int mt = M / 128, nkb = K / 64;
  *split = (mode == EPI_RESID && nkb >= 48) ? 2 : 1;
  const int slots = sms / *split;
  const int nt = std::max(1, slots / mt);
  const int want = (N + nt - 1) / nt;
  // tile widths whose accumulators fit tensor memory; a residual tile also
  // keeps its residual tile in shared memory beside a ring of 2 stages per pipeline
  const int cap = mode == EPI_RESID ? 96 : 160;
  static const int set[5] = {32, 64, 96, 128, 160};
  *bn = cap;
  for (int c : set)
    if (c >= want && c <= cap) {
      *bn = c;
      break;
    }
  return true;
}

void launch_gemm_wide(const WideGemm& g, int mode, const Epi& epi, int* status, cudaStream_t st) {
  switch (mode) {
    case EPI_QKV: launch_bn_wide<EPI_QKV>(g, epi, status, st); break;
    case EPI_Q: launch_bn_wide<EPI_Q>(g, epi, status, st); break;
    case EPI_GELU: launch_bn_wide<EPI_GELU>(g, epi, status, st); break;
    case EPI_RESID:
      if (g.split > 1) launch_bn<EPI_RESID, 2>(g, epi, status, st);
      else launch_bn<EPI_RESID, 1>(g, epi, status, st);
      break;
    default: break;
  }
}

}  // namespace asrspec
