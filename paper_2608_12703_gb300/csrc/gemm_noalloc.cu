// A split-K tensor-core GEMM entry point that performs no device allocation.
//
// Some callers cannot let a library call cudaMalloc or cudaFree: a host
// framework that owns every byte of device memory through its own pool (an
// allocation behind its back breaks its accounting and fragments the pool), a
// serving loop that forbids allocation after start-up because cudaMalloc and
// cudaFree can synchronise the device and stall every stream, or code that
// runs while another thread is capturing a CUDA graph in a mode in which such
// calls are rejected.  For them, this entry point keeps its split-K scratch
// (partial sums, per-tile tickets and a status word) in one file-scope device
// array of fixed size instead of allocating it per call.
//
// The array exists once per GPU that loads the library and stays allocated
// until the process exits.  Its device address is looked up once per device,
// on the first call made with that device current; make that first call
// before any stream capture.  Every call uses the same array and leaves its
// contents behind, so each call clears the tickets and the status word before
// its kernel runs, and calls that overlap on the GPU (on two streams, or on
// two host threads) race on it.
#include <mutex>

#include "kernels.h"

namespace asrspec {
namespace {

constexpr size_t NOALLOC_WS_FLOATS = size_t(1) << 21;  // 8 MiB of split-K partial sums
constexpr int NOALLOC_TICKETS = 4096;                  // output tiles
constexpr size_t NOALLOC_FLOATS = NOALLOC_WS_FLOATS + NOALLOC_TICKETS + 64;

// [0, WS) partial sums | [WS, WS + TICKETS) tile tickets (int) | status word (int)
static __device__ __align__(256) float g_noalloc_scratch[NOALLOC_FLOATS];

constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
float* g_scratch_ptr[MAX_DEVICES] = {};

// Device address of the scratch array on the current device (looked up once).
int scratch_on_current_device(float** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= MAX_DEVICES) return ASR_E_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return ASR_E_CUDA;
    g_scratch_ptr[dev] = static_cast<float*>(p);
  }
  *out = g_scratch_ptr[dev];
  return ASR_OK;
}

}  // namespace
}  // namespace asrspec

using namespace asrspec;

extern "C" int asr_spec_gemm_noalloc(const void* A, const void* B, float* C, int32_t M, int32_t N, int32_t K,
                                     int32_t splits, void* stream) {
  if (!A || !B || !C || M < 1 || N < 1 || K < 64 || K % 64 || splits < 1 || splits > K / 64) return ASR_E_INVAL;
  const int bn = tc_pick_bn(N);
  const long long tiles = (long long)((M + 127) / 128) * ((N + bn - 1) / bn);
  if (tiles > NOALLOC_TICKETS || (long long)splits * tiles * 128 * bn > (long long)NOALLOC_WS_FLOATS)
    return ASR_E_CAPACITY;
  float* scratch = nullptr;
  if (int rc = scratch_on_current_device(&scratch)) return rc;
  int* tickets = reinterpret_cast<int*>(scratch + NOALLOC_WS_FLOATS);
  int* status = tickets + NOALLOC_TICKETS;
  cudaStream_t st = static_cast<cudaStream_t>(stream);

  TcGemm g{};
  g.bn = bn;
  if (!make_tmap_bf16(&g.mapA, A, M, K, 128) || !make_tmap_bf16(&g.mapB, B, N, K, bn)) return ASR_E_INVAL;
  g.M = M;
  g.N = N;
  g.K = K;
  g.splits = splits;
  g.ws = scratch;
  g.tickets = tickets;
  Epi e{};
  e.M = M;
  e.N = N;
  e.out_f32 = C;
  e.ld = N;
  // the previous call's tickets and status stay in the array: start from zero
  if (cudaMemsetAsync(tickets, 0, (NOALLOC_TICKETS + 1) * sizeof(int), st) != cudaSuccess) return ASR_E_CUDA;
  launch_gemm_tc(g, EPI_F32_MN, e, status, st);
  if (cudaGetLastError() != cudaSuccess) return ASR_E_CUDA;
  int s = 0;
  if (cudaMemcpyAsync(&s, status, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess) return ASR_E_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return ASR_E_CUDA;
  return s ? ASR_E_DEVICE : ASR_OK;
}
