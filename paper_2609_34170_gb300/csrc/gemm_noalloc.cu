// Allocation-free entry point of the split-K tensor-core projection GEMM.
//
// Some callers cannot allocate device memory at all: code that runs inside
// another runtime's memory pool with raw allocation disabled, plugin hosts
// that forbid cudaMalloc, or real-time control loops that must not touch the
// allocator after start-up (an allocation may synchronise the device or
// stall for milliseconds).  Such a caller cannot create a ravel handle,
// because ravel_create allocates the handle's split-K workspace.  This entry
// point runs the same GEMM kernel with its split-K scratch in one fixed
// file-scope device array instead; the caller still supplies the operands and
// the output.
//
// The array is part of the library image: every GPU that loads the library
// holds it until the process exits.  All calls share it, so calls that
// overlap on the GPU (different streams, or different host threads) race on
// it and must be serialised by the caller.  It keeps the last call's
// contents; each call clears the part that must start at zero.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/ravel.h"
#include "kernels.h"

namespace ravel {
namespace {

constexpr size_t kPartialBytes = (size_t)8 << 20;   // split-K partial tiles (fp32)
constexpr int kCounters = 1024;                      // per-tile arrival counters
constexpr size_t kZeroBytes = (kCounters + 64) * sizeof(int);   // counters + error word, cleared per call
constexpr size_t kScratchBytes = kPartialBytes + kZeroBytes;
constexpr int kMaxDevices = 64;

// The scratch: [partials | counters | error word].  In host code the name is
// only a stand-in for the symbol; the device address comes from
// cudaGetSymbolAddress at set-up.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

struct DeviceState {
  bool ready = false;
  unsigned char* scratch = nullptr;   // device address of g_scratch on this device
  int num_sms = 0;
};

DeviceState g_state[kMaxDevices];
std::mutex g_mutex;

// Once per device, with that device current: resolve the array's device
// address, the SM count and the tensor-map encoder, and raise the kernel's
// shared-memory limit.  Nothing here allocates.
cudaError_t setup_device(int dev, DeviceState** out) {
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState& s = g_state[dev];
  if (!s.ready) {
    unsigned char* ptr = nullptr;
    cudaError_t e = cudaGetSymbolAddress((void**)&ptr, g_scratch);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&s.num_sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = init_tc_gemm();
    if (e != cudaSuccess) return e;
    s.scratch = ptr;
    s.ready = true;
  }
  *out = &s;
  return cudaSuccess;
}

}  // namespace
}  // namespace ravel

using namespace ravel;

extern "C" ravel_status ravel_gemm_noalloc(const void* X, int M, int K, int lda, const void* W, int N, int ldw,
                                           int epi, void* out, int ldo, int out_dtype, const float* bias,
                                           void* stream) {
  if (!X || !W || !out) return RAVEL_EINVAL;
  if (M < 0 || N < 1 || K < 1 || lda < K || ldw < K || epi < 0 || epi > 3 || (out_dtype != 0 && out_dtype != 1))
    return RAVEL_EINVAL;
  if (M > RAVEL_NOALLOC_MAX_M || N > RAVEL_NOALLOC_MAX_N || K > RAVEL_NOALLOC_MAX_K) return RAVEL_ESHAPE;
  if (epi == EPI_GEGLU && (N % 128 || out_dtype != 1 || ldo < N / 2)) return RAVEL_EINVAL;
  if (epi != EPI_GEGLU && ldo < N) return RAVEL_EINVAL;
  if (epi == EPI_ADD_F32 && out_dtype != 0) return RAVEL_EINVAL;
  GemmArgs g{X, lda, W, ldw, M, N, K, (Epi)epi, out, ldo, out_dtype ? DT_BF16 : DT_F32, bias};
  if (!tc_gemm_supported(g)) return RAVEL_EINVAL;   // 16-byte aligned operands, K, lda, ldw multiples of 8
  if (M == 0) return RAVEL_OK;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RAVEL_ECUDA;
  DeviceState* s = nullptr;
  if (setup_device(dev, &s) != cudaSuccess) return RAVEL_ECUDA;
  cudaStream_t st = (cudaStream_t)stream;
  unsigned char* zero = s->scratch + kPartialBytes;
  if (cudaMemsetAsync(zero, 0, kZeroBytes, st) != cudaSuccess) return RAVEL_ECUDA;
  // The split plan is chosen so that the partials fit the array (fewer
  // splits, or none, when they would not).
  TcWorkspace ws{(float*)s->scratch, kPartialBytes, (int*)zero, kCounters, (int*)zero + kCounters};
  if (launch_gemm_tc(g, ws, s->num_sms, st, /*cluster=*/false) != cudaSuccess) return RAVEL_ECUDA;
  return RAVEL_OK;
}
