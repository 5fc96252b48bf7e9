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
// contents; each call clears the part that must start at zero (the tile
// counters).  Its error word is sticky: a bounded wait that runs out inside a
// GEMM sets it, and it stays set until ravel_gemm_noalloc_status reads it.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/ravel.h"
#include "kernels.h"

namespace ravel {
namespace {

constexpr size_t kPartialBytes = (size_t)8 << 20;   // split-K partial tiles (fp32)
constexpr int kCounters = 1024;                      // per-tile arrival counters
constexpr size_t kCounterBytes = kCounters * sizeof(int);       // cleared by every call
constexpr size_t kScratchBytes = kPartialBytes + kCounterBytes + 64 * sizeof(int);   // + the error word
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
// shared-memory limit.  Nothing here allocates.  None of it may run while `st`
// is being captured into a graph (it would invalidate the capture): a first
// call under capture is refused.
ravel_status setup_device(int dev, cudaStream_t st, DeviceState** out) {
  std::lock_guard<std::mutex> lock(g_mutex);
  DeviceState& s = g_state[dev];
  if (!s.ready) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) return RAVEL_ECUDA;
    if (cs != cudaStreamCaptureStatusNone) return RAVEL_EINVAL;
    unsigned char* ptr = nullptr;
    if (cudaGetSymbolAddress((void**)&ptr, g_scratch) != cudaSuccess) return RAVEL_ECUDA;
    if (cudaDeviceGetAttribute(&s.num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return RAVEL_ECUDA;
    if (init_tc_gemm() != cudaSuccess) return RAVEL_ECUDA;
    s.scratch = ptr;
    s.ready = true;
  }
  *out = &s;
  return RAVEL_OK;
}

int* error_word(const DeviceState* s) { return (int*)(s->scratch + kPartialBytes + kCounterBytes); }

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
  cudaStream_t st = (cudaStream_t)stream;
  DeviceState* s = nullptr;
  const ravel_status rs = setup_device(dev, st, &s);
  if (rs != RAVEL_OK) return rs;
  int* counters = (int*)(s->scratch + kPartialBytes);
  if (cudaMemsetAsync(counters, 0, kCounterBytes, st) != cudaSuccess) return RAVEL_ECUDA;
  // The split plan is chosen so that the partials fit the array (fewer
  // splits, or none, when they would not).
  TcWorkspace ws{(float*)s->scratch, kPartialBytes, counters, kCounters, error_word(s)};
  if (launch_gemm_tc(g, ws, s->num_sms, st, /*cluster=*/false) != cudaSuccess) return RAVEL_ECUDA;
  return RAVEL_OK;
}

extern "C" ravel_status ravel_gemm_noalloc_status(void* stream) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return RAVEL_ECUDA;
  cudaStream_t st = (cudaStream_t)stream;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(st, &cs) != cudaSuccess) return RAVEL_ECUDA;
  if (cs != cudaStreamCaptureStatusNone) return RAVEL_EINVAL;
  const DeviceState* s = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_state[dev].ready) return RAVEL_OK;   // no call has run on this device
    s = &g_state[dev];
  }
  if (cudaStreamSynchronize(st) != cudaSuccess) return RAVEL_ECUDA;
  int bits = 0;   // a synchronous copy into host memory: no staging buffer of ours
  if (cudaMemcpy(&bits, error_word(s), sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess) return RAVEL_ECUDA;
  if (!bits) return RAVEL_OK;
  if (cudaMemset(error_word(s), 0, sizeof(int)) != cudaSuccess) return RAVEL_ECUDA;
  return (bits & ERR_TIMEOUT) ? RAVEL_ETIMEOUT : RAVEL_EDEVICE;
}
