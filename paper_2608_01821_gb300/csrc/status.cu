// status.cu -- status strings, the per-device error word and CUDA error
// bookkeeping shared by every entry point.
#include <mutex>

#include "common.cuh"

namespace davet {

namespace {
__device__ unsigned g_error_word;

thread_local int t_last_cuda_error = 0;

constexpr int kMaxDevices = 64;
unsigned* g_word_addr[kMaxDevices] = {};
std::mutex g_word_mu;
}  // namespace

davet_status cuda_fail(cudaError_t e) {
  t_last_cuda_error = static_cast<int>(e);
  return DAVET_ERR_CUDA;
}

davet_status check_launch() {
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}

unsigned* device_error_word() {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    cuda_fail(e);
    return nullptr;
  }
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> g(g_word_mu);
  if (!g_word_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_error_word);
    if (e != cudaSuccess) {
      cuda_fail(e);
      return nullptr;
    }
    g_word_addr[dev] = static_cast<unsigned*>(p);
  }
  return g_word_addr[dev];
}

}  // namespace davet

extern "C" int davet_version(void) { return 100; }

extern "C" const char* davet_status_string(int status) {
  switch (status) {
    case DAVET_OK: return "ok";
    case DAVET_ERR_INVALID_ARG: return "invalid argument";
    case DAVET_ERR_UNSUPPORTED: return "unsupported shape or size";
    case DAVET_ERR_CUDA: return "CUDA error";
    case DAVET_ERR_TIMEOUT: return "device wait timed out";
    case DAVET_ERR_DEVICE: return "device-side check failed";
    default: return "unknown status";
  }
}

extern "C" int davet_last_cuda_error(void) { return davet::t_last_cuda_error; }

extern "C" davet_status davet_device_status(unsigned* flags, int clear) {
  using namespace davet;
  if (device_error_word() == nullptr) return DAVET_ERR_CUDA;
  unsigned w = 0;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaMemcpyFromSymbol(&w, g_error_word, sizeof w);
  if (e != cudaSuccess) return cuda_fail(e);
  if (clear) {
    const unsigned zero = 0;
    e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof zero);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  if (flags) *flags = w;
  if (w & DEV_ERR_TIMEOUT) return DAVET_ERR_TIMEOUT;
  if (w) return DAVET_ERR_DEVICE;
  return DAVET_OK;
}

extern "C" davet_status davet_sync_status(void* stream, unsigned* flags) {
  using namespace davet;
  unsigned* word = device_error_word();
  if (word == nullptr) return DAVET_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  unsigned w = 0;
  cudaError_t e = cudaMemcpyAsync(&w, word, sizeof w, cudaMemcpyDeviceToHost, st);
  if (e != cudaSuccess) return cuda_fail(e);
  e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e);
  if (flags) *flags = w;
  if (w & DEV_ERR_TIMEOUT) return DAVET_ERR_TIMEOUT;
  if (w) return DAVET_ERR_DEVICE;
  return DAVET_OK;
}

extern "C" davet_status davet_step_attention_workspace(int batch, int64_t max_total_rows, int H, int D,
                                                       size_t* bytes) {
  if (!bytes || batch < 0 || max_total_rows < 0 || H < 1) return DAVET_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return DAVET_ERR_UNSUPPORTED;
  *bytes = 0;  // the attention kernel keeps its schedule in shared memory
  return DAVET_OK;
}

namespace davet {
namespace {
// One thread waits, with the library's bounded wait, on an mbarrier that
// nothing signals; the wait gives up after its budget and raises the timeout
// bit, the same path every producer/consumer wait of the kernels takes.
__global__ void selftest_wait_kernel(unsigned* err, int* gave_up) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
    const bool ok = mbar_wait(&bar, 0, err, nullptr);
    *gave_up = ok ? 0 : 1;
  }
}
}  // namespace
}  // namespace davet

extern "C" davet_status davet_selftest_wait_timeout(int* gave_up_dev, void* stream) {
  using namespace davet;
  if (!gave_up_dev) return DAVET_ERR_INVALID_ARG;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(err, gave_up_dev);
  return check_launch();
}
