// api.cu -- library-wide entry points: status strings, the device error word
// and the device-side wait limit.
#include <atomic>
#include <mutex>

#include "common.cuh"

namespace {

__device__ unsigned g_ssm_device_error = 0;

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned* g_err_ptr[kMaxDevices] = {};
std::atomic<uint64_t> g_wait_limit_ns{2000000000ull};

}  // namespace

namespace ssm {

unsigned* device_error_word() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_err_ptr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_ssm_device_error) != cudaSuccess) return nullptr;
    g_err_ptr[dev] = static_cast<unsigned*>(p);
  }
  return g_err_ptr[dev];
}

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(); }

}  // namespace ssm

extern "C" {

const char* ssm_status_str(ssm_status s) {
  switch (s) {
    case SSM_OK: return "ok";
    case SSM_ERR_INVALID_ARG: return "invalid argument";
    case SSM_ERR_SHAPE: return "inconsistent shapes";
    case SSM_ERR_CAPACITY: return "output or workspace too small";
    case SSM_ERR_CUDA: return "CUDA error";
    case SSM_ERR_TIMEOUT: return "device wait timed out";
    case SSM_ERR_UNSUPPORTED: return "unsupported configuration";
    case SSM_ERR_DEVICE_INPUT: return "device input out of range";
  }
  return "unknown status";
}

const char* ssm_version(void) { return "libssm 0.1 (sm_103a)"; }

ssm_status ssm_get_device_error(ssm_stream_t stream) {
  unsigned* w = ssm::device_error_word();
  if (!w) return SSM_ERR_CUDA;
  if (cudaStreamSynchronize(reinterpret_cast<cudaStream_t>(stream)) != cudaSuccess) return SSM_ERR_CUDA;
  unsigned h = 0;
  if (cudaMemcpy(&h, w, sizeof(h), cudaMemcpyDeviceToHost) != cudaSuccess) return SSM_ERR_CUDA;
  if (h != 0) {
    const unsigned zero = 0;
    if (cudaMemcpy(w, &zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess) return SSM_ERR_CUDA;
  }
  return static_cast<ssm_status>(h);
}

ssm_status ssm_set_wait_limit_ns(uint64_t ns) {
  g_wait_limit_ns.store(ns == 0 ? 2000000000ull : ns);
  return SSM_OK;
}

}  // extern "C"
