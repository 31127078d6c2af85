// fovea_retrieve_fuse_noalloc: the draft step for callers that cannot
// allocate device memory.  Its scratch is a file-scope device array instead
// of a caller-provided workspace; it calls no allocator of any kind.
#include <cstdio>
#include <mutex>

#include "common.cuh"

// The scratch every call of fovea_retrieve_fuse_noalloc uses.  Every GPU that
// loads the library holds it until the process exits.
static __device__ __align__(256) unsigned char g_noalloc_workspace[FOVEA_NOALLOC_WORKSPACE_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_addr[kMaxDevices] = {};   // device address of the array, per device

// Device address of the array on the current device.  In host code the
// array's name is only a host-side stand-in, so the address must come from
// cudaGetSymbolAddress, called once per device with that device current.
fovea_status workspace_address(void** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    char msg[256];
    snprintf(msg, sizeof(msg), "cudaGetDevice: %s", cudaGetErrorString(e));
    return fovea::report_error(FOVEA_ERR_CUDA, msg);
  }
  if (dev < 0 || dev >= kMaxDevices)
    return fovea::report_error(FOVEA_ERR_UNSUPPORTED, "device ordinal beyond the supported 64");
  std::lock_guard<std::mutex> lk(g_mu);
  if (g_addr[dev] == nullptr) {
    void* ptr = nullptr;
    e = cudaGetSymbolAddress(&ptr, g_noalloc_workspace);
    if (e != cudaSuccess || ptr == nullptr) {
      char msg[256];
      snprintf(msg, sizeof(msg), "cudaGetSymbolAddress of the static workspace: %s",
               cudaGetErrorString(e));
      return fovea::report_error(FOVEA_ERR_CUDA, msg);
    }
    g_addr[dev] = ptr;
  }
  *out = g_addr[dev];
  return FOVEA_OK;
}
}  // namespace

extern "C" FOVEA_API fovea_status fovea_retrieve_fuse_noalloc(
    const fovea_params* p, const fovea_memory* mem, const void* h, const int32_t* depth,
    const int32_t* row_offsets, const float* row_scale, float rho, int k_min, int k_max, int l_max,
    void* h_out, int32_t* counts, int32_t* indices, float* readout, float* gate, void* stream) {
  size_t need = 0;
  fovea_status st = fovea_workspace_size(p, mem, row_offsets, k_max, &need);
  if (st != FOVEA_OK) return st;
  if (need > (size_t)FOVEA_NOALLOC_WORKSPACE_BYTES) {
    char msg[256];
    snprintf(msg, sizeof(msg),
             "this call needs %zu bytes of scratch; the static workspace of "
             "fovea_retrieve_fuse_noalloc holds %zu (use fovea_retrieve_fuse with a larger "
             "workspace)",
             need, (size_t)FOVEA_NOALLOC_WORKSPACE_BYTES);
    return fovea::report_error(FOVEA_ERR_UNSUPPORTED, msg);
  }
  void* ws = nullptr;
  if ((st = workspace_address(&ws)) != FOVEA_OK) return st;
  // The array keeps the previous call's contents; the kernels expect the
  // header's reserved words at zero.  The error word is left as it is, so a
  // condition a call raised stays readable (fovea_noalloc_sync_errors) until
  // it is read.
  cudaError_t e = cudaMemsetAsync(static_cast<unsigned char*>(ws) + sizeof(int), 0,
                                  fovea::kWsHeaderBytes - sizeof(int),
                                  static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    char msg[256];
    snprintf(msg, sizeof(msg), "cudaMemsetAsync: %s", cudaGetErrorString(e));
    return fovea::report_error(FOVEA_ERR_CUDA, msg);
  }
  return fovea_retrieve_fuse(p, mem, h, depth, row_offsets, row_scale, rho, k_min, k_max, l_max,
                             h_out, counts, indices, readout, gate, ws,
                             FOVEA_NOALLOC_WORKSPACE_BYTES, stream);
}

extern "C" FOVEA_API fovea_status fovea_noalloc_sync_errors(void* stream) {
  void* ws = nullptr;
  fovea_status st = workspace_address(&ws);
  if (st != FOVEA_OK) return st;
  return fovea_sync_errors(ws, stream);
}
