// noalloc.cu -- env_policy_forward_noalloc: the bf16 policy/value network
// evaluation for callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc at the moment they need a policy
// output.  An on-vehicle control loop is the typical case: it runs under a
// hard period, and an allocation may synchronise the device or wait on the
// driver.  A host application that owns a fixed device-memory budget, and
// forbids any other allocator once it has started, is another.  This entry
// point serves both.  It needs no env handle, and its working memory (the
// packed bf16 weight images and a status word) is one file-scope device
// array, held by every GPU that loads it until the process exits.
//
// When the array and the kernels become resident depends on the CUDA
// runtime's module loading: with lazy loading (the default since CUDA 12.2)
// the module that holds the array is loaded by the first call on a device,
// and each kernel by its first launch, and that loading may itself take
// device memory and synchronise.  The first call on a device is therefore a
// warm-up: make it before the period in which nothing may allocate (and
// before any stream capture).  Later calls allocate nothing.
#include <climits>
#include <cstdint>
#include <mutex>

#include "auv_bf16.h"
#include "auvenv.h"

namespace {

constexpr size_t kStatusBytes = 256;
constexpr size_t kPolicyRegion = 160 * 1024;   // packed policy image (hidden 256, 16 outputs)
constexpr size_t kValueRegion = 152 * 1024;    // packed value image (hidden 256)
constexpr size_t kScratchBytes = kStatusBytes + kPolicyRegion + kValueRegion;   // 312.25 KiB

// The shared working memory of every call on a device.  In host code this
// name is only a stand-in for the device array: kernels get the address
// from cudaGetSymbolAddress (below), never the name itself.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
unsigned char* g_scratch_dev[kMaxDevices] = {nullptr};

// Device address of g_scratch on the current device, looked up once per
// device (the first call on each device does this).
int scratch_address(unsigned char** out) {
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return AUV_ERR_CUDA;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_dev[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_scratch) != cudaSuccess || !p) {
      cudaGetLastError();
      return AUV_ERR_CUDA;
    }
    g_scratch_dev[dev] = static_cast<unsigned char*>(p);
  }
  *out = g_scratch_dev[dev];
  return AUV_OK;
}

// Device memory of the current device (or managed memory).  A buffer on
// another GPU is rejected: the kernels would read or write it over the
// interconnect, or fault where peer access is off.
bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (a.type == cudaMemoryTypeManaged) return true;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice && a.device == dev;
}

}  // namespace

extern "C" int env_policy_forward_noalloc(int hidden, int policy_out, const float* policy,
                                          const float* value_w, const float* obs, int n,
                                          float* head, float* value, auv_status* status_out,
                                          void* stream) {
  // Shapes: the packed images of larger networks would not fit the array.
  if (hidden > 256 || policy_out > 16) return AUV_ERR_SIZE;
  if (hidden != 256 || policy_out != 16) return AUV_ERR_UNSUPPORTED;
  if (auv::bf16_policy_image_bytes() > kPolicyRegion ||
      auv::bf16_value_image_bytes() > kValueRegion)
    return AUV_ERR_SIZE;
  if (n < 1 || !policy || !obs || !head) return AUV_ERR_INVALID;
  if ((value == nullptr) != (value_w == nullptr)) return AUV_ERR_INVALID;
  const void* ptrs[5] = {policy, value_w, obs, head, value};
  for (const void* p : ptrs) {
    if (!p) continue;
    if (reinterpret_cast<uintptr_t>(p) % 16 || !is_device_ptr(p)) return AUV_ERR_SIZE;
  }
  if (status_out && (reinterpret_cast<uintptr_t>(status_out) % 4 || !is_device_ptr(status_out)))
    return AUV_ERR_SIZE;
  unsigned char* base = nullptr;
  int rc = scratch_address(&base);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  auv::Status* status = reinterpret_cast<auv::Status*>(base);
  static_assert(sizeof(auv::Status) == sizeof(auv_status), "status block layout");
  void* pol_img = base + kStatusBytes;
  void* val_img = base + kStatusBytes + kPolicyRegion;
  // The array keeps the previous call's contents: reset the status word; the
  // packing kernel rewrites every byte of the images the engine reads.
  if (cudaMemsetAsync(status, 0, sizeof(auv::Status), s) != cudaSuccess) return AUV_ERR_CUDA;
  auv::Model M0 = {};
  M0.hidden = hidden;
  M0.policy_out = policy_out;
  cudaError_t e = auv::launch_pack_bf16(M0, policy, value_w, pol_img, val_img, s);
  if (e != cudaSuccess) return AUV_ERR_CUDA;
  e = auv::launch_forward_bf16(M0, pol_img, val_img, nullptr, obs, n, head, value, status, s);
  if (e != cudaSuccess) return AUV_ERR_CUDA;
  // The call's status word (a wait that gave up) for the caller, copied on
  // the stream after the kernels.
  if (status_out && cudaMemcpyAsync(status_out, status, sizeof(auv_status),
                                    cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return AUV_ERR_CUDA;
  return AUV_OK;
}
