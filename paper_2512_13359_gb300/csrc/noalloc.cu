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
// array that is reserved when the library's GPU code is loaded and held until
// the process exits.
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

bool is_device_ptr(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

}  // namespace

extern "C" int env_policy_forward_noalloc(int hidden, int policy_out, const float* policy,
                                          const float* value_w, const float* obs, int n,
                                          float* head, float* value, void* stream) {
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
  unsigned char* base = nullptr;
  int rc = scratch_address(&base);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  auv::Status* status = reinterpret_cast<auv::Status*>(base);
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
  return e == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}
