// Attention whose split-KV partials live in a fixed device array of this
// file instead of caller memory: the kernels are those of attention.cu, run
// through launch_attention with this array as the scratch.
#include <cuda_runtime.h>

#include <mutex>

#include "kernels.hpp"

namespace mzc {

// The split-KV partials of mzc_k_attention_noalloc live in this file-scope
// device array instead of memory the caller allocates.  Every device that
// loads the library holds it until the process exits.  All calls share it:
// each call overwrites every partial it later reads (no part of it has to
// start at zero), so calls that overlap on the GPU race on its contents.
static __device__ __align__(256) uint8_t g_attn_noalloc_scratch[kAttnNoallocScratchBytes];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices] = {};

// Device address of the array on the current device.  In host code the
// array's name is only a host-side stand-in, so the address comes from
// cudaGetSymbolAddress, queried once per device with that device current.
cudaError_t noalloc_scratch(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lk(g_noalloc_mu);
  if (!g_noalloc_ptr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_attn_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_noalloc_ptr[dev] = p;
  }
  *out = g_noalloc_ptr[dev];
  return cudaSuccess;
}
}  // namespace

int64_t attention_noalloc_need(int64_t n, int32_t hq, int32_t hkv, int32_t hd, int64_t max_keys,
                               int num_sms) {
  int s = 1, per = 0;
  attention_split(n, hq, hkv, hd, max_keys, num_sms, &s, &per);
  return attention_scratch_bytes(n, hq, hd, s);
}

cudaError_t launch_attention_noalloc(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                                     int32_t hkv, int32_t hd, const int32_t* table,
                                     int64_t n_logical, const void* pool, int64_t pool_blocks,
                                     int32_t kv_dtype, uint16_t* out, int64_t max_keys,
                                     int num_sms, int32_t* status, cudaStream_t st) {
  if (attention_noalloc_need(n, hq, hkv, hd, max_keys, num_sms) > kAttnNoallocScratchBytes)
    return cudaErrorInvalidValue;  // checked by the caller first; no launch
  void* scratch = nullptr;
  cudaError_t e = noalloc_scratch(&scratch);
  if (e != cudaSuccess) return e;
  return launch_attention(q, pos, n, hq, hkv, hd, table, n_logical, pool, pool_blocks, kv_dtype,
                          out, scratch, kAttnNoallocScratchBytes, max_keys, num_sms, status, st);
}

}  // namespace mzc
