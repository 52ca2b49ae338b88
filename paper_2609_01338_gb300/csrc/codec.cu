// 8-bit swap codec for KV blocks: the paper keeps swapped KV compressed with
// 8-bit quantization as its default codec (Sec. 5).  Per group of 64
// consecutive values of a block (64 head_dim entries of one K or V row):
// fp32 min and step = (max - min) / 255, code = round-half-even((x - min) /
// step) clamped to [0, 255] (0 when step == 0), decoded value = code * step +
// min (two fp32 roundings), rounded to the KV type and stored fp16-encoded
// like every pool value.  A compressed block holds the codes in the block's
// element order, then the (min, step) pairs in group order.
//
// One warp per group, lane i holding values 2i and 2i + 1: the block reads and
// writes are 128-byte (codes: 64-byte) contiguous per warp.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "kernels.hpp"
#include "mzc.h"

namespace mzc {

namespace {

__device__ __forceinline__ uint32_t q8_code(float x, float mn, float step) {
  if (!(step > 0.0f)) return 0u;
  const float q = rintf(__fdiv_rn(__fsub_rn(x, mn), step));
  return q <= 0.0f ? 0u : (q >= 255.0f ? 255u : static_cast<uint32_t>(q));
}

__global__ void q8_encode_kernel(const uint16_t* __restrict__ pool, const int32_t* __restrict__ phys,
                                 int64_t n_blocks, int64_t block_elems, uint8_t* __restrict__ out) {
  const int64_t gid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t gpb = block_elems / 64;  // groups per block
  if (gid >= n_blocks * gpb) return;
  const int64_t b = gid / gpb, g = gid - b * gpb;
  const uint32_t two =
      reinterpret_cast<const uint32_t*>(pool + static_cast<int64_t>(phys[b]) * block_elems + g * 64)[lane];
  const float x0 = __half2float(__ushort_as_half(static_cast<unsigned short>(two & 0xFFFFu)));
  const float x1 = __half2float(__ushort_as_half(static_cast<unsigned short>(two >> 16)));
  float mn = fminf(x0, x1), mx = fmaxf(x0, x1);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  const float step = __fdiv_rn(__fsub_rn(mx, mn), 255.0f);
  uint8_t* dst = out + b * (block_elems + 8 * gpb);
  reinterpret_cast<uint16_t*>(dst + g * 64)[lane] =
      static_cast<uint16_t>(q8_code(x0, mn, step) | (q8_code(x1, mn, step) << 8));
  if (lane == 0) *reinterpret_cast<float2*>(dst + block_elems + 8 * g) = make_float2(mn, step);
}

// Destination block of compressed block b: phys[b], or phys_begin + b when phys
// is null (a contiguous restore run).
__global__ void q8_decode_kernel(const uint8_t* __restrict__ in, int64_t n_blocks, int64_t block_elems,
                                 const int32_t* __restrict__ phys, int64_t phys_begin, int kv_bf16,
                                 uint16_t* __restrict__ pool) {
  const int64_t gid = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  const int64_t gpb = block_elems / 64;
  if (gid >= n_blocks * gpb) return;
  const int64_t b = gid / gpb, g = gid - b * gpb;
  const uint8_t* src = in + b * (block_elems + 8 * gpb);
  const uint32_t codes = reinterpret_cast<const uint16_t*>(src + g * 64)[lane];
  const float2 p = *reinterpret_cast<const float2*>(src + block_elems + 8 * g);
  float y0 = __fadd_rn(__fmul_rn(static_cast<float>(codes & 0xFFu), p.y), p.x);
  float y1 = __fadd_rn(__fmul_rn(static_cast<float>(codes >> 8), p.y), p.x);
  if (kv_bf16) {
    y0 = __bfloat162float(__float2bfloat16_rn(y0));
    y1 = __bfloat162float(__float2bfloat16_rn(y1));
  }
  const int64_t dst_block = phys ? static_cast<int64_t>(phys[b]) : phys_begin + b;
  const uint32_t h = static_cast<uint32_t>(__half_as_ushort(__float2half_rn(y0))) |
                     (static_cast<uint32_t>(__half_as_ushort(__float2half_rn(y1))) << 16);
  reinterpret_cast<uint32_t*>(pool + dst_block * block_elems + g * 64)[lane] = h;
}

}  // namespace

int64_t q8_block_bytes(int64_t block_elems) { return block_elems + 8 * (block_elems / 64); }

cudaError_t launch_q8_encode(const void* pool, const int32_t* phys, int64_t n_blocks,
                             int64_t block_elems, void* out, cudaStream_t st) {
  if (n_blocks <= 0) return cudaSuccess;
  const int64_t threads = n_blocks * (block_elems / 64) * 32;
  q8_encode_kernel<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, st>>>(
      static_cast<const uint16_t*>(pool), phys, n_blocks, block_elems, static_cast<uint8_t*>(out));
  return cudaGetLastError();
}

cudaError_t launch_q8_decode(const void* in, int64_t n_blocks, int64_t block_elems,
                             const int32_t* phys, int64_t phys_begin, int32_t kv_dtype, void* pool,
                             cudaStream_t st) {
  if (n_blocks <= 0) return cudaSuccess;
  const int64_t threads = n_blocks * (block_elems / 64) * 32;
  q8_decode_kernel<<<static_cast<unsigned>((threads + 255) / 256), 256, 0, st>>>(
      static_cast<const uint8_t*>(in), n_blocks, block_elems, phys, phys_begin,
      kv_dtype == MZC_KV_BF16 ? 1 : 0, static_cast<uint16_t*>(pool));
  return cudaGetLastError();
}

}  // namespace mzc
