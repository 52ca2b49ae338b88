// Memory-bound kernels of the prefill path: embedding gather, RMSNorm,
// rotary embedding fused with the KV-block write, the LM-head GEMV, and the
// block gather/poison used by eviction.  All global accesses are 16-byte
// vectors along the contiguous dimension.
#include <algorithm>
#include <cstdio>

#include <cstdlib>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

bool pdl_enabled() {
  static const bool on = [] {
    const char* e = std::getenv("MZC_PDL");
    return !(e && e[0] == '0');
  }();
  return on;
}

namespace {

__device__ __forceinline__ float bf16_lo(uint32_t u) { return __uint_as_float(u << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t u) { return __uint_as_float(u & 0xFFFF0000u); }

__device__ __forceinline__ void unpack8_f16(const uint4& v, float* f) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

__device__ __forceinline__ void unpack8_bf16(const uint4& v, float* f) {
  f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x);
  f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
  f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z);
  f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

// A value rounded to the KV storage precision (bf16 when !F16KV), encoded as
// fp16 so that the attention reads one format.  The encoding is exact for
// bf16 values of magnitude 0 or in [2^-14, 65504]; below 2^-14 only fp16's
// subnormal precision is kept, and from 65520 on the value becomes infinite
// (the kernel then records MZC_ERR_OVERFLOW).
template <bool F16KV>
__device__ __forceinline__ float kv_round(float x) {
  if constexpr (F16KV) {
    return x;
  } else {
    return __bfloat162float(__float2bfloat16_rn(x));
  }
}

template <bool F16>
__device__ __forceinline__ uint4 pack8(const float* f) {
  return make_uint4(pack2<F16>(f[0], f[1]), pack2<F16>(f[2], f[3]), pack2<F16>(f[4], f[5]),
                    pack2<F16>(f[6], f[7]));
}

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  const int nw = blockDim.x >> 5;
  float t = lane < nw ? red[lane] : 0.0f;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
  __syncthreads();
  return t;
}

// x[i][:] = embed[tokens[i]][:] widened to fp32; one CTA per row.
__global__ void embed_kernel(const int32_t* __restrict__ tokens, const uint16_t* __restrict__ emb,
                             int d, int64_t vocab, float* __restrict__ x, int32_t* status) {
  pdl_enter();
  const int64_t i = blockIdx.x;
  const int32_t t = tokens[i];
  if (t < 0 || t >= vocab) {
    if (threadIdx.x == 0) set_status(status, kStatusDevice);
    return;
  }
  const uint4* src = reinterpret_cast<const uint4*>(emb + static_cast<int64_t>(t) * d);
  float4* dst = reinterpret_cast<float4*>(x + i * d);
  for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
    float f[8];
    unpack8_bf16(src[c], f);
    dst[2 * c] = make_float4(f[0], f[1], f[2], f[3]);
    dst[2 * c + 1] = make_float4(f[4], f[5], f[6], f[7]);
  }
}

// y = x * rsqrt(mean(x^2) + eps) * g, fp32 math, fp16 out; one CTA per row.
__global__ void rmsnorm_kernel(const float* __restrict__ x, const float* __restrict__ g, int d,
                               float eps, uint16_t* __restrict__ y, int32_t* status) {
  pdl_enter();
  __shared__ float red[32];
  const int64_t i = blockIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + i * d);
  float ss = 0.0f;
  for (int c = threadIdx.x; c < d / 4; c += blockDim.x) {
    float4 v = xr[c];
    ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  const float4* gr = reinterpret_cast<const float4*>(g);
  uint4* yr = reinterpret_cast<uint4*>(y + i * d);
  float amax = 0.0f;
  for (int c = threadIdx.x; c < d / 8; c += blockDim.x) {
    float4 a = xr[2 * c], b = xr[2 * c + 1], ga = gr[2 * c], gb = gr[2 * c + 1];
    float f[8] = {a.x * r * ga.x, a.y * r * ga.y, a.z * r * ga.z, a.w * r * ga.w,
                  b.x * r * gb.x, b.y * r * gb.y, b.z * r * gb.z, b.w * r * gb.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) amax = fmaxf(amax, fabsf(f[e]));
    yr[c] = pack8<true>(f);
  }
  note_f16_overflow(status, amax);
}

// The same RMSNorm, one warp per row with the row held in registers (read
// once, reduced with shuffles, no block barrier): for d = 256 * G, G <= 16.
// Lane c owns the 8-float groups c, c + 32, ...  G is a template constant so
// a row takes only the registers it needs (more warps per SM in flight).
constexpr int kRowVecs = 16;  // 8-float groups per lane: d <= 4096

template <int G>
__global__ void __launch_bounds__(256, G <= 8 ? 3 : (G <= 12 ? 2 : 1)) rmsnorm_warp_kernel(const float* __restrict__ x,
                                                           const float* __restrict__ g, int64_t n,
                                                           float eps, uint16_t* __restrict__ y,
                                                           int32_t* status) {
  pdl_enter();
  constexpr int d = 256 * G;
  const int64_t i = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (i >= n) return;
  const float4* xr = reinterpret_cast<const float4*>(x + i * d);
  float4 a[G], b[G];
  float ss = 0.0f;
#pragma unroll
  for (int k = 0; k < G; ++k) {
    const int c = k * 32 + lane;
    a[k] = xr[2 * c];
    b[k] = xr[2 * c + 1];
  }
#pragma unroll
  for (int k = 0; k < G; ++k)
    ss += a[k].x * a[k].x + a[k].y * a[k].y + a[k].z * a[k].z + a[k].w * a[k].w +
          b[k].x * b[k].x + b[k].y * b[k].y + b[k].z * b[k].z + b[k].w * b[k].w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, o);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  const float4* gr = reinterpret_cast<const float4*>(g);
  uint4* yr = reinterpret_cast<uint4*>(y + i * d);
  float amax = 0.0f;
#pragma unroll
  for (int k = 0; k < G; ++k) {
    const int c = k * 32 + lane;
    const float4 ga = gr[2 * c], gb = gr[2 * c + 1];
    float f[8] = {a[k].x * r * ga.x, a[k].y * r * ga.y, a[k].z * r * ga.z, a[k].w * r * ga.w,
                  b[k].x * r * gb.x, b[k].y * r * gb.y, b[k].z * r * gb.z, b[k].w * r * gb.w};
#pragma unroll
    for (int e = 0; e < 8; ++e) amax = fmaxf(amax, fabsf(f[e]));
    yr[c] = pack8<true>(f);
  }
  note_f16_overflow(status, amax);  // the whole warp holds this row
}

// The same RMSNorm for short row sets (a prompt of a few hundred rows): one
// 128-thread CTA per row, the row and the scale vector loaded together and
// held in registers.  With one warp per row a 128-row call ran on 16 SMs, each
// pulling 96 KB through one round trip of loads; here 128 SMs share it.
template <int G>
__global__ void __launch_bounds__(128) rmsnorm_cta_kernel(const float* __restrict__ x,
                                                          const float* __restrict__ g, float eps,
                                                          uint16_t* __restrict__ y, int32_t* status) {
  pdl_enter();
  __shared__ float red[32];
  constexpr int d = 256 * G, NG = 32 * G;   // 8-float groups in a row
  constexpr int PER = (NG + 127) / 128;     // groups per thread
  const int64_t i = blockIdx.x;
  const int t = threadIdx.x;
  const float4* xr = reinterpret_cast<const float4*>(x + i * d);
  const float4* gr = reinterpret_cast<const float4*>(g);
  float4 a[PER], b[PER], ga[PER], gb[PER];
  float ss = 0.0f;
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int c = k * 128 + t;
    if (c < NG) {
      a[k] = xr[2 * c];
      b[k] = xr[2 * c + 1];
      ga[k] = gr[2 * c];
      gb[k] = gr[2 * c + 1];
    }
  }
#pragma unroll
  for (int k = 0; k < PER; ++k)
    if (k * 128 + t < NG)
      ss += a[k].x * a[k].x + a[k].y * a[k].y + a[k].z * a[k].z + a[k].w * a[k].w +
            b[k].x * b[k].x + b[k].y * b[k].y + b[k].z * b[k].z + b[k].w * b[k].w;
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  uint4* yr = reinterpret_cast<uint4*>(y + i * d);
  float amax = 0.0f;
#pragma unroll
  for (int k = 0; k < PER; ++k) {
    const int c = k * 128 + t;
    if (c >= NG) continue;
    float f[8] = {a[k].x * r * ga[k].x, a[k].y * r * ga[k].y, a[k].z * r * ga[k].z, a[k].w * r * ga[k].w,
                  b[k].x * r * gb[k].x, b[k].y * r * gb[k].y, b[k].z * r * gb[k].z, b[k].w * r * gb[k].w};
#pragma unroll
    for (int e = 0; e < 8; ++e) amax = fmaxf(amax, fabsf(f[e]));
    yr[c] = pack8<true>(f);
  }
  note_f16_overflow(status, amax);
}

// rows up to which the one-CTA-per-row form is used
constexpr int64_t kRmsCtaRows = 512;

template <int G>
void launch_rmsnorm_warp(const float* x, const float* g, int64_t n, float eps, uint16_t* y,
                         int32_t* status, cudaStream_t st) {
  if (n <= kRmsCtaRows) {
    launch_k(rmsnorm_cta_kernel<G>, dim3(static_cast<unsigned>(n)), dim3(128), 0, st, x, g, eps, y, status);
    return;
  }
  launch_k(rmsnorm_warp_kernel<G>, dim3(static_cast<unsigned>((n + 7) / 8)), dim3(256), 0, st, x, g, n, eps, y,
           status);
}

// Rotary embedding (pairs (i, i + hd/2), angle pos * theta^(-2i/hd) from the
// fp32 tables) of q and k (fp16 projection output), then K/V rounded to the KV
// storage precision and stored, fp16-encoded, into their KV block slot:
// pool[table[pos/16]] = K [hkv][16][hd] then V [hkv][16][hd], slot pos % 16.
// q goes to q_out [n][hq][hd] in fp16.  One CTA per row.
template <bool F16KV>
__global__ void rope_kv_kernel(const uint16_t* __restrict__ qkv, const int32_t* __restrict__ pos,
                               int hq, int hkv, int hd, const float* __restrict__ cos_t,
                               const float* __restrict__ sin_t, const int32_t* __restrict__ table,
                               int64_t n_logical, uint16_t* __restrict__ pool,
                               int64_t pool_blocks, uint16_t* __restrict__ q_out,
                               int32_t* status) {
  pdl_enter();
  const int64_t i = blockIdx.x;
  const int p = pos[i];
  const int half = hd / 2;
  const int64_t blk = p >> 4;
  if (p < 0 || blk >= n_logical) {  // the rotary tables cover positions < n_logical * 16
    if (threadIdx.x == 0) set_status(status, kStatusDevice);
    return;
  }
  const int32_t phys = table[blk];
  const bool kv_ok = phys >= 0 && phys < pool_blocks;
  if (!kv_ok && threadIdx.x == 0) set_status(status, kStatusDevice);
  const int64_t blk_elems = 2LL * hkv * 16 * hd;
  uint16_t* kbase = pool + (kv_ok ? phys : 0) * blk_elems;
  uint16_t* vbase = kbase + static_cast<int64_t>(hkv) * 16 * hd;
  const int slot = p & 15;
  const uint16_t* row = qkv + i * static_cast<int64_t>(hq + 2 * hkv) * hd;
  const int rot_chunks = half / 8;              // 8-element chunks per half
  const int n_rot = (hq + hkv) * rot_chunks;    // q and k heads
  const int n_v = hkv * (hd / 8);
  const float* cs = cos_t + static_cast<int64_t>(p) * half;
  const float* sn = sin_t + static_cast<int64_t>(p) * half;
  float amax = 0.0f;  // largest |value| this thread stores fp16-encoded
  for (int w = threadIdx.x; w < n_rot + n_v; w += blockDim.x) {
    if (w < n_rot) {
      const int head = w / rot_chunks, c = (w % rot_chunks) * 8;
      const uint16_t* src = row + static_cast<int64_t>(head) * hd;
      float x1[8], x2[8], y1[8], y2[8];
      unpack8_f16(*reinterpret_cast<const uint4*>(src + c), x1);
      unpack8_f16(*reinterpret_cast<const uint4*>(src + c + half), x2);
      const float4 c0 = *reinterpret_cast<const float4*>(cs + c);
      const float4 c1 = *reinterpret_cast<const float4*>(cs + c + 4);
      const float4 s0 = *reinterpret_cast<const float4*>(sn + c);
      const float4 s1 = *reinterpret_cast<const float4*>(sn + c + 4);
      const float cc[8] = {c0.x, c0.y, c0.z, c0.w, c1.x, c1.y, c1.z, c1.w};
      const float ss[8] = {s0.x, s0.y, s0.z, s0.w, s1.x, s1.y, s1.z, s1.w};
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        y1[j] = x1[j] * cc[j] - x2[j] * ss[j];
        y2[j] = x2[j] * cc[j] + x1[j] * ss[j];
      }
      uint16_t* dst;
      if (head < hq) {
        dst = q_out + (i * hq + head) * hd;
      } else {
        if (!kv_ok) continue;
        dst = kbase + (static_cast<int64_t>(head - hq) * 16 + slot) * hd;
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          y1[j] = kv_round<F16KV>(y1[j]);
          y2[j] = kv_round<F16KV>(y2[j]);
        }
      }
#pragma unroll
      for (int j = 0; j < 8; ++j) amax = fmaxf(amax, fmaxf(fabsf(y1[j]), fabsf(y2[j])));
      *reinterpret_cast<uint4*>(dst + c) = pack8<true>(y1);
      *reinterpret_cast<uint4*>(dst + c + half) = pack8<true>(y2);
    } else {
      if (!kv_ok) continue;
      const int v = w - n_rot;
      const int head = v / (hd / 8), c = (v % (hd / 8)) * 8;
      const uint16_t* src = row + static_cast<int64_t>(hq + hkv + head) * hd + c;
      uint4 raw = *reinterpret_cast<const uint4*>(src);
      uint16_t* dst = vbase + (static_cast<int64_t>(head) * 16 + slot) * hd + c;
      if constexpr (!F16KV) {  // fp16 projection output rounded to bf16 precision
        float f[8];
        unpack8_f16(raw, f);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          f[j] = kv_round<false>(f[j]);
          amax = fmaxf(amax, fabsf(f[j]));
        }
        raw = pack8<true>(f);
      }
      *reinterpret_cast<uint4*>(dst) = raw;
    }
  }
  note_f16_overflow(status, amax);
}

// logits[v] = sum_k h[k] * W[v][k], h = RMSNorm(x_row) * g kept in fp32.
// Each CTA normalises the row into shared memory, then every warp streams
// whole vocabulary rows (16-byte loads, 4 rows in flight per warp).
__global__ void __launch_bounds__(256) lm_head_kernel(const float* __restrict__ x,
                                                      const float* __restrict__ g, int d,
                                                      float eps, const uint16_t* __restrict__ w,
                                                      int64_t vocab, float* __restrict__ logits) {
  pdl_enter();
  extern __shared__ float sh[];
  __shared__ float red[32];
  float ss = 0.0f;
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float v = x[c];
    ss += v * v;
  }
  ss = block_sum(ss, red);
  const float r = rsqrtf(ss / static_cast<float>(d) + eps);
  for (int c = threadIdx.x; c < d; c += blockDim.x) sh[c] = x[c] * r * g[c];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t gw = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + warp;
  const int64_t nw = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  const int chunks = d / 8;
  constexpr int R = 4;
  for (int64_t v0 = gw * R; v0 < vocab; v0 += nw * R) {
    float acc[R] = {0.f, 0.f, 0.f, 0.f};
    for (int c = lane; c < chunks; c += 32) {
      float hv[8];
      const float4 h0 = *reinterpret_cast<const float4*>(sh + c * 8);
      const float4 h1 = *reinterpret_cast<const float4*>(sh + c * 8 + 4);
      hv[0] = h0.x; hv[1] = h0.y; hv[2] = h0.z; hv[3] = h0.w;
      hv[4] = h1.x; hv[5] = h1.y; hv[6] = h1.z; hv[7] = h1.w;
      uint4 wv[R];
#pragma unroll
      for (int j = 0; j < R; ++j)
        if (v0 + j < vocab)
          wv[j] = __ldcs(reinterpret_cast<const uint4*>(w + (v0 + j) * d) + c);
#pragma unroll
      for (int j = 0; j < R; ++j) {
        if (v0 + j < vocab) {
          float f[8];
          unpack8_bf16(wv[j], f);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc[j] += hv[e] * f[e];
        }
      }
    }
#pragma unroll
    for (int j = 0; j < R; ++j) {
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[j] += __shfl_xor_sync(0xffffffffu, acc[j], o);
      if (lane == 0 && v0 + j < vocab) logits[v0 + j] = acc[j];
    }
  }
}

// dst[i] = src[i] for n 16-byte words; src may be mapped pinned host memory,
// read over the host link by the SMs (no copy engine involved).
__global__ void copy16_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int64_t n) {
  pdl_enter();
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n;
       i += static_cast<int64_t>(gridDim.x) * blockDim.x)
    dst[i] = src[i];
}

__global__ void gather_blocks_kernel(const uint4* __restrict__ pool, const int32_t* __restrict__ phys,
                                     int64_t chunks_per_block, uint4* __restrict__ dst) {
  const int64_t b = blockIdx.x;
  const uint4* src = pool + static_cast<int64_t>(phys[b]) * chunks_per_block;
  uint4* d = dst + b * chunks_per_block;
  for (int64_t c = threadIdx.x; c < chunks_per_block; c += blockDim.x) d[c] = src[c];
}

// Block b of the list (phys non-null) or of the run phys_begin + b (phys null).
__global__ void poison_blocks_kernel(uint4* __restrict__ pool, const int32_t* __restrict__ phys,
                                     int64_t phys_begin, int64_t chunks_per_block, uint32_t pattern2) {
  const int64_t b = blockIdx.x;
  const int64_t pb = phys ? static_cast<int64_t>(phys[b]) : phys_begin + b;
  uint4* d = pool + pb * chunks_per_block;
  const uint4 v = make_uint4(pattern2, pattern2, pattern2, pattern2);
  for (int64_t c = threadIdx.x; c < chunks_per_block; c += blockDim.x) d[c] = v;
}

// A wait that runs out: one thread waits on an mbarrier that nothing arrives
// on (or, with arrive != 0, that it arrived on first) through the same bounded
// wait as every kernel's pipeline waits, with a caller-chosen limit.
__global__ void wait_probe_kernel(int32_t arrive, int64_t limit_cycles, int32_t* status,
                                  int32_t* completed) {
  __shared__ uint64_t bar;
  mbar_init(&bar, 1);
  fence_barrier_init();
  if (arrive) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(&bar)) : "memory");
  *completed = mbar_wait(&bar, 0, status, limit_cycles) ? 1 : 0;
}

}  // namespace

cudaError_t launch_embed(const int32_t* tokens, int64_t n, const uint16_t* embed, int32_t d,
                         int64_t vocab, float* x, int32_t* status, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  launch_k(embed_kernel, dim3(static_cast<unsigned>(n)), dim3(256), 0, st, tokens, embed, d, vocab, x, status);
  return cudaGetLastError();
}

cudaError_t launch_rmsnorm(const float* x, const float* g, int64_t n, int32_t d, float eps,
                           uint16_t* y, cudaStream_t st, int32_t* status) {
  if (n <= 0) return cudaSuccess;
  switch (d % 256 == 0 ? d / 256 : 0) {
#define MZC_RMS_CASE(G)                         \
  case G:                                       \
    launch_rmsnorm_warp<G>(x, g, n, eps, y, status, st); \
    break;
    MZC_RMS_CASE(1)
    MZC_RMS_CASE(2)
    MZC_RMS_CASE(3)
    MZC_RMS_CASE(4)
    MZC_RMS_CASE(5)
    MZC_RMS_CASE(6)
    MZC_RMS_CASE(7)
    MZC_RMS_CASE(8)
    MZC_RMS_CASE(9)
    MZC_RMS_CASE(10)
    MZC_RMS_CASE(11)
    MZC_RMS_CASE(12)
    MZC_RMS_CASE(13)
    MZC_RMS_CASE(14)
    MZC_RMS_CASE(15)
    MZC_RMS_CASE(16)
#undef MZC_RMS_CASE
    default:
      launch_k(rmsnorm_kernel, dim3(static_cast<unsigned>(n)), dim3(256), 0, st, x, g, d, eps, y, status);
  }
  static_assert(kRowVecs == 16, "warp kernel instances for d = 256 .. 4096");
  return cudaGetLastError();
}

cudaError_t launch_rope_kv_write(const uint16_t* qkv, const int32_t* pos, int64_t n, int32_t hq,
                                 int32_t hkv, int32_t hd, const float* cos_t, const float* sin_t,
                                 const int32_t* table, int64_t n_logical, void* pool,
                                 int64_t pool_blocks, int32_t kv_dtype, uint16_t* q_out,
                                 int32_t* status, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  // a short row set (a prompt) has one CTA per row on as many SMs, each thread
  // walking its work items one load round trip after another: up to 1024
  // threads then give each item its own thread; longer row sets, bound by
  // HBM, keep 128-thread CTAs, several per SM
  const int items = (hq + hkv) * (hd / 16) + hkv * (hd / 8);
  const int threads = n <= 512 ? std::min(1024, std::max(128, (items + 31) / 32 * 32)) : 128;
  if (kv_dtype == 1)
    launch_k(rope_kv_kernel<true>, dim3(static_cast<unsigned>(n)), dim3(static_cast<unsigned>(threads)), 0, st,
        qkv, pos, hq, hkv, hd, cos_t, sin_t, table, n_logical, static_cast<uint16_t*>(pool),
        pool_blocks, q_out, status);
  else
    launch_k(rope_kv_kernel<false>, dim3(static_cast<unsigned>(n)), dim3(static_cast<unsigned>(threads)), 0, st,
        qkv, pos, hq, hkv, hd, cos_t, sin_t, table, n_logical, static_cast<uint16_t*>(pool),
        pool_blocks, q_out, status);
  return cudaGetLastError();
}

cudaError_t launch_lm_head(const float* x_row, const float* g, int32_t d, float eps,
                           const uint16_t* w, int64_t vocab, float* logits, int num_sms,
                           cudaStream_t st) {
  const int grid = num_sms * 4;
  launch_k(lm_head_kernel, dim3(grid), dim3(256), static_cast<size_t>(d) * sizeof(float), st, x_row, g, d, eps, w,
                                                                            vocab, logits);
  return cudaGetLastError();
}

cudaError_t launch_wait_probe(int32_t arrive, int64_t limit_cycles, int32_t* status,
                              int32_t* completed, cudaStream_t st) {
  wait_probe_kernel<<<1, 1, 0, st>>>(arrive, limit_cycles, status, completed);
  return cudaGetLastError();
}

cudaError_t launch_copy16(const void* src, void* dst, int64_t bytes, cudaStream_t st) {
  const int64_t n = (bytes + 15) / 16;
  if (n <= 0) return cudaSuccess;
  const int64_t blocks = std::min<int64_t>((n + 255) / 256, 1024);
  launch_k(copy16_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, st, static_cast<const uint4*>(src),
                                                                static_cast<uint4*>(dst), n);
  return cudaGetLastError();
}

cudaError_t launch_gather_blocks(const void* pool, const int32_t* phys, int64_t n,
                                 int64_t block_bytes, void* dst, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  gather_blocks_kernel<<<static_cast<unsigned>(n), 256, 0, st>>>(
      static_cast<const uint4*>(pool), phys, block_bytes / 16, static_cast<uint4*>(dst));
  return cudaGetLastError();
}

cudaError_t launch_poison_blocks(void* pool, const int32_t* phys, int64_t n, int64_t block_bytes,
                                 int32_t kv_dtype, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  // the largest finite fp16 value: finite, so a masked key (weight 0)
  // contributes exactly 0, and far outside any real K/V, so a read of a block
  // before its restore lands shows up in the results
  (void)kv_dtype;
  const uint32_t v16 = 0x7BFFu;  // the pool is fp16-encoded for both KV types
  poison_blocks_kernel<<<static_cast<unsigned>(n), 256, 0, st>>>(static_cast<uint4*>(pool), phys, 0,
                                                                  block_bytes / 16, v16 | (v16 << 16));
  return cudaGetLastError();
}

cudaError_t launch_poison_run(void* pool, int64_t phys_begin, int64_t n, int64_t block_bytes,
                              cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  const uint32_t v16 = 0x7BFFu;
  poison_blocks_kernel<<<static_cast<unsigned>(n), 256, 0, st>>>(static_cast<uint4*>(pool), nullptr,
                                                                  phys_begin, block_bytes / 16,
                                                                  v16 | (v16 << 16));
  return cudaGetLastError();
}

}  // namespace mzc
