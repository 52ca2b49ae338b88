// Causal grouped-query flash attention for prefill over a block-table KV
// cache (the paper's single-pass attention over non-contiguous KV chunks with
// online softmax, Sec. 4.2).
//
// Rows: for KV head g, the n tokens x (hq/hkv) query heads sharing g are
// flattened token-major (row r = token r / group, head g*group + r % group),
// so one CTA's 64 rows reuse every K/V tile group times.  Each CTA walks
// 64-key tiles of its key range: the 16-token blocks of a tile are located
// through the block table and copied into shared memory with cp.async
// (double-buffered, 16-byte chunks, XOR-swizzled rows), S = Q K^T and
// O += P V run on warp-level tensor-core MMA (m16n8k16, fp32 accumulate),
// and the softmax is the online (running max / running sum) form in base 2.
// Keys past the tile's largest query position are zero-filled, never read.
//
// Long key ranges with few rows are split across CTAs (split-KV); each split
// writes its normalised partial output and log-sum-exp to scratch and a
// combine kernel merges them.
#include <cmath>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {

constexpr int kRows = 64;  // query rows per CTA (4 warps x 16)
constexpr int kKeys = 64;  // keys per tile

__device__ __forceinline__ uint32_t swz(int row, int chunk) {
  return static_cast<uint32_t>(chunk ^ (row & 7));
}

template <int HD, bool F16>
__global__ void __launch_bounds__(128) attn_kernel(
    const uint16_t* __restrict__ q, const int32_t* __restrict__ pos, int n, int hq, int hkv,
    const int32_t* __restrict__ table, int64_t n_logical, const uint16_t* __restrict__ pool,
    int64_t pool_blocks, uint16_t* __restrict__ out, float* __restrict__ part_o,
    float* __restrict__ part_lse, int keys_per_split, int n_splits, float scale_log2,
    int32_t* status) {
  constexpr int CH = HD / 8;  // 16-byte chunks per row
  extern __shared__ __align__(128) uint8_t smem[];
  uint16_t* sQ = reinterpret_cast<uint16_t*>(smem);
  uint16_t* sK = sQ + kRows * HD;
  uint16_t* sV = sK + 2 * kKeys * HD;
  __shared__ int s_maxpos;

  const int g = blockIdx.y;
  const int group = hq / hkv;
  const int R = n * group;
  const int r0 = blockIdx.x * kRows;
  const int split = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t blk_elems = 2LL * hkv * 16 * HD;
  const int64_t v_off = static_cast<int64_t>(hkv) * 16 * HD;

  if (tid == 0) s_maxpos = -1;
  // Q tile
  for (int i = tid; i < kRows * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const int rr = r0 + r;
    uint16_t* dst = sQ + r * HD + swz(r, c) * 8;
    if (rr < R) {
      const int t = rr / group, h = g * group + rr % group;
      cp_async16(smem_u32(dst), q + (static_cast<int64_t>(t) * hq + h) * HD + c * 8);
    } else {
      *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
  }
  cp_async_commit();
  __syncthreads();
  if (tid < kRows && r0 + tid < R) atomicMax(&s_maxpos, pos[(r0 + tid) / group]);
  __syncthreads();
  const int kv_len = s_maxpos + 1;
  const int k_begin = split * keys_per_split;
  const int k_end = min(kv_len, k_begin + keys_per_split);

  // this thread's two rows in the m16n8 accumulator layout
  const int rowA = r0 + warp * 16 + (lane >> 2);
  const int rowB = rowA + 8;
  const int posA = rowA < R ? pos[rowA / group] : -1;
  const int posB = rowB < R ? pos[rowB / group] : -1;

  float o[HD / 8][4];
#pragma unroll
  for (int j = 0; j < HD / 8; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.0f;
  float mA = -INFINITY, mB = -INFINITY, lA = 0.0f, lB = 0.0f;

  auto load_tile = [&](int kb, int buf) {
    uint16_t* dk = sK + buf * kKeys * HD;
    uint16_t* dv = sV + buf * kKeys * HD;
    for (int i = tid; i < kKeys * CH; i += 128) {
      const int kr = i / CH, c = i % CH;
      const int key = kb + kr;
      const uint32_t off = kr * HD + swz(kr, c) * 8;
      bool ok = key < k_end;
      int32_t phys = -1;
      if (ok) {
        const int blk = key >> 4;
        phys = blk < n_logical ? table[blk] : -1;
        if (phys < 0 || phys >= pool_blocks) {
          set_status(status, kStatusDevice);
          ok = false;
        }
      }
      if (ok) {
        const uint16_t* src = pool + static_cast<int64_t>(phys) * blk_elems +
                              (static_cast<int64_t>(g) * 16 + (key & 15)) * HD + c * 8;
        cp_async16(smem_u32(dk + off), src);
        cp_async16(smem_u32(dv + off), src + v_off);
      } else {
        *reinterpret_cast<uint4*>(dk + off) = make_uint4(0, 0, 0, 0);
        *reinterpret_cast<uint4*>(dv + off) = make_uint4(0, 0, 0, 0);
      }
    }
    cp_async_commit();
  };

  const int n_tiles = k_end > k_begin ? (k_end - k_begin + kKeys - 1) / kKeys : 0;
  uint32_t qf[HD / 16][4];
  if (n_tiles > 0) load_tile(k_begin, 0);
  cp_async_wait<0>();  // (the Q tile is complete once the first K/V group is)
  if (n_tiles > 0) {
    // not all of tile 0 may be complete: wait_group 0 above waited for all groups
  }
  __syncthreads();
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk) {
    const int r = warp * 16 + (lane & 15);
    const int c = kk * 2 + (lane >> 4);
    ldsm_x4(smem_u32(sQ + r * HD + swz(r, c) * 8), qf[kk][0], qf[kk][1], qf[kk][2], qf[kk][3]);
  }

  for (int t = 0; t < n_tiles; ++t) {
    const int buf = t & 1;
    const int kb = k_begin + t * kKeys;
    if (t + 1 < n_tiles) {
      load_tile(kb + kKeys, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint16_t* tk = sK + buf * kKeys * HD;
    const uint16_t* tv = sV + buf * kKeys * HD;

    float s[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.0f;
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk) {
#pragma unroll
      for (int np = 0; np < 4; ++np) {
        const int key = np * 16 + (lane & 7) + ((lane >> 4) << 3);
        const int c = kk * 2 + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(smem_u32(tk + key * HD + swz(key, c) * 8), b0, b1, b2, b3);
        mma_16816<F16>(s[2 * np], qf[kk], b0, b1);
        mma_16816<F16>(s[2 * np + 1], qf[kk], b2, b3);
      }
    }
    // mask, scale, running max
    float tmA = -INFINITY, tmB = -INFINITY;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int key = kb + j * 8 + 2 * (lane & 3) + e;
        const bool va = key <= posA && key < k_end;
        const bool vb = key <= posB && key < k_end;
        s[j][e] = va ? s[j][e] * scale_log2 : -INFINITY;
        s[j][2 + e] = vb ? s[j][2 + e] * scale_log2 : -INFINITY;
        tmA = fmaxf(tmA, s[j][e]);
        tmB = fmaxf(tmB, s[j][2 + e]);
      }
    }
#pragma unroll
    for (int o2 = 1; o2 <= 2; o2 <<= 1) {
      tmA = fmaxf(tmA, __shfl_xor_sync(0xffffffffu, tmA, o2));
      tmB = fmaxf(tmB, __shfl_xor_sync(0xffffffffu, tmB, o2));
    }
    const float nmA = fmaxf(mA, tmA), nmB = fmaxf(mB, tmB);
    const float baseA = nmA == -INFINITY ? 0.0f : nmA;
    const float baseB = nmB == -INFINITY ? 0.0f : nmB;
    const float alA = exp2f(mA - baseA), alB = exp2f(mB - baseB);
    mA = nmA;
    mB = nmB;
    float rsA = 0.0f, rsB = 0.0f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      s[j][0] = exp2f(s[j][0] - baseA);
      s[j][1] = exp2f(s[j][1] - baseA);
      s[j][2] = exp2f(s[j][2] - baseB);
      s[j][3] = exp2f(s[j][3] - baseB);
      rsA += s[j][0] + s[j][1];
      rsB += s[j][2] + s[j][3];
    }
    lA = lA * alA + rsA;
    lB = lB * alB + rsB;
#pragma unroll
    for (int j = 0; j < HD / 8; ++j) {
      o[j][0] *= alA;
      o[j][1] *= alA;
      o[j][2] *= alB;
      o[j][3] *= alB;
    }
    // O += P V
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
      uint32_t a[4];
      a[0] = pack2<F16>(s[2 * kk][0], s[2 * kk][1]);
      a[1] = pack2<F16>(s[2 * kk][2], s[2 * kk][3]);
      a[2] = pack2<F16>(s[2 * kk + 1][0], s[2 * kk + 1][1]);
      a[3] = pack2<F16>(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
      for (int dp = 0; dp < HD / 16; ++dp) {
        const int key = kk * 16 + (lane & 7) + (((lane >> 3) & 1) << 3);
        const int c = dp * 2 + (lane >> 4);
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(smem_u32(tv + key * HD + swz(key, c) * 8), b0, b1, b2, b3);
        mma_16816<F16>(o[2 * dp], a, b0, b1);
        mma_16816<F16>(o[2 * dp + 1], a, b2, b3);
      }
    }
    __syncthreads();
  }

#pragma unroll
  for (int o2 = 1; o2 <= 2; o2 <<= 1) {
    lA += __shfl_xor_sync(0xffffffffu, lA, o2);
    lB += __shfl_xor_sync(0xffffffffu, lB, o2);
  }
  const float invA = lA > 0.0f ? 1.0f / lA : 0.0f;
  const float invB = lB > 0.0f ? 1.0f / lB : 0.0f;
  const int col0 = 2 * (lane & 3);
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int rr = half ? rowB : rowA;
    if (rr >= R) continue;
    const float inv = half ? invB : invA;
    const int t = rr / group, h = g * group + rr % group;
    const int64_t orow = static_cast<int64_t>(t) * hq + h;
    if (n_splits == 1) {
      uint16_t* dst = out + orow * HD;
#pragma unroll
      for (int j = 0; j < HD / 8; ++j)
        *reinterpret_cast<uint32_t*>(dst + j * 8 + col0) =
            pack2<true>(o[j][2 * half] * inv, o[j][2 * half + 1] * inv);
    } else {
      float* dst = part_o + (static_cast<int64_t>(split) * n * hq + orow) * HD;
#pragma unroll
      for (int j = 0; j < HD / 8; ++j)
        *reinterpret_cast<float2*>(dst + j * 8 + col0) =
            make_float2(o[j][2 * half] * inv, o[j][2 * half + 1] * inv);
      if ((lane & 3) == 0) {
        const float l = half ? lB : lA, m = half ? mB : mA;
        part_lse[static_cast<int64_t>(split) * n * hq + orow] =
            l > 0.0f ? m + log2f(l) : -INFINITY;
      }
    }
  }
}

// out[row] = sum_s 2^(lse_s - lse_max) o_s / sum_s 2^(lse_s - lse_max); one warp per row.
template <int HD>
__global__ void attn_combine_kernel(const float* __restrict__ part_o,
                                    const float* __restrict__ part_lse, int64_t rows, int n_splits,
                                    uint16_t* __restrict__ out) {
  const int64_t row = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  float mx = -INFINITY;
  for (int s = 0; s < n_splits; ++s) mx = fmaxf(mx, part_lse[s * rows + row]);
  constexpr int PER = HD / 32;
  float acc[PER];
#pragma unroll
  for (int j = 0; j < PER; ++j) acc[j] = 0.0f;
  float wsum = 0.0f;
  for (int s = 0; s < n_splits; ++s) {
    const float l = part_lse[s * rows + row];
    if (l == -INFINITY) continue;
    const float w = exp2f(l - mx);
    wsum += w;
    const float* src = part_o + (s * rows + row) * HD + lane * PER;
#pragma unroll
    for (int j = 0; j < PER; ++j) acc[j] += w * src[j];
  }
  const float inv = wsum > 0.0f ? 1.0f / wsum : 0.0f;
  uint16_t* dst = out + row * HD + lane * PER;
#pragma unroll
  for (int j = 0; j < PER; j += 2)
    *reinterpret_cast<uint32_t*>(dst + j) = pack2<true>(acc[j] * inv, acc[j + 1] * inv);
}

template <int HD, bool F16>
cudaError_t launch_hd(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq, int32_t hkv,
                      const int32_t* table, int64_t n_logical, const void* pool,
                      int64_t pool_blocks, uint16_t* out, float* part_o, float* part_lse,
                      int n_splits, int keys_per_split, int32_t* status, cudaStream_t st) {
  constexpr int SMEM = (kRows + 4 * kKeys) * HD * 2;
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(attn_kernel<HD, F16>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int group = hq / hkv;
  const int64_t R = n * group;
  dim3 grid(static_cast<unsigned>((R + kRows - 1) / kRows), static_cast<unsigned>(hkv),
            static_cast<unsigned>(n_splits));
  const float scale_log2 = static_cast<float>(1.0 / std::sqrt(static_cast<double>(HD)) * 1.4426950408889634);
  attn_kernel<HD, F16><<<grid, 128, SMEM, st>>>(
      q, pos, static_cast<int>(n), hq, hkv, table, n_logical,
      static_cast<const uint16_t*>(pool), pool_blocks, out, part_o, part_lse, keys_per_split,
      n_splits, scale_log2, status);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || n_splits == 1) return e;
  const int64_t rows = n * hq;
  attn_combine_kernel<HD><<<static_cast<unsigned>((rows + 7) / 8), 256, 0, st>>>(
      part_o, part_lse, rows, n_splits, out);
  return cudaGetLastError();
}

}  // namespace

void attention_split(int64_t n, int32_t hq, int32_t hkv, int64_t max_keys, int num_sms,
                     int* n_splits, int* keys_per_split) {
  const int64_t ctas = ((n * (hq / hkv) + kRows - 1) / kRows) * hkv;
  int s = 1;
  const int64_t target = 2LL * num_sms;
  if (ctas < target && max_keys > 1024) {
    s = static_cast<int>((target + ctas - 1) / ctas);
    const int64_t max_s = (max_keys + 511) / 512;  // at least 512 keys per split
    if (s > max_s) s = static_cast<int>(max_s);
    if (s > 64) s = 64;
    if (s < 1) s = 1;
  }
  int64_t per = (max_keys + s - 1) / s;
  per = (per + kKeys - 1) / kKeys * kKeys;
  if (per < kKeys) per = kKeys;
  *n_splits = s;
  *keys_per_split = static_cast<int>(per);
}

int64_t attention_scratch_bytes(int64_t n, int32_t hq, int32_t hd, int n_splits) {
  if (n_splits <= 1) return 0;
  return static_cast<int64_t>(n_splits) * n * hq * (static_cast<int64_t>(hd) + 1) * 4;
}

cudaError_t launch_attention(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                             int32_t hkv, int32_t hd, const int32_t* table, int64_t n_logical,
                             const void* pool, int64_t pool_blocks, int32_t kv_dtype,
                             uint16_t* out, void* scratch, int64_t scratch_bytes,
                             int64_t max_keys, int num_sms, int32_t* status, cudaStream_t st) {
  if (n <= 0) return cudaSuccess;
  int s = 1, per = 0;
  attention_split(n, hq, hkv, max_keys, num_sms, &s, &per);
  if (s > 1 && (scratch == nullptr || scratch_bytes < attention_scratch_bytes(n, hq, hd, s))) {
    s = 1;
    per = static_cast<int>((max_keys + kKeys - 1) / kKeys * kKeys);
  }
  float* part_o = static_cast<float*>(scratch);
  float* part_lse = s > 1 ? part_o + static_cast<int64_t>(s) * n * hq * hd : nullptr;
  const bool f16 = kv_dtype == 1;
  if (hd == 64)
    return f16 ? launch_hd<64, true>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks, out,
                                     part_o, part_lse, s, per, status, st)
               : launch_hd<64, false>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks,
                                      out, part_o, part_lse, s, per, status, st);
  if (hd == 128)
    return f16 ? launch_hd<128, true>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks,
                                      out, part_o, part_lse, s, per, status, st)
               : launch_hd<128, false>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks,
                                       out, part_o, part_lse, s, per, status, st);
  return cudaErrorInvalidValue;
}

}  // namespace mzc
