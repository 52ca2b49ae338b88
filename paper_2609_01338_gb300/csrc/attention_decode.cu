// Block-table attention for a few query tokens (decode after the first token,
// the step that follows time-to-first-token): R = n * (hq / hkv) <= 4 query
// rows per KV head, so there is no tile of 128 rows to give the tensor cores,
// and the kernel is bound by reading K and V once from HBM.
//
// Grid: x = KV head g, y = split of the key range (split-KV).  The 16 warps of
// a CTA form 8 pairs; pair p owns every 8th 16-token block of the split and
// keeps a ring of such blocks in shared memory: lane 0 of the pair's first warp
// fetches a block's K rows and V rows of head g (two contiguous 16 x hd runs of
// the pool block) with 1-D bulk copies that complete on the slot's mbarrier,
// several blocks ahead, and refills a slot once both warps released it.  The
// block numbers come from the block table, read one per lane 32 blocks at a
// time.  Warp h of the pair takes keys 8h..8h+7 of each block; lane L owns the
// head-dim columns [L*hd/32, (L+1)*hd/32) and keeps those q values in registers:
//   - scores: each lane forms its 8 partial dot products, ordered by
//     key XOR x (x = lane bits 2..4), so three shuffle-add rounds leave lane L
//     with key x's sum over its lane group and two more finish the reduction
//     without any selects;
//   - online softmax per row in base 2 (exact rescale: O lives in registers);
//   - P V: p of key k broadcast by a shuffle from lane 4k, fp32 FMAs into the
//     lane's output columns.
// The warps' partial (m, l, O) merge in shared memory at the end; with several
// splits the CTA writes its normalised O and base-2 log-sum-exp for the
// combine kernel of the prefill attention.
#include <cmath>
#include <mutex>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {

constexpr int kDecWarps = 16;
constexpr int kDecPairs = kDecWarps / 2;
constexpr int kDecThreads = kDecWarps * 32;

template <int HD>
struct DecCfg {
  static constexpr int STAGES = HD == 64 ? 6 : 3;         // blocks in flight per pair
  static constexpr int HALF = HD * 16 * 2;                // bytes of K (or V) of one block, one head
  static constexpr int SLOT = 2 * HALF;                   // K rows then V rows
  static constexpr int DPL = HD / 32;                     // head-dim columns per lane
  static constexpr int RING = kDecPairs * STAGES * SLOT;  // bytes
};

template <int HD>
constexpr int dec_smem_bytes() {
  return DecCfg<HD>::RING + 2 * kDecPairs * DecCfg<HD>::STAGES * 8 + 128;
}

__device__ __forceinline__ void bulk_load_1d(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// packed fp32 pair FMA: d = a * b + c elementwise (two registers as one operand)
__device__ __forceinline__ uint64_t f2fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ uint64_t f2(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}
__device__ __forceinline__ float2 f2u(uint64_t r) {
  float2 v;
  asm("mov.b64 {%0, %1}, %2;" : "=f"(v.x), "=f"(v.y) : "l"(r));
  return v;
}

__device__ __forceinline__ float ex2a(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// DPL fp16 values at p (DPL = 2 or 4, 4- or 8-byte aligned) as fp32
template <int DPL>
__device__ __forceinline__ void load_h(const uint16_t* p, float* f) {
  if constexpr (DPL == 4) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u.x));
    const float2 b = __half22float2(*reinterpret_cast<const __half2*>(&u.y));
    f[0] = a.x;
    f[1] = a.y;
    f[2] = b.x;
    f[3] = b.y;
  } else {
    const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
    const float2 a = __half22float2(*reinterpret_cast<const __half2*>(&u));
    f[0] = a.x;
    f[1] = a.y;
  }
}

// R = n * (hq / hkv) query rows per KV head, a template constant so that no
// instruction is spent on absent rows
template <int HD, int R>
__global__ void __launch_bounds__(kDecThreads, 1) attn_decode_kernel(
    const uint16_t* __restrict__ q, const int32_t* __restrict__ pos, int n, int hq, int hkv,
    const int32_t* __restrict__ table, int64_t n_logical, const uint16_t* __restrict__ pool,
    int64_t pool_blocks, uint16_t* __restrict__ out, float* __restrict__ part_o,
    float* __restrict__ part_lse, int blocks_per_split, int n_splits, float scale_log2,
    int32_t* status, const int32_t* __restrict__ flags, long long flag_wait_cycles,
    const uint16_t* __restrict__ host_pool, int64_t host_blocks) {
  using C = DecCfg<HD>;
  constexpr int DPL = C::DPL;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) &
                                             ~static_cast<uintptr_t>(127));
  uint8_t* ring = smem;                                          // [pair][stage] K rows, V rows
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + C::RING);  // [pair][stage] data landed
  uint64_t* empty = full + kDecPairs * C::STAGES;                // [pair][stage] both warps done
  __shared__ int s_maxpos;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int pair = warp >> 1, hk = warp & 1;  // hk: keys 8hk..8hk+7 of each block
  const int g = blockIdx.x, split = blockIdx.y;
  const int group = hq / hkv;
  // query row r of this KV head: token r / group, head g * group + r % group
  const int64_t blk_elems = static_cast<int64_t>(2) * hkv * 16 * HD;

  if (tid == 0) {
    s_maxpos = -1;
    for (int i = 0; i < kDecPairs * C::STAGES; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 2);  // one arrival per warp of the pair
    }
    fence_barrier_init();
  }
  // the prologue above touches no memory another kernel writes
  pdl_enter();
  __syncthreads();
  if (tid < n) atomicMax(&s_maxpos, pos[tid]);
  // this lane's head-dim columns of every q row, and every row's position
  float qv[R][DPL];
  int rpos[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int t = r / group, h = g * group + r % group;
    rpos[r] = pos[t];
    load_h<DPL>(q + (static_cast<int64_t>(t) * hq + h) * HD + lane * DPL, qv[r]);
  }
  __syncthreads();
  const int kv_len = s_maxpos + 1;
  const int nblk = (kv_len + 15) / 16;
  const int b_begin = split * blocks_per_split;
  const int b_end = min(nblk, b_begin + blocks_per_split);
  // this pair's blocks: b_begin + pair + kDecPairs * i, i < nb
  const int nb = b_end > b_begin + pair ? (b_end - b_begin - pair + kDecPairs - 1) / kDecPairs : 0;
  uint8_t* pring = ring + pair * C::STAGES * C::SLOT;
  uint64_t* pfull = full + pair * C::STAGES;
  uint64_t* pempty = empty + pair * C::STAGES;
  const bool issuer = hk == 0 && lane == 0;

  // physical blocks of this pair's blocks 32c .. 32c+31, one per lane (-1: none,
  // or a table entry outside the pool, which is flagged and its keys masked);
  // two windows, the current one and the next, so refills STAGES ahead find theirs
  auto load_tab = [&](int c) -> int32_t {
    const int i = 32 * c + lane;
    const int b = b_begin + pair + kDecPairs * i;
    if (i >= nb) return -1;
    if (b >= n_logical) {
      set_status(status, kStatusDevice);  // a key past the block table
      return -1;
    }
    const int32_t p = table[b];
    if (p >= 0 && p < pool_blocks) return p;
    // a swapped block read in place: entry -2 - slot of the pinned store
    if (host_pool != nullptr && p <= -2 && -static_cast<int64_t>(p) - 2 < host_blocks) return p;
    set_status(status, kStatusDevice);
    return -1;
  };
  int32_t tab_cur = load_tab(0), tab_nxt = load_tab(1);
  int win = 0;  // window of tab_cur
  auto phys = [&](int i) {
    return __shfl_sync(0xffffffffu, (i >> 5) == win ? tab_cur : tab_nxt, i & 31);
  };
  auto issue = [&](int i, int32_t p) {  // issuer lane, physical block p of block i
    const int s = i % C::STAGES;
    if (p == -1) {
      mbar_arrive(&pfull[s]);  // completes the phase with no data
      return;
    }
    if (p <= -2) {
      // in pinned host memory: the block's K and V rows of head g over the
      // host link with 16-byte cp.async (plain loads), tracked by the slot's
      // barrier, then this thread's own arrival
      const uint16_t* hb = host_pool + (-static_cast<int64_t>(p) - 2) * blk_elems;
      const uint16_t* ks = hb + static_cast<int64_t>(g) * 16 * HD;
      const uint16_t* vs = hb + static_cast<int64_t>(hkv + g) * 16 * HD;
      const uint32_t dk = smem_u32(pring + s * C::SLOT), dv = dk + C::HALF;
#pragma unroll 4
      for (int c = 0; c < C::HALF / 16; ++c) {
        cp_async16(dk + c * 16, ks + c * 8);
        cp_async16(dv + c * 16, vs + c * 8);
      }
      cp_async_mbar_arrive(&pfull[s]);
      mbar_arrive(&pfull[s]);
      return;
    }
    if (flags != nullptr) {
      // a restore copy into this block may still be in flight: wait (bounded)
      // for its residency flag; on a timeout the status word says so and the
      // phase completes with no data
      if (!flag_wait(flags, p, status, flag_wait_cycles)) {
        mbar_arrive(&pfull[s]);
        return;
      }
      fence_proxy_async_global();
    }
    fence_proxy_async_smem();  // earlier generic reads of the slot before the async writes
    mbar_arrive_expect_tx(&pfull[s], C::SLOT);
    const uint16_t* blk = pool + static_cast<int64_t>(p) * blk_elems;
    bulk_load_1d(pring + s * C::SLOT, blk + static_cast<int64_t>(g) * 16 * HD, C::HALF, &pfull[s]);
    bulk_load_1d(pring + s * C::SLOT + C::HALF, blk + static_cast<int64_t>(hkv + g) * 16 * HD, C::HALF,
                 &pfull[s]);
  };

  // per row: reference maximum m (raised only when a score exceeds it by more
  // than 2^8, so every weight stays <= 256), this lane's share of the weight
  // sum l, and its output columns as packed pairs
  float m[R], l[R];
  uint64_t o2[R][DPL / 2];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    m[r] = -INFINITY;
    l[r] = 0.0f;
#pragma unroll
    for (int j = 0; j < DPL / 2; ++j) o2[r][j] = f2(0.0f, 0.0f);
  }
  const int x = (lane >> 2) & 7;  // key (of this warp's 8) whose score this lane ends up with
  {
    const int np = nb < C::STAGES ? nb : C::STAGES;
    for (int i = 0; i < np; ++i) {
      const int32_t p = phys(i);
      if (issuer) issue(i, p);
    }
  }
  int done = 0;  // blocks consumed
  bool ok = true;
  for (int i = 0; i < nb; ++i) {
    const int s = i % C::STAGES;
    if (i > 0 && (i & 31) == 0) {
      tab_cur = tab_nxt;
      win = i >> 5;
      tab_nxt = load_tab(win + 1);
    }
    const int32_t pblk = phys(i);
    const bool got = mbar_wait(&pfull[s], (i / C::STAGES) & 1, status, kWaitCycles);
    if (!__all_sync(0xffffffffu, got)) {  // the warp leaves together
      ok = false;
      break;
    }
    done = i + 1;
    const int b = b_begin + pair + kDecPairs * i;
    const bool valid = pblk != -1;  // in the pool, or in host memory (<= -2)
    const uint16_t* kh = reinterpret_cast<const uint16_t*>(pring + s * C::SLOT) + (8 * hk) * HD + lane * DPL;
    const uint16_t* vh = reinterpret_cast<const uint16_t*>(pring + s * C::SLOT + C::HALF) + (8 * hk) * HD +
                         lane * DPL;
    if (valid) {
      // ---- scores: partial dot of key (j ^ x) in slot j, then the butterfly ----
      float part[R][8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        float kf[DPL];
        load_h<DPL>(kh + (j ^ x) * HD, kf);
#pragma unroll
        for (int r = 0; r < R; ++r) {
          float acc = 0.0f;
#pragma unroll
          for (int d = 0; d < DPL; ++d) acc = fmaf(qv[r][d], kf[d], acc);
          part[r][j] = acc;
        }
      }
      const int key = b * 16 + 8 * hk + x;
      float p[R];
#pragma unroll
      for (int r = 0; r < R; ++r) {
#pragma unroll
        for (int j = 0; j < 4; ++j) part[r][j] += __shfl_xor_sync(0xffffffffu, part[r][j + 4], 16);
#pragma unroll
        for (int j = 0; j < 2; ++j) part[r][j] += __shfl_xor_sync(0xffffffffu, part[r][j + 2], 8);
        float sc = part[r][0] + __shfl_xor_sync(0xffffffffu, part[r][1], 4);
        sc += __shfl_xor_sync(0xffffffffu, sc, 2);
        sc += __shfl_xor_sync(0xffffffffu, sc, 1);
        p[r] = (key <= rpos[r] && key < kv_len) ? sc * scale_log2 : -INFINITY;
      }
      // ---- online softmax per row (lazy rebase of the reference maximum) ----
#pragma unroll
      for (int r = 0; r < R; ++r) {
        float tmax = p[r];
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 4));
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 8));
        tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, 16));
        if (tmax > m[r] + 8.0f) {  // warp-uniform; also the first finite maximum
          const float alpha = ex2a(m[r] - tmax);  // 0 while m is -inf
          l[r] *= alpha;
          const uint64_t a2 = f2(alpha, alpha), z2 = f2(0.0f, 0.0f);
#pragma unroll
          for (int j = 0; j < DPL / 2; ++j) o2[r][j] = f2fma(o2[r][j], a2, z2);
          m[r] = tmax;
        }
        // a row with no key yet keeps weight 0 (and no NaN from -inf - -inf)
        p[r] = m[r] == -INFINITY ? 0.0f : ex2a(p[r] - m[r]);
        if ((lane & 3) == 0) l[r] += p[r];
      }
      // ---- P V ----
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) {
        float vf[DPL];
        load_h<DPL>(vh + kk * HD, vf);
#pragma unroll
        for (int r = 0; r < R; ++r) {
          const float pk = __shfl_sync(0xffffffffu, p[r], 4 * kk);
          const uint64_t pk2 = f2(pk, pk);
#pragma unroll
          for (int j = 0; j < DPL / 2; ++j) o2[r][j] = f2fma(pk2, f2(vf[2 * j], vf[2 * j + 1]), o2[r][j]);
        }
      }
    }
    __syncwarp();  // every lane of this warp is done with the slot
    if (lane == 0) mbar_arrive(&pempty[s]);
    if (i + C::STAGES < nb) {
      const int32_t pn = phys(i + C::STAGES);
      if (issuer) {
        // both warps released the slot before it is refilled
        if (mbar_wait(&pempty[s], (i / C::STAGES) & 1, status, kWaitCycles)) issue(i + C::STAGES, pn);
      }
    }
  }
  if (!ok && issuer) {
    // copies still in flight land before the CTA's shared memory is released
    for (int i = done; i < nb && i < done + C::STAGES; ++i)
      mbar_wait(&pfull[i % C::STAGES], (i / C::STAGES) & 1, status, kWaitCycles);
  }
#pragma unroll
  for (int r = 0; r < R; ++r) {
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) l[r] += __shfl_xor_sync(0xffffffffu, l[r], off);
  }
  __syncthreads();  // the rings are free: merge the warps' partials there
  float* wm = reinterpret_cast<float*>(ring);  // [warp][R]
  float* wl = wm + kDecWarps * R;              // [warp][R]
  float* wo = wl + kDecWarps * R;              // [warp][R][HD]
#pragma unroll
  for (int r = 0; r < R; ++r) {
    if (lane == 0) {
      wm[warp * R + r] = m[r];
      wl[warp * R + r] = l[r];
    }
#pragma unroll
    for (int j = 0; j < DPL / 2; ++j) {
      const float2 v = f2u(o2[r][j]);
      wo[(warp * R + r) * HD + lane * DPL + 2 * j] = v.x;
      wo[(warp * R + r) * HD + lane * DPL + 2 * j + 1] = v.y;
    }
  }
  __syncthreads();
  for (int idx = tid; idx < R * HD; idx += kDecThreads) {
    const int r = idx / HD, d = idx % HD;
    float M = -INFINITY;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) M = fmaxf(M, wm[w * R + r]);
    float L = 0.0f, O = 0.0f;
    if (M != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) {
        const float mw = wm[w * R + r];
        if (mw == -INFINITY) continue;
        const float sw = ex2a(mw - M);
        L += sw * wl[w * R + r];
        O += sw * wo[(w * R + r) * HD + d];
      }
    }
    const float on = L > 0.0f ? O / L : 0.0f;
    const int t = r / group, h = g * group + r % group;
    const int64_t row = static_cast<int64_t>(t) * hq + h;
    if (n_splits == 1) {
      out[row * HD + d] = __half_as_ushort(__float2half_rn(on));
    } else {
      part_o[(static_cast<int64_t>(split) * n * hq + row) * HD + d] = on;
      if (d == 0) part_lse[static_cast<int64_t>(split) * n * hq + row] = L > 0.0f ? M + log2f(L) : -INFINITY;
    }
  }
}

template <int HD, int R>
cudaError_t launch_dec(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq, int32_t hkv,
                       const int32_t* table, int64_t n_logical, const void* pool, int64_t pool_blocks,
                       uint16_t* out, float* part_o, float* part_lse, int n_splits, int blocks_per_split,
                       int32_t* status, const int32_t* flags, long long flag_wait,
                       const uint16_t* host_pool, int64_t host_blocks, cudaStream_t st) {
  constexpr int SMEM = dec_smem_bytes<HD>();
  static_assert(SMEM <= 232448, "shared memory of one CTA");
  static_assert(kDecWarps * R * (HD + 2) * 4 <= DecCfg<HD>::RING, "warp partials fit in the rings");
  static_assert(DecCfg<HD>::STAGES < 32, "refills stay inside the 32-block table window");
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(attn_decode_kernel<HD, R>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    SMEM);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const float scale_log2 = static_cast<float>(1.0 / std::sqrt(static_cast<double>(HD)) * 1.4426950408889634);
  dim3 grid(static_cast<unsigned>(hkv), static_cast<unsigned>(n_splits));
  launch_k(attn_decode_kernel<HD, R>, dim3(grid), dim3(kDecThreads), SMEM, st,
      q, pos, static_cast<int>(n), hq, hkv, table, n_logical, static_cast<const uint16_t*>(pool), pool_blocks,
      out, part_o, part_lse, blocks_per_split, n_splits, scale_log2, status, flags, flag_wait, host_pool,
      host_blocks);
  return cudaGetLastError();
}

}  // namespace

bool attention_decode_applies(int64_t n, int32_t hq, int32_t hkv, int32_t hd) {
  return n >= 1 && hkv > 0 && hq % hkv == 0 && (hd == 64 || hd == 128) &&
         n * (hq / hkv) <= kAttnDecodeMaxRows;
}

void attention_decode_split(int32_t hkv, int64_t max_keys, int num_sms, int* n_splits, int* keys_per_split) {
  // one CTA per SM: hkv x splits CTAs, and at least one block per warp per split
  const int64_t nblk = std::max<int64_t>(1, (max_keys + 15) / 16);
  int64_t s = std::max<int64_t>(1, num_sms / std::max(1, hkv));
  s = std::min<int64_t>(s, std::max<int64_t>(1, nblk / kDecWarps));
  s = std::min<int64_t>(s, 64);
  const int64_t per = (nblk + s - 1) / s;
  *n_splits = static_cast<int>((nblk + per - 1) / per);
  *keys_per_split = static_cast<int>(per * 16);
}

cudaError_t launch_attention_decode(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq, int32_t hkv,
                                    int32_t hd, const int32_t* table, int64_t n_logical, const void* pool,
                                    int64_t pool_blocks, uint16_t* out, float* part_o, float* part_lse,
                                    int n_splits, int keys_per_split, int32_t* status,
                                    const int32_t* flags, long long flag_wait, const uint16_t* host_pool,
                                    int64_t host_blocks, cudaStream_t st) {
  if (!attention_decode_applies(n, hq, hkv, hd) || keys_per_split % 16 != 0 ||
      reinterpret_cast<uintptr_t>(pool) % 16 != 0)  // bulk copies start on 16-byte boundaries
    return cudaErrorInvalidValue;
  const int bps = keys_per_split / 16;
  const int64_t R = n * (hq / hkv);
  static_assert(kAttnDecodeMaxRows == 4, "instances for 1 to 4 rows");
#define MZC_DEC_CASE(HDV, RV)                                                                              \
  if (hd == HDV && R == RV)                                                                                \
    return launch_dec<HDV, RV>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks, out, part_o, part_lse, \
                               n_splits, bps, status, flags, flag_wait, host_pool, host_blocks, st);
  MZC_DEC_CASE(64, 1)
  MZC_DEC_CASE(64, 2)
  MZC_DEC_CASE(64, 3)
  MZC_DEC_CASE(64, 4)
  MZC_DEC_CASE(128, 1)
  MZC_DEC_CASE(128, 2)
  MZC_DEC_CASE(128, 3)
  MZC_DEC_CASE(128, 4)
#undef MZC_DEC_CASE
  return cudaErrorInvalidValue;
}

}  // namespace mzc
