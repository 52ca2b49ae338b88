// Projections of a few hundred rows (a short prompt), where the GEMM is bound
// by streaming the weights: C[m][n] = A[m][k] W[n][k]^T with m <= 256.
//
// With 128 x BN tiles over N alone, an O or down projection (n = 3072) has
// 24-48 tiles, so only that many SMs pull weight bytes, and at narrow BN the
// shared activation tiles make up most of every SM's traffic.  Here the K
// range is split as well, over the S CTAs of a thread-block cluster
// (grid = S x N tiles of 128 columns):
//   - CTA s of the cluster accumulates its k-blocks [s*nkb/S, (s+1)*nkb/S) of
//     the 128-column tile for all (one or two) 128-row M tiles into TMEM, with
//     the same TMA ring / single-thread tcgen05.mma / commit pipeline as the
//     persistent GEMM;
//   - the epilogue warps copy the fp32 partial to shared memory (the ring is
//     free by then) and the cluster synchronises;
//   - CTA s then sums rows [s*RS, (s+1)*RS) of the S partials, read through
//     distributed shared memory in split order (the same sum on every run;
//     all threads, several row chunks' loads in flight per thread), applies
//     the epilogue (fp16 store, fp32 residual add, SwiGLU) and writes the
//     rows out; a second cluster barrier keeps every partial alive until all
//     CTAs have read it.
// Folded RMSNorm (RowNorm): the residual-add form also writes h = fp16(x * g)
// and each row's sum of x^2 over the tile (one warp holds a row's 128 columns
// in the reduction, so a shuffle tree sums them); the fp16-store and SwiGLU
// forms scale each row by its rstd, which the epilogue warps compute from
// those sums while the main loop runs.
// EPI_QKV_ROPE (the QKV projection of a short row set): the summed rows go
// through the rotary embedding and the KV-block write in the reduction, so
// no separate rotary launch and no fp16 QKV round trip.  A warp holds a row's
// 128 columns, i.e. whole heads (hd 64 or 128), so the other half of each
// rotary pair comes from lane ^ (hd / 8) by shuffle.
// Every thread of every CTA passes both cluster barriers exactly once (no
// early exit on any path); the pipeline waits are bounded as elsewhere.
#include <algorithm>
#include <climits>
#include <mutex>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {

constexpr int SBM = 128, SBN = 128, SBK = 64;
// row chunks whose remote loads each thread has in flight in the reduction
#ifndef MZC_SK_ITEMS
#define MZC_SK_ITEMS 2
#endif

template <int MT>
struct SKCfg {
  static constexpr int STAGES = MT == 1 ? 6 : 4;
  static constexpr int A_BYTES = SBM * SBK * 2;  // one M tile's k-block
  static constexpr int B_BYTES = SBN * SBK * 2;
  static constexpr int STAGE_BYTES = MT * A_BYTES + B_BYTES;
  static constexpr int RING = STAGES * STAGE_BYTES;
  static constexpr int PART_BYTES = MT * SBM * SBN * 4;  // fp32 partial, reuses the ring
  static constexpr int OFF_BAR = RING;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr uint32_t TMEM_COLS = MT * SBN;
  static_assert(PART_BYTES <= RING, "the partial fits in the ring");
  static_assert(2 * STAGES * 8 + 8 <= 256, "barriers");
};

__device__ __forceinline__ bool skwait(uint64_t* bar, uint32_t parity, int32_t* status, volatile int* abort) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      set_status(status, kStatusTimeout);
      *abort = 1;
      return false;
    }
  }
}

__device__ __forceinline__ float silu_s(float g) { return g / (1.0f + __expf(-g)); }

__device__ __forceinline__ uint2 pack4_f16(float a, float b, float c, float d) {
  return make_uint2(pack2<true>(a, b), pack2<true>(c, d));
}

__device__ __forceinline__ float bf16_round(float x) { return __bfloat162float(__float2bfloat16_rn(x)); }

// marks a row whose position lies outside the rotary tables and the block
// table (no block-table entry takes this value: entries are blocks >= 0, -1
// for none, -2 - i for host block i)
constexpr int kNoPos = INT_MIN;

// Partial layout: row r (0 .. MT*128) of 32 float4 chunks, chunk c stored at
// c ^ (r & 7) so that eight lanes writing one chunk of eight rows hit eight
// different bank groups.
__device__ __forceinline__ uint32_t part_off(int r, int c) {
  return static_cast<uint32_t>((r * 32 + (c ^ (r & 7))) * 16);
}

template <int MT, int EPI>
__global__ void __launch_bounds__(192, 1) gemm_splitk_kernel(
    const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmw, void* __restrict__ out,
    int m, int n, int k, int32_t* status, const RowNorm rn, const RopeKV rk) {
  using C = SKCfg<MT>;
  constexpr int STAGES = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ float s_rs[MT * SBM];  // folded RMSNorm: rstd of rows r_begin ..
  // EPI_QKV_ROPE: position and physical block of rows r_begin .. (kNoPos:
  // the position is outside the rotary tables and the block table)
  __shared__ int s_pos[MT * SBM], s_phys[MT * SBM];
  volatile int* abort_flag = &s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = static_cast<int>(cluster_size()), s = static_cast<int>(cluster_rank());
  const int nt = blockIdx.y;
  const int nkb = (k + SBK - 1) / SBK;
  const int kb0 = static_cast<int>(static_cast<int64_t>(s) * nkb / S);
  const int kb1 = static_cast<int>(static_cast<int64_t>(s + 1) * nkb / S);
  // the output rows this CTA sums and writes: [r_begin, r_end)
  const int rows = min(MT * SBM, m);
  const int RS = (rows + S - 1) / S;
  const int r_begin = s * RS, r_end = min(rows, r_begin + RS);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tma);
    tma_prefetch_desc(&tmw);
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(acc_full, 1);
    fence_barrier_init();
    s_abort = 0;
  }
  if (warp == 1) tmem_alloc(&s_tmem, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // The prologue above touches no memory another kernel writes.  Neither do
  // the weights: the producer issues the first stages' W loads before it waits
  // for the previous kernel (whose output A is), so weight streaming starts
  // under that kernel's tail.
  const int pre = (warp == 0 && lane == 0) ? min(STAGES, kb1 - kb0) : 0;
  for (int i = 0; i < pre; ++i) {
    mbar_arrive_expect_tx(&full[i], C::STAGE_BYTES);
    tma_load_2d(smem + i * C::STAGE_BYTES + MT * C::A_BYTES, &tmw, &full[i], (kb0 + i) * SBK, nt * SBN);
  }
  pdl_enter();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer: the split's k-blocks, every M tile and the W tile ----
      bool ok = true;
      int it = 0;
      for (int kb = kb0; ok && kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (it >= STAGES && !skwait(&empty[st], ((it / STAGES) - 1) & 1, status, abort_flag)) {
          ok = false;
          break;
        }
        uint8_t* base = smem + st * C::STAGE_BYTES;
        if (it >= pre) mbar_arrive_expect_tx(&full[st], C::STAGE_BYTES);  // else done above
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) tma_load_2d(base + mt * C::A_BYTES, &tma, &full[st], kb * SBK, mt * SBM);
        if (it >= pre) tma_load_2d(base + MT * C::A_BYTES, &tmw, &full[st], kb * SBK, nt * SBN);
      }
      // every fill issued has landed before the ring is reused for the partial
      for (int i = it - STAGES < 0 ? 0 : it - STAGES; i < it; ++i)
        skwait(&full[i % STAGES], (i / STAGES) & 1, status, abort_flag);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- UMMA issuer: accumulator of M tile mt at TMEM columns mt*128 ----
      constexpr uint32_t idesc = idesc_f16_f32(SBM, SBN);
      bool ok = true;
      int it = 0;
      for (int kb = kb0; ok && kb < kb1; ++kb, ++it) {
        const int st = it % STAGES;
        if (!skwait(&full[st], (it / STAGES) & 1, status, abort_flag)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t base = smem_u32(smem + st * C::STAGE_BYTES);
        const uint64_t bd = sdesc_k_sw128(base + MT * C::A_BYTES);
#pragma unroll
        for (int mt = 0; mt < MT; ++mt) {
          const uint64_t ad = sdesc_k_sw128(base + mt * C::A_BYTES);
#pragma unroll
          for (int kk = 0; kk < SBK / 16; ++kk)
            umma_f16(tmem + mt * SBN, ad + 2 * kk, bd + 2 * kk, idesc, (it | kk) != 0 ? 1u : 0u);
        }
        umma_commit(&empty[st]);
      }
      umma_commit(acc_full);  // all of this thread's UMMAs (none for an empty split)
    }
    __syncwarp();
  } else {
    // ---- epilogue warps 2-5: TMEM accumulator -> shared-memory partial ----
    const int q = warp & 3;  // TMEM lane quarter: rows q*32 .. q*32+31 of each M tile
    if constexpr (EPI != EPI_ADD_F32) {
      // folded RMSNorm: the rows' rstd while the main loop runs (the sums of
      // squares come from the previous kernel, complete after pdl_enter)
      if (rn.ss != nullptr)
        for (int i = threadIdx.x - 64; r_begin + i < r_end; i += 128)
          s_rs[i] = row_rstd(rn.ss, rn.nt, rn.d, rn.eps, r_begin + i);
    }
    if constexpr (EPI == EPI_QKV_ROPE) {
      // the rows' positions and KV blocks, looked up while the main loop runs
      for (int i = threadIdx.x - 64; r_begin + i < r_end; i += 128) {
        const int p = rk.pos[r_begin + i];
        int ph = kNoPos;
        if (p >= 0 && (p >> 4) < rk.n_logical) ph = rk.table[p >> 4];
        s_pos[i] = p;
        s_phys[i] = ph;
      }
    }
    bool ok = skwait(acc_full, 0, status, abort_flag);
    __syncwarp();
    ok = __all_sync(0xffffffffu, ok);
    tc_fence_after();
    const bool have = ok && kb1 > kb0;
#pragma unroll 1
    for (int mt = 0; mt < MT; ++mt) {
      const int r = mt * SBM + q * 32 + lane;
      const uint32_t trow = tmem + mt * SBN + (static_cast<uint32_t>(q * 32) << 16);
#pragma unroll 1
      for (int c = 0; c < SBN; c += 32) {
        float v[32];
        if (have) {
          tmem_ld32w(trow + c, v);
        } else {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] = 0.0f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<float4*>(smem + part_off(r, c / 4 + u)) =
              make_float4(v[4 * u], v[4 * u + 1], v[4 * u + 2], v[4 * u + 3]);
      }
    }
    tc_fence_before();
  }

  // ---- every partial of the cluster is in shared memory ----
  cluster_sync_all();

  {
    // ---- rows [s*RS, (s+1)*RS) summed over the S partials in split order
    // (the same sum on every run), by all 192 threads.  Each thread issues
    // the remote loads (and residual reads) of ITEMS row chunks before it
    // sums any of them: one chunk at a time left every thread waiting out
    // the distributed-shared-memory latency once per chunk ----
    const uint32_t part = smem_u32(smem);
    constexpr int CH = EPI == EPI_SWIGLU_BF16 ? 16 : 32;  // float4 chunks handled per row
    constexpr int ITEMS = EPI == EPI_SWIGLU_BF16 ? 2 : MZC_SK_ITEMS;
    const int n_items = max(0, r_end - r_begin) * CH;
    float amax = 0.0f;  // largest |value| this thread stores as fp16
    const bool norm_out = EPI == EPI_ADD_F32 && rn.h != nullptr;
    const bool norm_in = EPI != EPI_ADD_F32 && rn.ss != nullptr;
    for (int i0 = threadIdx.x; i0 < n_items; i0 += ITEMS * 192) {
      float4 v[ITEMS][8], u[ITEMS][8], x[ITEMS], gv[ITEMS], rc[ITEMS], rsn[ITEMS];
#pragma unroll
      for (int h = 0; h < ITEMS; ++h) {
        const int idx = i0 + h * 192;
        if (idx < n_items) {
          const int r = r_begin + idx / CH, c = idx % CH;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            if (j < S) {
              v[h][j] = ld_cluster_f4(map_rank(part + part_off(r, c), j));
              if constexpr (EPI == EPI_SWIGLU_BF16) u[h][j] = ld_cluster_f4(map_rank(part + part_off(r, c + 16), j));
            }
          }
          if constexpr (EPI == EPI_ADD_F32) {
            const int col = nt * SBN + c * 4;
            if (col < n) {
              x[h] = *reinterpret_cast<const float4*>(static_cast<const float*>(out) + static_cast<int64_t>(r) * n + col);
              if (norm_out) gv[h] = *reinterpret_cast<const float4*>(rn.g + col);
            }
          }
          if constexpr (EPI == EPI_QKV_ROPE) {
            // the rotary angles of q and k columns, loaded with the partials
            const int col = nt * SBN + c * 4;
            const int head = col / rk.hd, e = col - head * rk.hd, half = rk.hd >> 1;
            const int p = s_pos[r - r_begin];
            if (head < rk.hq + rk.hkv && s_phys[r - r_begin] != kNoPos) {
              const int64_t t = static_cast<int64_t>(p) * half + (e < half ? e : e - half);
              rc[h] = *reinterpret_cast<const float4*>(rk.cos_t + t);
              rsn[h] = *reinterpret_cast<const float4*>(rk.sin_t + t);
            }
          }
        }
      }
#pragma unroll
      for (int h = 0; h < ITEMS; ++h) {
        const int idx = i0 + h * 192;
        if (idx >= n_items) continue;
        const int r = r_begin + idx / CH, c = idx % CH;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f), acc2 = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          if (j < S) {
            acc.x += v[h][j].x;
            acc.y += v[h][j].y;
            acc.z += v[h][j].z;
            acc.w += v[h][j].w;
            if constexpr (EPI == EPI_SWIGLU_BF16) {
              acc2.x += u[h][j].x;
              acc2.y += u[h][j].y;
              acc2.z += u[h][j].z;
              acc2.w += u[h][j].w;
            }
          }
        }
        if (norm_in) {
          const float rs = s_rs[r - r_begin];
          acc.x *= rs;
          acc.y *= rs;
          acc.z *= rs;
          acc.w *= rs;
          acc2.x *= rs;
          acc2.y *= rs;
          acc2.z *= rs;
          acc2.w *= rs;
        }
        if constexpr (EPI == EPI_QKV_ROPE) {
          // every lane of the warp is here (n_items is a multiple of 32, and
          // a warp's items are one row): the rotary partner by shuffle first
          const int pl = rk.hd >> 3;  // chunks between the two halves of a pair
          float4 pr;
          pr.x = __shfl_xor_sync(0xffffffffu, acc.x, pl);
          pr.y = __shfl_xor_sync(0xffffffffu, acc.y, pl);
          pr.z = __shfl_xor_sync(0xffffffffu, acc.z, pl);
          pr.w = __shfl_xor_sync(0xffffffffu, acc.w, pl);
          const int col = nt * SBN + c * 4;
          const int head = col / rk.hd, e = col - head * rk.hd, half = rk.hd >> 1;
          const int p = s_pos[r - r_begin], phys = s_phys[r - r_begin];
          if (phys == kNoPos) {
            set_status(status, kStatusDevice);  // outside the rotary tables and the block table
          } else {
            float y0 = acc.x, y1 = acc.y, y2 = acc.z, y3 = acc.w;
            if (head < rk.hq + rk.hkv) {
              const float4 cs = rc[h], sn = rsn[h];
              const float sg = e < half ? -1.0f : 1.0f;  // x1 c - x2 s, or x2 c + x1 s
              y0 = acc.x * cs.x + sg * (pr.x * sn.x);
              y1 = acc.y * cs.y + sg * (pr.y * sn.y);
              y2 = acc.z * cs.z + sg * (pr.z * sn.z);
              y3 = acc.w * cs.w + sg * (pr.w * sn.w);
            }
            uint16_t* dst = nullptr;
            if (head < rk.hq) {
              dst = rk.q_out + (static_cast<int64_t>(r) * rk.hq + head) * rk.hd + e;
            } else {
              if (phys < 0 || phys >= rk.pool_blocks) {
                set_status(status, kStatusDevice);
              } else {
                if (!rk.f16kv) {
                  y0 = bf16_round(y0);
                  y1 = bf16_round(y1);
                  y2 = bf16_round(y2);
                  y3 = bf16_round(y3);
                }
                // K heads then V heads: head - hq indexes [2 hkv][16][hd] of the block
                dst = rk.pool + static_cast<int64_t>(phys) * (2LL * rk.hkv * 16 * rk.hd) +
                      (static_cast<int64_t>(head - rk.hq) * 16 + (p & 15)) * rk.hd + e;
              }
            }
            if (dst != nullptr) {
              amax = fmaxf(amax, fmaxf(fmaxf(fabsf(y0), fabsf(y1)), fmaxf(fabsf(y2), fabsf(y3))));
              *reinterpret_cast<uint2*>(dst) = pack4_f16(y0, y1, y2, y3);
            }
          }
        } else if constexpr (EPI == EPI_STORE_BF16) {
          const int col = nt * SBN + c * 4;
          if (col < n) {
            amax = fmaxf(amax, fmaxf(fmaxf(fabsf(acc.x), fabsf(acc.y)), fmaxf(fabsf(acc.z), fabsf(acc.w))));
            *reinterpret_cast<uint2*>(static_cast<uint16_t*>(out) + static_cast<int64_t>(r) * n + col) =
                pack4_f16(acc.x, acc.y, acc.z, acc.w);
          }
        } else if constexpr (EPI == EPI_ADD_F32) {
          const int col = nt * SBN + c * 4;
          if (col < n) {
            float4 y = x[h];
            y.x += acc.x;
            y.y += acc.y;
            y.z += acc.z;
            y.w += acc.w;
            *reinterpret_cast<float4*>(static_cast<float*>(out) + static_cast<int64_t>(r) * n + col) = y;
            if (norm_out) {
              // the warp holds the row's 128 columns of this tile (CH = 32
              // chunks, n a multiple of 128): h = fp16(x * g) and the tile's
              // sum of x^2 for the consumer's rstd
              const float h0 = y.x * gv[h].x, h1 = y.y * gv[h].y, h2 = y.z * gv[h].z, h3 = y.w * gv[h].w;
              amax = fmaxf(amax, fmaxf(fmaxf(fabsf(h0), fabsf(h1)), fmaxf(fabsf(h2), fabsf(h3))));
              *reinterpret_cast<uint2*>(rn.h + static_cast<int64_t>(r) * n + col) = pack4_f16(h0, h1, h2, h3);
              float sq = y.x * y.x + y.y * y.y + y.z * y.z + y.w * y.w;
#pragma unroll
              for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
              if (lane == 0) rn.ss[static_cast<int64_t>(r) * rn.nt + nt] = sq;
            }
          }
        } else {
          // gate columns 0..63 of the tile pair with up columns 64..127
          const int col = nt * (SBN / 2) + c * 4;
          if (col < n / 2) {
            const float y0 = silu_s(acc.x) * acc2.x, y1 = silu_s(acc.y) * acc2.y;
            const float y2 = silu_s(acc.z) * acc2.z, y3 = silu_s(acc.w) * acc2.w;
            amax = fmaxf(amax, fmaxf(fmaxf(fabsf(y0), fabsf(y1)), fmaxf(fabsf(y2), fabsf(y3))));
            *reinterpret_cast<uint2*>(static_cast<uint16_t*>(out) + static_cast<int64_t>(r) * (n / 2) + col) =
                pack4_f16(y0, y1, y2, y3);
          }
        }
      }
    }
    if (EPI != EPI_ADD_F32 || norm_out) note_f16_overflow(status, amax);
  }

  // ---- no CTA leaves while another may still read its partial ----
  __syncwarp();
  cluster_sync_all();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int MT, int EPI>
cudaError_t launch_sk(const CUtensorMap& ta, const CUtensorMap& tw128, void* out, int64_t m, int64_t n, int64_t k,
                      int S, int32_t* status, cudaStream_t st, const RowNorm& rn, const RopeKV& rk) {
  using C = SKCfg<MT>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(gemm_splitk_kernel<MT, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    C::SMEM);
  });
  if (attr_err != cudaSuccess) return attr_err;
  const int num_n = static_cast<int>((n + SBN - 1) / SBN);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(S), static_cast<unsigned>(num_n), 1);
  cfg.blockDim = dim3(192, 1, 1);
  cfg.dynamicSmemBytes = C::SMEM;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(S);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, gemm_splitk_kernel<MT, EPI>, ta, tw128, out, static_cast<int>(m),
                            static_cast<int>(n), static_cast<int>(k), status, rn, rk);
}

// The largest cluster size S <= 8 whose S x num_n CTAs are all resident at
// once (one wave), from the occupancy query for this kernel; 1 if none.
template <int MT, int EPI>
int pick_splits(int num_n, int num_sms) {
  using C = SKCfg<MT>;
  static std::once_flag once;
  static int max_clusters[9] = {};
  std::call_once(once, [] {
    if (cudaFuncSetAttribute(gemm_splitk_kernel<MT, EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) !=
        cudaSuccess)
      return;
    for (int sz = 2; sz <= 8; ++sz) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(static_cast<unsigned>(sz), 1, 1);
      cfg.blockDim = dim3(192, 1, 1);
      cfg.dynamicSmemBytes = C::SMEM;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = static_cast<unsigned>(sz);
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int count = 0;
      if (cudaOccupancyMaxActiveClusters(&count, gemm_splitk_kernel<MT, EPI>, &cfg) == cudaSuccess)
        max_clusters[sz] = count;
    }
    cudaGetLastError();  // a refused query leaves no error behind
  });
  for (int sz = std::min(8, num_sms / std::max(1, num_n)); sz >= 2; --sz)
    if (max_clusters[sz] >= num_n) return sz;
  return 1;
}

}  // namespace

cudaError_t launch_gemm_splitk(const CUtensorMap& ta, const GemmWeight& w, void* out, int64_t m, int64_t n,
                               int64_t k, int epilogue, int num_sms, int32_t* status, cudaStream_t st,
                               bool* launched, const RowNorm* rn, const RopeKV* rk) {
  *launched = false;
  if (m <= 0 || m > 2 * SBM || n % SBN != 0 || k % 8 != 0) return cudaSuccess;
  const int num_n = static_cast<int>(n / SBN);
  const bool two = m > SBM;
  const RowNorm norm = rn != nullptr ? *rn : RowNorm{};
  const RopeKV rope = rk != nullptr ? *rk : RopeKV{};
  if (epilogue == EPI_QKV_ROPE &&
      (rk == nullptr || (rope.hd != 64 && rope.hd != 128) || static_cast<int64_t>(rope.hq + 2 * rope.hkv) * rope.hd != n ||
       rope.pos == nullptr || rope.cos_t == nullptr || rope.sin_t == nullptr || rope.table == nullptr ||
       rope.pool == nullptr || rope.q_out == nullptr))
    return cudaErrorInvalidValue;
#define MZC_SK(MTV, EPIV)                                                                   \
  {                                                                                        \
    const int S = pick_splits<MTV, EPIV>(num_n, num_sms);                                  \
    if (S < 2) return cudaSuccess;                                                         \
    *launched = true;                                                                      \
    return launch_sk<MTV, EPIV>(ta, w.box128, out, m, n, k, S, status, st, norm, rope);    \
  }
  switch (epilogue) {
    case EPI_STORE_BF16:
      if (two) MZC_SK(2, EPI_STORE_BF16) else MZC_SK(1, EPI_STORE_BF16)
    case EPI_ADD_F32:
      if (two) MZC_SK(2, EPI_ADD_F32) else MZC_SK(1, EPI_ADD_F32)
    case EPI_SWIGLU_BF16:
      if (two) MZC_SK(2, EPI_SWIGLU_BF16) else MZC_SK(1, EPI_SWIGLU_BF16)
    case EPI_QKV_ROPE:
      if (two) MZC_SK(2, EPI_QKV_ROPE) else MZC_SK(1, EPI_QKV_ROPE)
    default:
      return cudaErrorInvalidValue;
  }
#undef MZC_SK
}

bool gemm_splitk_launches(int64_t m, int64_t n, int64_t k, int epilogue, int num_sms) {
  if (m <= 0 || m > 2 * SBM || n % SBN != 0 || k % 8 != 0) return false;
  const int num_n = static_cast<int>(n / SBN);
  const bool two = m > SBM;
  switch (epilogue) {
    case EPI_STORE_BF16:
      return (two ? pick_splits<2, EPI_STORE_BF16>(num_n, num_sms) : pick_splits<1, EPI_STORE_BF16>(num_n, num_sms)) >= 2;
    case EPI_ADD_F32:
      return (two ? pick_splits<2, EPI_ADD_F32>(num_n, num_sms) : pick_splits<1, EPI_ADD_F32>(num_n, num_sms)) >= 2;
    case EPI_SWIGLU_BF16:
      return (two ? pick_splits<2, EPI_SWIGLU_BF16>(num_n, num_sms) : pick_splits<1, EPI_SWIGLU_BF16>(num_n, num_sms)) >= 2;
    case EPI_QKV_ROPE:
      return (two ? pick_splits<2, EPI_QKV_ROPE>(num_n, num_sms) : pick_splits<1, EPI_QKV_ROPE>(num_n, num_sms)) >= 2;
    default:
      return false;
  }
}

}  // namespace mzc
