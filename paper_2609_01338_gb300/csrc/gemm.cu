// FP16 GEMM on the 5th-generation tensor cores: C[m][n] = A[m][k] W[n][k]^T,
// fp32 accumulation.  (fp16 operands: same tensor rate as bf16, 3 more
// mantissa bits for the activations; the bf16 model weights convert exactly
// at their scale.)
//
// A 128 x BN output tile: TMA streams 128x64 A and BNx64 W tiles (128-byte
// swizzle) into a shared-memory ring, one thread issues tcgen05.mma (M=128,
// N=BN, K=16 per instruction) accumulating fp32 in TMEM and releases each
// ring slot with tcgen05.commit, and the epilogue warps read the accumulator
// back with tcgen05.ld (one tile row per thread) and apply:
//   EPI_STORE_BF16  out fp16 = C                      (QKV projection)
//   EPI_ADD_F32     out fp32 += C                     (O / down projection + residual)
//   EPI_SWIGLU_BF16 out fp16 = silu(C_gate) * C_up    (gate/up projection, rows interleaved
//                                                     in groups of 64, see kSwigluGroup)
// writing each 32-row x 128-byte piece to shared memory and out with a TMA
// store (fp16) or a TMA reduce-add (the fp32 residual: the add happens in L2,
// one fp32 add per element as in a read-modify-write).  The output tensor map
// spans exactly m rows and n columns, so rows >= m (computed on whatever the A
// buffer holds) are clipped by the TMA unit.
//
// Folded RMSNorm (RowNorm, rows <= 256): the persistent kernel's row-scaled
// form (RS) multiplies row r of the accumulator by its rstd, computed from the
// producer's per-tile sums of squares before the tile's accumulator is ready,
// ahead of the fp16 store or SwiGLU.
//
// Two kernels: the single-CTA persistent kernel (gemm_persistent_kernel) and,
// for the tensor-bound projections above 512 rows, the paired-SM kernel
// (gemm_pair_kernel: 256 x 256 tiles over the two CTAs of a cluster with
// tcgen05.mma.cta_group::2, each CTA staging only its own A rows and half of
// the W k-block).  Both share the epilogue (EpiWarp).
#include <cstdio>
#include <mutex>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;  // 64 fp16 = 128 bytes = one swizzle row

__device__ __forceinline__ float silu_f(float g) { return g / (1.0f + __expf(-g)); }

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Persistent GEMM: one CTA per SM walks 128 x BN tiles
// (grouped order: a band of `band` tiles of N down all of M, so a band of
// weight tiles stays in L2 while the activations stream; a weight small
// enough to stay in L2 whole takes one band of all N, so the activations are
// read once), with a double-buffered TMEM accumulator so that the epilogue of
// tile i overlaps the main loop of tile i+1.  Warp 0: TMA producer; warp 1:
// UMMA issuer (and TMEM owner); warps 2-5: epilogue (warp w reads TMEM lanes
// 32*(w%4)..+31).
//
// Residual-add epilogue: the tiles of the last, partial wave can be split
// over k (stream-K).  Tiles [0, first) are whole, CTA c taking c, c + grid,
// ...; the k-blocks of tiles [first, tiles), numbered tile-major, are cut
// into `ctas` contiguous ranges, CTA c < ctas taking range c (at most two
// segments: the high-k end of one tile, then the low-k start of the next).
// Each segment reduce-adds its partial sum into the fp32 output, in a fixed
// order per tile, high k first: a segment that does not reach the tile's last
// k-block waits until the flag of the tile reads (epoch << 32 | its end), and
// a segment that does not start at k-block 0 sets the flag to (epoch << 32 |
// its start) once its adds are complete.  The sums are therefore
// deterministic, and the waits go only to segments that run first in their
// own CTA (a high-k end) or finish with it.
constexpr int kBandN = 4;
constexpr int kSplitMinK = 4;    // k-blocks per CTA at least, when splitting
constexpr int kSplitGainK = 24;  // k-blocks the split must save
#ifndef MZC_GEMM_FULL_BAND_MB
#define MZC_GEMM_FULL_BAND_MB 56
#endif
// weights up to this size walk one band of all N
constexpr double kFullBandBytes = MZC_GEMM_FULL_BAND_MB * static_cast<double>(1 << 20);

// epilogue staging box: 32 rows x 128 bytes
constexpr int kOutBox = 32 * 128;

template <int BN, int STAGES>
struct PCfg {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // epilogue staging: per epilogue warp two 32-row x 128-byte boxes
  static constexpr int OFF_OUT = STAGES * STAGE_BYTES;
  static constexpr int OFF_BAR = OFF_OUT + 4 * 2 * kOutBox;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr uint32_t TMEM_COLS = 2 * BN;  // two accumulators
};

__device__ __forceinline__ bool pwait(uint64_t* bar, uint32_t parity, int32_t* status,
                                      volatile int* abort) {
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

__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int bw, int* mt,
                                            int* nt) {
  const int band = tile / (num_m * bw);
  const int width = min(bw, num_n - band * bw);
  const int within = tile - band * num_m * bw;
  *mt = within / width;
  *nt = band * bw + within % width;
}

// One unit of a CTA's work: k-blocks [kb0, kb1) of a tile; seg = -1 for a
// whole tile, else the index (0, 1) of the CTA's split segment.
struct WorkItem {
  int tile, kb0, kb1, seg;
};

// c / G: this worker (a CTA, or a CTA pair) and the number of workers.
struct Sched {
  int num_k, first, n_dp, c, G;
  long long u0, u1;  // this CTA's range of split k-blocks
};

__device__ __forceinline__ Sched make_sched(int tiles, int num_k, int first, int ctas, int c, int G) {
  Sched s;
  s.num_k = num_k;
  s.first = first;
  s.c = c;
  s.G = G;
  s.n_dp = c < first ? (first - 1 - c) / G + 1 : 0;
  s.u0 = s.u1 = 0;
  if (c < ctas) {
    const long long units = static_cast<long long>(tiles - first) * num_k;
    s.u0 = units * c / ctas;
    s.u1 = units * (c + 1) / ctas;
  }
  return s;
}

__device__ __forceinline__ bool sched_item(const Sched& s, int i, WorkItem* w) {
  if (i < s.n_dp) {
    *w = {s.c + i * s.G, 0, s.num_k, -1};
    return true;
  }
  const int j = i - s.n_dp;
  long long u = s.u0;
  if (j == 1 && u < s.u1) u = min((u / s.num_k + 1) * s.num_k, s.u1);  // past segment 0
  if (j > 1 || u >= s.u1) return false;
  const long long r = u / s.num_k;
  w->tile = s.first + static_cast<int>(r);
  w->kb0 = static_cast<int>(u - r * s.num_k);
  w->kb1 = static_cast<int>(min((r + 1) * s.num_k, s.u1) - r * s.num_k);
  w->seg = j;
  return true;
}

__device__ __forceinline__ uint64_t ld_acquire_u64(const uint64_t* p) {
  uint64_t v;
  asm volatile("ld.acquire.gpu.global.b64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_release_u64(uint64_t* p, uint64_t v) {
  asm volatile("st.release.gpu.global.b64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

// Bounded wait until *flag == want; false once the CTA aborted, another wait
// recorded a timeout, or kWaitCycles passed (then MZC_ERR_TIMEOUT is recorded
// and the CTA aborts).
__device__ __forceinline__ bool split_wait(const uint64_t* flag, uint64_t want, int32_t* status,
                                           volatile int* abort) {
  if (ld_acquire_u64(flag) == want) return true;
  const long long t0 = clock64();
  while (true) {
    __nanosleep(64);
    if (ld_acquire_u64(flag) == want) return true;
    if (*abort) return false;
    if (status != nullptr && *reinterpret_cast<volatile int32_t*>(status) == kStatusTimeout) {
      *abort = 1;
      return false;
    }
    if (clock64() - t0 > kWaitCycles) {
      set_status(status, kStatusTimeout);
      *abort = 1;
      return false;
    }
  }
}

// One epilogue warp's output path for a 128 x BN tile: warp q owns rows
// q*32..+31 (its TMEM lane quarter), lane = row, and two 32 x 128-byte staging
// boxes.  Each box goes out as one TMA store (fp16 outputs) or TMA reduce-add
// into the fp32 residual stream, so the epilogue never reads the output and
// writes whole 128-byte lines.
template <int BN, int EPI, bool RS = false>
struct EpiWarp {
  uint8_t* box0;      // this warp's two staging boxes
  int lane;
  int nbox = 0;       // boxes issued by this warp (buffer = nbox & 1)
  float amax = 0.0f;  // largest |value| this lane stores as fp16

  __device__ EpiWarp(uint8_t* b, int l) : box0(b), lane(l) {}

  // one staging row: 8 16-byte units, unit u at u ^ (row & 7) (128-byte swizzle)
  __device__ __forceinline__ uint8_t* stage_row(const uint32_t* w) {
    uint8_t* box = box0 + (nbox & 1) * kOutBox;
    if (lane == 0 && nbox >= 2) bulk_wait_read<1>();  // the store that last used this box
    __syncwarp();
    uint8_t* r = box + lane * 128;
#pragma unroll
    for (int u = 0; u < 8; ++u)
      *reinterpret_cast<uint4*>(r + ((u ^ (lane & 7)) << 4)) =
          make_uint4(w[4 * u], w[4 * u + 1], w[4 * u + 2], w[4 * u + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    return box;
  }

  // The warp's 32 rows of the tile from TMEM row address trow: rows y..y+31
  // of the output (none stored when y >= m), columns from n0 (of n).  RS:
  // the lane's row is scaled by rs first.
  __device__ __forceinline__ void tile(const CUtensorMap* tmo, uint32_t trow, int y, int n0, int m,
                                       int n, float rs = 1.0f) {
    if constexpr (EPI == EPI_SWIGLU_BF16) {
#pragma unroll 1
      for (int g = 0; g < BN / (2 * kSwigluGroup); ++g) {
        uint32_t pk[32];
#pragma unroll
        for (int c = 0; c < kSwigluGroup; c += 32) {
          float vg[32], vu[32];
          tmem_ld32w(trow + g * 2 * kSwigluGroup + c, vg);
          tmem_ld32w(trow + g * 2 * kSwigluGroup + kSwigluGroup + c, vu);
          if constexpr (RS) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              vg[i] *= rs;
              vu[i] *= rs;
            }
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            const float y0 = silu_f(vg[2 * i]) * vu[2 * i], y1 = silu_f(vg[2 * i + 1]) * vu[2 * i + 1];
            amax = fmaxf(amax, fmaxf(fabsf(y0), fabsf(y1)));
            pk[c / 2 + i] = pack2<true>(y0, y1);
          }
        }
        uint8_t* box = stage_row(pk);
        if (lane == 0) {
          if (y < m && n0 / 2 + g * kSwigluGroup < n / 2)
            tma_store_2d(tmo, box, n0 / 2 + g * kSwigluGroup, y);
          bulk_commit();
        }
        ++nbox;
      }
    } else if constexpr (EPI == EPI_STORE_BF16) {
#pragma unroll 1
      for (int c = 0; c < BN; c += 64) {
        uint32_t pk[32];
#pragma unroll
        for (int h = 0; h < 64; h += 32) {
          float v[32];
          tmem_ld32w(trow + c + h, v);
          if constexpr (RS) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= rs;
          }
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            amax = fmaxf(amax, fmaxf(fabsf(v[2 * i]), fabsf(v[2 * i + 1])));
            pk[h / 2 + i] = pack2<true>(v[2 * i], v[2 * i + 1]);
          }
        }
        uint8_t* box = stage_row(pk);
        if (lane == 0) {
          if (y < m && n0 + c < n) tma_store_2d(tmo, box, n0 + c, y);
          bulk_commit();
        }
        ++nbox;
      }
    } else {
#pragma unroll 1
      for (int c = 0; c < BN; c += 32) {
        float v[32];
        tmem_ld32w(trow + c, v);
        uint8_t* box = stage_row(reinterpret_cast<const uint32_t*>(v));
        if (lane == 0) {
          if (y < m && n0 + c < n) tma_reduce_add_2d(tmo, box, n0 + c, y);
          bulk_commit();
        }
        ++nbox;
      }
    }
  }
};

template <int BN, int STAGES, int EPI, bool RS = false>
__global__ void __launch_bounds__(192, 1) gemm_persistent_kernel(
    const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmw,
    const __grid_constant__ CUtensorMap tmo, int m, int n, int k, int band, int first, int ctas,
    uint64_t* split_flags, uint32_t epoch, int32_t* status, const RowNorm rn) {
  using C = PCfg<BN, STAGES>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + STAGES * C::A_BYTES;
  uint8_t* sOut = smem + C::OFF_OUT;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + STAGES;
  uint64_t* acc_full = empty + STAGES;  // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2]
  uint64_t* mma_done = acc_empty + 2;   // every UMMA issued has completed (teardown)
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  __shared__ int s_split_done[2];  // epilogue warps done with split segment 0 / 1
  volatile int* abort_flag = &s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_m = (m + BM - 1) / BM, num_n = (n + BN - 1) / BN;
  const int num_k = (k + BK - 1) / BK;
  const int tiles = num_m * num_n;
  const Sched sched = make_sched(tiles, num_k, first, ctas, blockIdx.x, gridDim.x);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tma);
    tma_prefetch_desc(&tmw);
    tma_prefetch_desc(&tmo);
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 4);  // one arrival per epilogue warp
    }
    mbar_init(mma_done, 1);
    fence_barrier_init();
    s_abort = 0;
    s_split_done[0] = s_split_done[1] = 0;
  }
  if (warp == 1) tmem_alloc(&s_tmem, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // The prologue above touches no memory another kernel writes.  Neither do
  // the weights: the producer issues the W loads of its first tile's first
  // stages before it waits for the previous kernel (whose output A is), so
  // weight streaming starts under that kernel's tail.
  int pre = 0;
  if (warp == 0 && lane == 0) {
    WorkItem w0;
    if (sched_item(sched, 0, &w0)) {
      int mt0, nt0;
      tile_coords(w0.tile, num_m, num_n, band, &mt0, &nt0);
      pre = min(STAGES, w0.kb1 - w0.kb0);
      for (int i = 0; i < pre; ++i) {
        mbar_arrive_expect_tx(&full[i], C::STAGE_BYTES);
        tma_load_2d(sB + i * C::B_BYTES, &tmw, &full[i], (w0.kb0 + i) * BK, nt0 * BN);
      }
    }
  }
  pdl_enter();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer over all tiles of this CTA ----
      int it = 0;  // global k-block counter (ring position)
      bool ok = true;
      WorkItem w;
      for (int i = 0; ok && sched_item(sched, i, &w); ++i) {
        int mt, nt;
        tile_coords(w.tile, num_m, num_n, band, &mt, &nt);
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const int s = it % STAGES;
          if (it >= STAGES && !pwait(&empty[s], ((it / STAGES) - 1) & 1, status, abort_flag)) {
            ok = false;
            break;
          }
          if (it >= pre) mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);  // else done above
          tma_load_2d(sA + s * C::A_BYTES, &tma, &full[s], kb * BK, mt * BM);
          if (it >= pre) tma_load_2d(sB + s * C::B_BYTES, &tmw, &full[s], kb * BK, nt * BN);
        }
      }
      // drain the last fill of every ring slot before shared memory is
      // released (bounded, and also after an abort: loads still in flight
      // land before the CTA exits)
      for (int i = it - STAGES < 0 ? 0 : it - STAGES; i < it; ++i)
        mbar_wait(&full[i % STAGES], (i / STAGES) & 1, status);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- UMMA issuer ----
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN);
      int it = 0;
      bool ok = true;
      WorkItem w;
      for (int local = 0; ok && sched_item(sched, local, &w); ++local) {
        const int a = local & 1;
        // the epilogue has drained this accumulator (its use two tiles ago)
        if (local >= 2 && !pwait(&acc_empty[a], ((local >> 1) - 1) & 1, status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d = tmem + a * BN;
        for (int kb = w.kb0; kb < w.kb1; ++kb, ++it) {
          const int s = it % STAGES;
          if (!pwait(&full[s], (it / STAGES) & 1, status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sdesc_k_sw128(smem_u32(sA + s * C::A_BYTES));
          const uint64_t bd = sdesc_k_sw128(smem_u32(sB + s * C::B_BYTES));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_f16(d, ad + 2 * kk, bd + 2 * kk, idesc, (kb != w.kb0 || kk != 0) ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&acc_full[a]);
      }
      // every UMMA issued has written TMEM before it is freed (an abort can
      // leave some that no epilogue waited for)
      umma_commit(mma_done);
      mbar_wait(mma_done, 0, status);
    }
  } else {
    // ---- epilogue warps 2-5: TMEM -> registers -> swizzled staging box -> TMA ----
    const int q = warp & 3;
    EpiWarp<BN, EPI, RS> ew(sOut + q * 2 * kOutBox, lane);
    bool ok = true;
    WorkItem w;
    for (int local = 0; sched_item(sched, local, &w); ++local) {
      const int a = local & 1;
      float rs = 1.0f;
      if constexpr (RS) {
        // folded RMSNorm: the lane's row's rstd before the accumulator is ready
        int mt_r, nt_r;
        tile_coords(w.tile, num_m, num_n, band, &mt_r, &nt_r);
        const int row = mt_r * BM + q * 32 + lane;
        if (row < m) rs = row_rstd(rn.ss, rn.nt, rn.d, rn.eps, row);
      }
      ok = ok && pwait(&acc_full[a], (local >> 1) & 1, status, abort_flag);
      __syncwarp();
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      int mt, nt;
      tile_coords(w.tile, num_m, num_n, band, &mt, &nt);
      const int y = mt * BM + q * 32;
      const uint32_t trow = tmem + a * BN + (static_cast<uint32_t>(q * 32) << 16);
      const int n0 = nt * BN;
      if constexpr (EPI != EPI_ADD_F32) {
        ew.tile(&tmo, trow, y, n0, m, n, rs);
      } else {
        uint64_t* flag = w.seg >= 0 ? split_flags + (w.tile - first) : nullptr;
        bool go = true;
        if (flag != nullptr && w.kb1 < num_k) {
          // the segment above (higher k) adds first
          if (lane == 0) {
            go = split_wait(flag, (static_cast<uint64_t>(epoch) << 32) | static_cast<uint32_t>(w.kb1),
                            status, abort_flag);
            if (go) fence_proxy_async_global();
          }
          go = __shfl_sync(0xffffffffu, go, 0);
        }
        if (go) ew.tile(&tmo, trow, y, n0, m, n);
        if (flag != nullptr && w.kb0 > 0) {
          // the segment below waits for this one: the last epilogue warp to
          // finish its adds (complete in global memory) sets the flag
          if (lane == 0) {
            bulk_wait_all();
            fence_proxy_async_global();
            __threadfence();
            if (atomicAdd(&s_split_done[w.seg], 1) == 3) {
              __threadfence();
              if (!*abort_flag)
                st_release_u64(flag, (static_cast<uint64_t>(epoch) << 32) | static_cast<uint32_t>(w.kb0));
            }
          }
          __syncwarp();
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[a]);
    }
    // every store has finished reading shared memory and reached global memory
    if (lane == 0) bulk_wait_all();
    __syncwarp();
    if constexpr (EPI != EPI_ADD_F32) note_f16_overflow(status, ew.amax);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// ---- paired-SM GEMM for the tensor-bound projections (m > 512) ----
//
// The two CTAs of a cluster pair compute one 256 x 256 output tile with
// tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 16), issued by one thread of
// the even CTA.  Each CTA stages only its own operand halves per k-block: its
// 128 A rows and 128 of the tile's 256 W rows (32 KB, against 48 KB for a
// single-CTA 128 x 256 tile), so the TMA writes into each SM's shared memory
// fall by a third while the tensor work per SM stays the same; each CTA's TMEM
// holds its 128 rows x 256 columns.  Per CTA: warp 0 is the TMA producer,
// whose loads complete on the even CTA's `full` barrier (the even CTA
// expects both CTAs' bytes), warp 1 of the even CTA issues the UMMAs, and
// warps 2-5 run the same epilogue as the single-CTA kernel on the CTA's own
// rows, then release the accumulator on the even CTA's `acc_empty` (8
// arrivals: both CTAs' epilogue warps).  The UMMA commits arrive on both
// CTAs' barriers (multicast).  Work units are the
// pair tiles (p, nt), M tiles 2p (even CTA) and 2p + 1 (odd CTA); an odd last
// M tile pairs with a tile of padding rows that computes on zeros or stale rows
// and stores nothing.
constexpr int kPairStages = 6;

struct PairCfg {
  static constexpr int A_BYTES = BM * BK * 2;     // this CTA's 128 A rows
  static constexpr int B_BYTES = 128 * BK * 2;    // this CTA's 128 of the 256 W rows
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  static constexpr int OFF_OUT = kPairStages * STAGE_BYTES;
  static constexpr int OFF_BAR = OFF_OUT + 4 * 2 * kOutBox;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;
  static constexpr uint32_t TMEM_COLS = 512;  // two 256-column accumulators
  static_assert((2 * kPairStages + 5) * 8 <= 256, "barriers");
};

__device__ __forceinline__ bool pwait_cluster(uint64_t* bar, uint32_t parity, int32_t* status,
                                              volatile int* abort) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const long long t0 = clock64();
  while (true) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if (*abort) return false;
    if (clock64() - t0 > kWaitCycles) {
      set_status(status, kStatusTimeout);
      *abort = 1;
      return false;
    }
  }
}

template <int EPI>
__global__ void __launch_bounds__(192, 1) gemm_pair_kernel(
    const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmw,
    const __grid_constant__ CUtensorMap tmo, int m, int n, int k, int band, int32_t* status) {
  using C = PairCfg;
  constexpr int BN = 256, S = kPairStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + S * C::A_BYTES;
  uint8_t* sOut = smem + C::OFF_OUT;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);  // even CTA: both CTAs' stage
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;       // [2]
  uint64_t* acc_empty = acc_full + 2;   // [2] even CTA: both CTAs drained the accumulator
  uint64_t* mma_done = acc_empty + 2;   // even CTA: every UMMA issued has completed
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  volatile int* abort_flag = &s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int rank = static_cast<int>(cluster_rank());
  const int num_m = (m + BM - 1) / BM, num_n = (n + BN - 1) / BN;
  const int num_k = (k + BK - 1) / BK;
  const int unit_m = (num_m + 1) / 2;
  const int units = unit_m * num_n;
  const int cid = static_cast<int>(blockIdx.x >> 1), ncl = static_cast<int>(gridDim.x >> 1);

  if (threadIdx.x == 0) {
    tma_prefetch_desc(&tma);
    tma_prefetch_desc(&tmw);
    tma_prefetch_desc(&tmo);
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&acc_full[a], 1);
      mbar_init(&acc_empty[a], 8);  // four epilogue warps in each CTA
    }
    mbar_init(mma_done, 1);
    fence_barrier_init();
    s_abort = 0;
  }
  if (warp == 1) tmem_alloc_pair(&s_tmem, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  // both CTAs' barriers are initialised before either arrives on the other's
  cluster_sync_all();
  tc_fence_after();
  // The prologue above touches no memory another kernel writes.  Neither do
  // the weights: each producer issues its W half of the first unit's first
  // stages before it waits for the previous kernel (whose output A is).
  int pre = 0;
  if (warp == 0 && lane == 0 && cid < units) {
    int mp0, nt0;
    tile_coords(cid, unit_m, num_n, band, &mp0, &nt0);
    pre = min(S, num_k);
    const uint32_t full0 = map_rank(smem_u32(full), 0);
    for (int i = 0; i < pre; ++i) {
      if (rank == 0) mbar_arrive_expect_tx(&full[i], 2 * C::STAGE_BYTES);
      tma_load_2d_pair(sB + i * C::B_BYTES, &tmw, full0 + i * 8, i * BK, nt0 * BN + rank * 128);
    }
  }
  pdl_enter();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer: this CTA's A rows and W half of every k-block ----
      int it = 0;
      bool ok = true;
      const uint32_t full0 = map_rank(smem_u32(full), 0);  // the even CTA's full[0]
      for (int u = cid; ok && u < units; u += ncl) {
        int mp, nt;
        tile_coords(u, unit_m, num_n, band, &mp, &nt);
        const int mt = 2 * mp + rank;
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int s = it % S;
          if (it >= S && !pwait(&empty[s], ((it / S) - 1) & 1, status, abort_flag)) {
            ok = false;
            break;
          }
          if (rank == 0 && it >= pre) mbar_arrive_expect_tx(&full[s], 2 * C::STAGE_BYTES);
          tma_load_2d_pair(sA + s * C::A_BYTES, &tma, full0 + s * 8, kb * BK, mt * BM);
          if (it >= pre) tma_load_2d_pair(sB + s * C::B_BYTES, &tmw, full0 + s * 8, kb * BK, nt * BN + rank * 128);
        }
      }
      // every fill issued (by both CTAs) has landed before shared memory is
      // released: the even CTA waits for its barriers, and the final cluster
      // barrier holds the odd CTA until then
      if (rank == 0)
        for (int i = it - S < 0 ? 0 : it - S; i < it; ++i) mbar_wait(&full[i % S], (i / S) & 1, status);
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0) {
      // ---- even CTA: UMMA issuer for the pair ----
      constexpr uint32_t idesc = idesc_f16_f32(256, BN);
      int it = 0, local = 0;
      bool ok = true;
      for (int u = cid; ok && u < units; u += ncl, ++local) {
        const int a = local & 1;
        // both CTAs have drained this accumulator (its use two units ago)
        if (local >= 2 && !pwait_cluster(&acc_empty[a], ((local >> 1) - 1) & 1, status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d = tmem + a * BN;
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int s = it % S;
          if (!pwait_cluster(&full[s], (it / S) & 1, status, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t ad = sdesc_k_sw128(smem_u32(sA + s * C::A_BYTES));
          const uint64_t bd = sdesc_k_sw128(smem_u32(sB + s * C::B_BYTES));
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            umma_pair_f16(d, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit_pair(&empty[s], 0x3);  // the slot is free in both CTAs
        }
        if (ok) umma_commit_pair(&acc_full[a], 0x3);
      }
      // every UMMA issued has written both CTAs' TMEM before it is freed
      umma_commit_pair(mma_done, 0x1);
      mbar_wait(mma_done, 0, status);
    }
  } else {
    // ---- epilogue warps 2-5 of both CTAs: this CTA's 128 rows of the tile ----
    const int q = warp & 3;
    EpiWarp<BN, EPI> ew(sOut + q * 2 * kOutBox, lane);
    bool ok = true;
    int local = 0;
    for (int u = cid; u < units; u += ncl, ++local) {
      const int a = local & 1;
      ok = ok && pwait(&acc_full[a], (local >> 1) & 1, status, abort_flag);
      __syncwarp();
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      int mp, nt;
      tile_coords(u, unit_m, num_n, band, &mp, &nt);
      const int y = (2 * mp + rank) * BM + q * 32;
      const uint32_t trow = tmem + a * BN + (static_cast<uint32_t>(q * 32) << 16);
      ew.tile(&tmo, trow, y, nt * BN, m, n);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0) {
          mbar_arrive(&acc_empty[a]);
        } else {
          mbar_arrive_remote(&acc_empty[a], 0);
        }
      }
    }
    // every store has finished reading shared memory and reached global memory
    if (lane == 0) bulk_wait_all();
    __syncwarp();
    if constexpr (EPI != EPI_ADD_F32) note_f16_overflow(status, ew.amax);
  }

  tc_fence_before();
  __syncthreads();
  // neither CTA frees TMEM or leaves while the pair's UMMAs or arrivals may
  // still reach it
  cluster_sync_all();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc_pair(tmem, C::TMEM_COLS);
  }
}

using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                              const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                              const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                              CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

// Output [rows][cols] (fp16, or fp32 for the residual stream) in boxes of
// 32 rows x 128 bytes with 128-byte swizzle, matching the epilogue's staging.
bool make_out_map(CUtensorMap* map, void* base, uint64_t rows, uint64_t cols, bool f32) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  const uint64_t esz = f32 ? 4 : 2;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * esz};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(128 / esz), 32};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, base,
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

#ifndef MZC_GEMM_PAIR
#define MZC_GEMM_PAIR 1
#endif

// Resident clusters of the paired kernel (0 when the query fails).
template <int EPI>
int pair_clusters() {
  static std::once_flag once;
  static int count = 0;
  std::call_once(once, [] {
    if (cudaFuncSetAttribute(gemm_pair_kernel<EPI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             PairCfg::SMEM) != cudaSuccess) {
      cudaGetLastError();
      return;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2, 1, 1);
    cfg.blockDim = dim3(192, 1, 1);
    cfg.dynamicSmemBytes = PairCfg::SMEM;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int c = 0;
    if (cudaOccupancyMaxActiveClusters(&c, gemm_pair_kernel<EPI>, &cfg) == cudaSuccess) count = c;
    cudaGetLastError();  // a refused query leaves no error behind
  });
  return count;
}

// The paired kernel over 256 x 256 pair tiles; tw128: W with 128-row boxes.
// *launched is false (nothing launched) when no cluster pair can be resident,
// or when the pair tiles need more waves over the resident pairs than the
// single-CTA 128 x 256 tiles need over the SMs (a pair wave does the work of
// a single-CTA wave in about the same time or less; measured on the 1B and
// 3B projections).
template <int EPI>
cudaError_t launch_pair(const CUtensorMap& ta, const CUtensorMap& tw128, void* out, int64_t m,
                        int64_t n, int64_t k, int32_t* status, cudaStream_t st, int sms,
                        bool* launched) {
  *launched = false;
  const int clusters = pair_clusters<EPI>();
  if (clusters <= 0) return cudaSuccess;
  {
    const int64_t num_m = (m + BM - 1) / BM, num_n = (n + 255) / 256;
    const int64_t units = (num_m + 1) / 2 * num_n, tiles = num_m * num_n;
    if ((units + clusters - 1) / clusters > (tiles + sms - 1) / sms) return cudaSuccess;
  }
  CUtensorMap tmo;
  if (!make_out_map(&tmo, out, static_cast<uint64_t>(m),
                    static_cast<uint64_t>(EPI == EPI_SWIGLU_BF16 ? n / 2 : n), EPI == EPI_ADD_F32))
    return cudaErrorInvalidValue;
  const int64_t num_m = (m + BM - 1) / BM, num_n = (n + 255) / 256;
  const int64_t units = (num_m + 1) / 2 * num_n;
  const int band = static_cast<double>(n) * static_cast<double>(k) * 2.0 <= kFullBandBytes
                       ? static_cast<int>(num_n) : kBandN;
  const int64_t g = units < clusters ? units : clusters;
  *launched = true;
  launch_k_cluster(gemm_pair_kernel<EPI>, dim3(static_cast<unsigned>(2 * g)), dim3(192),
                   PairCfg::SMEM, st, 2u, ta, tw128, tmo, static_cast<int>(m), static_cast<int>(n),
                   static_cast<int>(k), band, status);
  return cudaGetLastError();
}

template <int BN, int STAGES, int EPI, bool RS = false>
cudaError_t launch_persistent(const CUtensorMap& ta, const CUtensorMap& tw, void* out, int64_t m, int64_t n, int64_t k, int32_t* status,
                              cudaStream_t st, GemmSplit* split, const RowNorm* rn = nullptr) {
  using C = PCfg<BN, STAGES>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  static int sms = 0;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(gemm_persistent_kernel<BN, STAGES, EPI, RS>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    int dev = 0;
    if (attr_err == cudaSuccess) attr_err = cudaGetDevice(&dev);
    if (attr_err == cudaSuccess)
      attr_err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  });
  if (attr_err != cudaSuccess) return attr_err;
  CUtensorMap tmo;
  const bool f32 = EPI == EPI_ADD_F32;
  if (!make_out_map(&tmo, out, static_cast<uint64_t>(m),
                    static_cast<uint64_t>(EPI == EPI_SWIGLU_BF16 ? n / 2 : n), f32))
    return cudaErrorInvalidValue;
  const int64_t num_m = (m + BM - 1) / BM;
  const int64_t num_n = (n + BN - 1) / BN;
  const int64_t tiles = num_m * num_n;
  const int band = static_cast<double>(n) * static_cast<double>(k) * 2.0 <= kFullBandBytes
                       ? static_cast<int>(num_n) : kBandN;
  if (split != nullptr) split->last_ctas = 0;
  int64_t grid = tiles < sms ? tiles : sms;
  int64_t first = tiles, ctas = 0;
  uint64_t* flags = nullptr;
  uint32_t epoch = 0;
  if (EPI == EPI_ADD_F32 && split != nullptr && split->flags != nullptr && split->n_flags >= sms) {
    // split the last wave's R tiles over up to 2R CTAs (all SMs at most),
    // each taking at least kSplitMinK k-blocks, when the k-blocks the last
    // wave saves, (1 - R / SMs) of a tile's, reach kSplitGainK: the ordered
    // adds at the end cost about that much (measured on the 1B and 3B O and
    // down projections: a gain at K 8192, a loss at K 2048-3072)
    const int64_t num_k = (k + BK - 1) / BK;
    const int64_t f = ((tiles + sms - 1) / sms - 1) * sms;
    const int64_t r = tiles - f;
    int64_t g = 2 * r < sms ? 2 * r : sms;
    if (r * num_k / kSplitMinK < g) g = r * num_k / kSplitMinK;
    if (r < sms && g > r && (sms - r) * num_k >= kSplitGainK * sms) {
      first = f;
      ctas = g;
      if (grid < g) grid = g;
      flags = split->flags;
      epoch = next_split_epoch(split);
      split->last_ctas = g;
    }
  }
  const RowNorm norm = rn != nullptr ? *rn : RowNorm{};
  launch_k(gemm_persistent_kernel<BN, STAGES, EPI, RS>, dim3(static_cast<unsigned>(grid)),
      dim3(192), C::SMEM, st, ta, tw, tmo, static_cast<int>(m), static_cast<int>(n),
      static_cast<int>(k), band, static_cast<int>(first), static_cast<int>(ctas), flags, epoch,
      status, norm);
  return cudaGetLastError();
}

}  // namespace

bool make_tmap_f16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols,
                    uint32_t box_rows) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {cols, rows};
  cuuint64_t strides[1] = {cols * 2};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), box_rows};
  cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

uint32_t gemm_box_n(int64_t m, int64_t n, int epilogue) {
  if (m > 512) return 256;  // tensor-bound: 128 x 256 tiles
  // Weight-streaming bound: the tile width with the fewest waves over the SMs
  // and, among those, the most tiles (the most SMs pulling weight bytes).
  // SwiGLU tiles hold whole 128-row gate/up groups.
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (sms <= 0) sms = 1;
  }
  const int64_t mt = (m + BM - 1) / BM;
  uint32_t best = 256;
  int64_t best_waves = 0, best_tiles = 0;
  for (uint32_t bn : {256u, 128u, 64u}) {
    if (epilogue == EPI_SWIGLU_BF16 && bn < 128) continue;
    const int64_t tiles = mt * ((n + bn - 1) / bn);
    const int64_t waves = (tiles + sms - 1) / sms;
    if (best_tiles == 0 || waves < best_waves || (waves == best_waves && tiles > best_tiles)) {
      best = bn;
      best_waves = waves;
      best_tiles = tiles;
    }
  }
  return best;
}

bool make_gemm_weight(GemmWeight* gw, const void* base, uint64_t n, uint64_t k) {
  gw->ptr = static_cast<const uint16_t*>(base);
  return make_tmap_f16(&gw->box64, base, n, k, 64) && make_tmap_f16(&gw->box128, base, n, k, 128) &&
         make_tmap_f16(&gw->box256, base, n, k, 256);
}

// Tile choice (gemm_box_n): above 512 rows the GEMM is tensor-bound and takes
// 128 x 256 tiles with a 4-stage ring; at or below it streams the weights and
// takes the width that keeps the most SMs busy in the fewest waves, with a
// deeper ring for the narrower tiles.  The W map passed has the matching box.
cudaError_t launch_gemm(const CUtensorMap& ta, const GemmWeight& w, void* out, int64_t m,
                        int64_t n, int64_t k, int epilogue, int32_t* status, cudaStream_t st,
                        const uint16_t* a_ptr, GemmSplit* split, const RowNorm* rn) {
  if (m <= 0) return cudaSuccess;
  const bool norm_out = rn != nullptr && rn->h != nullptr && epilogue == EPI_ADD_F32;
  const bool norm_in = rn != nullptr && rn->ss != nullptr && epilogue != EPI_ADD_F32;
  if ((norm_out || norm_in) && m == 1 && a_ptr && w.ptr)
    return launch_gemv(a_ptr, w.ptr, out, m, n, k, epilogue, status, st, rn);  // one-row fold
  if (norm_out || norm_in) {
    // a folded RMSNorm: 5 to 256 rows, 128-column tiles of x
    if (m <= kGemvMaxRows || m > 256 || rn->nt <= 0 || rn->ss == nullptr ||
        (norm_out && (rn->g == nullptr || static_cast<int64_t>(rn->nt) * 128 != n)))
      return cudaErrorInvalidValue;
  }
  if (a_ptr && w.ptr && m <= kGemvMaxRows)
    return launch_gemv(a_ptr, w.ptr, out, m, n, k, epilogue, status, st);
  if (m <= 256) {
    // weight-streaming bound with few N tiles: split K over a cluster
    static int sms = 0;
    if (sms == 0) {
      int dev = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (sms <= 0) sms = 1;
    }
    bool launched = false;
    const cudaError_t e = launch_gemm_splitk(ta, w, out, m, n, k, epilogue, sms, status, st, &launched,
                                             (norm_out || norm_in) ? rn : nullptr);
    if (launched || e != cudaSuccess) return e;
  }
  const uint32_t bn = gemm_box_n(m, n, epilogue);
  if (norm_out) return cudaErrorInvalidValue;  // only the split-K kernel writes h and the sums
  if (norm_in) {
    // the row-scaled persistent kernel (no paired form)
    if (epilogue == EPI_SWIGLU_BF16) {
      if (bn == 256) return launch_persistent<256, 4, EPI_SWIGLU_BF16, true>(ta, w.box256, out, m, n, k, status, st, split, rn);
      return launch_persistent<128, 6, EPI_SWIGLU_BF16, true>(ta, w.box128, out, m, n, k, status, st, split, rn);
    }
    if (bn == 256) return launch_persistent<256, 4, EPI_STORE_BF16, true>(ta, w.box256, out, m, n, k, status, st, split, rn);
    if (bn == 128) return launch_persistent<128, 6, EPI_STORE_BF16, true>(ta, w.box128, out, m, n, k, status, st, split, rn);
    return launch_persistent<64, 8, EPI_STORE_BF16, true>(ta, w.box64, out, m, n, k, status, st, split, rn);
  }
  if (bn == 256 && MZC_GEMM_PAIR && m > BM) {
    // tensor-bound: the paired-SM kernel over 256 x 256 tiles
    static int sms = 0;
    if (sms == 0) {
      int dev = 0;
      cudaGetDevice(&dev);
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
      if (sms <= 0) sms = 1;
    }
    bool launched = false;
    cudaError_t e = cudaSuccess;
    switch (epilogue) {
      case EPI_STORE_BF16:
        e = launch_pair<EPI_STORE_BF16>(ta, w.box128, out, m, n, k, status, st, sms, &launched);
        break;
      case EPI_ADD_F32:
        e = launch_pair<EPI_ADD_F32>(ta, w.box128, out, m, n, k, status, st, sms, &launched);
        break;
      case EPI_SWIGLU_BF16:
        e = launch_pair<EPI_SWIGLU_BF16>(ta, w.box128, out, m, n, k, status, st, sms, &launched);
        break;
      default:
        return cudaErrorInvalidValue;
    }
    if (launched || e != cudaSuccess) {
      if (split != nullptr) split->last_ctas = 0;
      return e;
    }
  }
  if (bn == 256) {
    switch (epilogue) {
      case EPI_STORE_BF16:
        return launch_persistent<256, 4, EPI_STORE_BF16>(ta, w.box256, out, m, n, k, status, st, split);
      case EPI_ADD_F32:
        return launch_persistent<256, 4, EPI_ADD_F32>(ta, w.box256, out, m, n, k, status, st, split);
      case EPI_SWIGLU_BF16:
        return launch_persistent<256, 4, EPI_SWIGLU_BF16>(ta, w.box256, out, m, n, k, status, st, split);
      default:
        return cudaErrorInvalidValue;
    }
  }
  if (bn == 128) {
    switch (epilogue) {
      case EPI_STORE_BF16:
        return launch_persistent<128, 6, EPI_STORE_BF16>(ta, w.box128, out, m, n, k, status, st, split);
      case EPI_ADD_F32:
        return launch_persistent<128, 6, EPI_ADD_F32>(ta, w.box128, out, m, n, k, status, st, split);
      case EPI_SWIGLU_BF16:
        return launch_persistent<128, 6, EPI_SWIGLU_BF16>(ta, w.box128, out, m, n, k, status, st, split);
      default:
        return cudaErrorInvalidValue;
    }
  }
  switch (epilogue) {
    case EPI_STORE_BF16:
      return launch_persistent<64, 8, EPI_STORE_BF16>(ta, w.box64, out, m, n, k, status, st, split);
    case EPI_ADD_F32:
      return launch_persistent<64, 8, EPI_ADD_F32>(ta, w.box64, out, m, n, k, status, st, split);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace mzc
