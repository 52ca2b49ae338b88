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
// (grouped order: a band of kBandN tiles of N down all of M, so a band of
// weight tiles stays in L2 while the activations stream), with a
// double-buffered TMEM accumulator so that the epilogue of tile i overlaps
// the main loop of tile i+1.  Warp 0: TMA producer; warp 1: UMMA issuer
// (and TMEM owner); warps 2-5: epilogue (warp w reads TMEM lanes
// 32*(w%4)..+31).
constexpr int kBandN = 4;

template <int BN, int STAGES>
struct PCfg {
  static constexpr int A_BYTES = BM * BK * 2;
  static constexpr int B_BYTES = BN * BK * 2;
  static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
  // epilogue staging: per epilogue warp two 32-row x 128-byte boxes
  static constexpr int OUT_BOX = 32 * 128;
  static constexpr int OFF_OUT = STAGES * STAGE_BYTES;
  static constexpr int OFF_BAR = OFF_OUT + 4 * 2 * OUT_BOX;
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

__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int* mt, int* nt) {
  const int band = tile / (num_m * kBandN);
  const int width = min(kBandN, num_n - band * kBandN);
  const int within = tile - band * num_m * kBandN;
  *mt = within / width;
  *nt = band * kBandN + within % width;
}

template <int BN, int STAGES, int EPI>
__global__ void __launch_bounds__(192, 1) gemm_persistent_kernel(
    const __grid_constant__ CUtensorMap tma, const __grid_constant__ CUtensorMap tmw,
    const __grid_constant__ CUtensorMap tmo, int m, int n, int k, int32_t* status) {
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
  __shared__ uint32_t s_tmem;
  __shared__ int s_abort;
  volatile int* abort_flag = &s_abort;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int num_m = (m + BM - 1) / BM, num_n = (n + BN - 1) / BN;
  const int tiles = num_m * num_n;
  const int num_k = (k + BK - 1) / BK;

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
    fence_barrier_init();
    s_abort = 0;
  }
  if (warp == 1) tmem_alloc(&s_tmem, C::TMEM_COLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // the prologue above touches no memory another kernel writes
  pdl_enter();
  const uint32_t tmem = s_tmem;

  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer over all tiles of this CTA ----
      int it = 0;  // global k-block counter (ring position)
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x) {
        int mt, nt;
        tile_coords(tile, num_m, num_n, &mt, &nt);
        for (int kb = 0; kb < num_k; ++kb, ++it) {
          const int s = it % STAGES;
          if (it >= STAGES && !pwait(&empty[s], ((it / STAGES) - 1) & 1, status, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], C::STAGE_BYTES);
          tma_load_2d(sA + s * C::A_BYTES, &tma, &full[s], kb * BK, mt * BM);
          tma_load_2d(sB + s * C::B_BYTES, &tmw, &full[s], kb * BK, nt * BN);
        }
      }
      // drain the last fill of every ring slot before shared memory is released
      for (int i = it - STAGES < 0 ? 0 : it - STAGES; i < it; ++i)
        pwait(&full[i % STAGES], (i / STAGES) & 1, status, abort_flag);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ---- UMMA issuer ----
      constexpr uint32_t idesc = idesc_f16_f32(BM, BN);
      int it = 0, local = 0;
      bool ok = true;
      for (int tile = blockIdx.x; ok && tile < tiles; tile += gridDim.x, ++local) {
        const int a = local & 1;
        // the epilogue has drained this accumulator (its use two tiles ago)
        if (local >= 2 && !pwait(&acc_empty[a], ((local >> 1) - 1) & 1, status, abort_flag)) break;
        tc_fence_after();
        const uint32_t d = tmem + a * BN;
        for (int kb = 0; kb < num_k; ++kb, ++it) {
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
            umma_f16(d, ad + 2 * kk, bd + 2 * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          umma_commit(&empty[s]);
        }
        if (ok) umma_commit(&acc_full[a]);
      }
    }
  } else {
    // ---- epilogue warps 2-5: TMEM -> registers -> swizzled staging box -> TMA ----
    // Warp q owns rows q*32..+31 of the tile (its TMEM lane quarter) and two
    // 32 x 128-byte staging boxes; lane = row.  Each box goes out as one TMA
    // store (fp16 outputs) or TMA reduce-add into the fp32 residual stream, so
    // the epilogue never reads the output and writes whole 128-byte lines.
    const int q = warp & 3;
    uint8_t* box0 = sOut + q * 2 * C::OUT_BOX;
    int nbox = 0;  // boxes issued by this warp (buffer = nbox & 1)
    // one staging row: 8 16-byte units, unit u at u ^ (row & 7) (128-byte swizzle)
    auto stage_row = [&](const uint32_t* w) -> uint8_t* {
      uint8_t* box = box0 + (nbox & 1) * C::OUT_BOX;
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
    };
    int local = 0;
    bool ok = true;
    float amax = 0.0f;  // largest |value| this lane stores as fp16
    for (int tile = blockIdx.x; tile < tiles; tile += gridDim.x, ++local) {
      const int a = local & 1;
      ok = ok && pwait(&acc_full[a], (local >> 1) & 1, status, abort_flag);
      __syncwarp();
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      int mt, nt;
      tile_coords(tile, num_m, num_n, &mt, &nt);
      const int y = mt * BM + q * 32;
      const uint32_t trow = tmem + a * BN + (static_cast<uint32_t>(q * 32) << 16);
      const int n0 = nt * BN;
      if constexpr (EPI == EPI_SWIGLU_BF16) {
#pragma unroll 1
        for (int g = 0; g < BN / (2 * kSwigluGroup); ++g) {
          uint32_t pk[32];
#pragma unroll
          for (int c = 0; c < kSwigluGroup; c += 32) {
            float vg[32], vu[32];
            tmem_ld32w(trow + g * 2 * kSwigluGroup + c, vg);
            tmem_ld32w(trow + g * 2 * kSwigluGroup + kSwigluGroup + c, vu);
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
              tma_store_2d(&tmo, box, n0 / 2 + g * kSwigluGroup, y);
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
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              amax = fmaxf(amax, fmaxf(fabsf(v[2 * i]), fabsf(v[2 * i + 1])));
              pk[h / 2 + i] = pack2<true>(v[2 * i], v[2 * i + 1]);
            }
          }
          uint8_t* box = stage_row(pk);
          if (lane == 0) {
            if (y < m && n0 + c < n) tma_store_2d(&tmo, box, n0 + c, y);
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
            if (y < m && n0 + c < n) tma_reduce_add_2d(&tmo, box, n0 + c, y);
            bulk_commit();
          }
          ++nbox;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[a]);
    }
    // every store has finished reading shared memory and reached global memory
    if (lane == 0) bulk_wait_all();
    __syncwarp();
    if constexpr (EPI != EPI_ADD_F32) note_f16_overflow(status, amax);
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, C::TMEM_COLS);
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

template <int BN, int STAGES, int EPI>
cudaError_t launch_persistent(const CUtensorMap& ta, const CUtensorMap& tw, void* out, int64_t m,
                              int64_t n, int64_t k, int32_t* status, cudaStream_t st) {
  using C = PCfg<BN, STAGES>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  static int sms = 0;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(gemm_persistent_kernel<BN, STAGES, EPI>,
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
  const int64_t tiles = ((m + BM - 1) / BM) * ((n + BN - 1) / BN);
  const unsigned grid = static_cast<unsigned>(tiles < sms ? tiles : sms);
  launch_k(gemm_persistent_kernel<BN, STAGES, EPI>, dim3(grid), dim3(192), C::SMEM, st,
      ta, tw, tmo, static_cast<int>(m), static_cast<int>(n), static_cast<int>(k), status);
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
                        const uint16_t* a_ptr) {
  if (m <= 0) return cudaSuccess;
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
    const cudaError_t e = launch_gemm_splitk(ta, w, out, m, n, k, epilogue, sms, status, st, &launched);
    if (launched || e != cudaSuccess) return e;
  }
  const uint32_t bn = gemm_box_n(m, n, epilogue);
  if (bn == 256) {
    switch (epilogue) {
      case EPI_STORE_BF16:
        return launch_persistent<256, 4, EPI_STORE_BF16>(ta, w.box256, out, m, n, k, status, st);
      case EPI_ADD_F32:
        return launch_persistent<256, 4, EPI_ADD_F32>(ta, w.box256, out, m, n, k, status, st);
      case EPI_SWIGLU_BF16:
        return launch_persistent<256, 4, EPI_SWIGLU_BF16>(ta, w.box256, out, m, n, k, status, st);
      default:
        return cudaErrorInvalidValue;
    }
  }
  if (bn == 128) {
    switch (epilogue) {
      case EPI_STORE_BF16:
        return launch_persistent<128, 6, EPI_STORE_BF16>(ta, w.box128, out, m, n, k, status, st);
      case EPI_ADD_F32:
        return launch_persistent<128, 6, EPI_ADD_F32>(ta, w.box128, out, m, n, k, status, st);
      case EPI_SWIGLU_BF16:
        return launch_persistent<128, 6, EPI_SWIGLU_BF16>(ta, w.box128, out, m, n, k, status, st);
      default:
        return cudaErrorInvalidValue;
    }
  }
  switch (epilogue) {
    case EPI_STORE_BF16:
      return launch_persistent<64, 8, EPI_STORE_BF16>(ta, w.box64, out, m, n, k, status, st);
    case EPI_ADD_F32:
      return launch_persistent<64, 8, EPI_ADD_F32>(ta, w.box64, out, m, n, k, status, st);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace mzc
