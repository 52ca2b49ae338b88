// Causal grouped-query flash attention for prefill over a block-table KV
// cache (the paper's single-pass attention over non-contiguous KV chunks with
// online softmax, Sec. 4.2), on the 5th-generation tensor cores.
//
// One CTA owns two tiles of 128 query rows of one KV head g: the n tokens x
// (hq/hkv) query heads that share g are flattened token-major (row r = token
// r / group, head g*group + r % group), so every K/V tile serves both Q tiles
// and `group` heads.  Per BN-key tile of its key range:
//   - warp 8 looks the tile's 16-token blocks up in the block table (one lane
//     per block, a tile ahead) and fetches their K and V rows with TMA into a
//     4-5-stage ring, 128-byte swizzle: one box per 64-column slice when the
//     blocks are consecutive in the pool, else one 16-row box per block;
//   - warps 9 and 10 (one thread each, one per Q tile t, so neither tile's
//     UMMAs queue behind the other's waits) issue tcgen05.mma: S_t = Q_t K^T
//     into the tile's TMEM S buffer (M=128, N=BN, K-major operands from shared
//     memory), and, once its softmax warpgroup has written P_t, O_t += P_t V
//     into the tile's TMEM accumulator with P_t read from TMEM (A operand) and
//     V from shared memory as an MN-major operand in its stored layout;
//   - warps 0-3 and 4-7 are the softmax warpgroups of the two Q tiles, one
//     thread per row: the whole S row comes out of TMEM together with its
//     maximum (tcgen05.ld.red; the S buffer is released right away, so the
//     next S runs on the tensor cores during the exponentials), is masked by
//     the row's position on diagonal tiles (their maximum is then reduced in
//     registers),
//     exponentiated in base 2 against a running reference maximum into fp16
//     registers, and written as P into its TMEM columns once the previous P V
//     has released them.  O is rescaled in TMEM only when the maximum grows by
//     more than 2^8 ("lazy" rescale), so P stays <= 256.  The two warpgroups
//     never wait for each other, so one exponentiates while the other waits on
//     its S.
// Keeping P in TMEM leaves shared-memory bandwidth to the K/V operands: at
// head dim 64 an M=128 x N=64 P V with P in shared memory reads more bytes
// per FLOP than the tensor core consumes.
// Long key ranges with few rows are split across CTAs (split-KV); each split
// writes its normalised partial output and base-2 log-sum-exp, and a combine
// kernel merges them.
#include <algorithm>
#include <climits>
#include <cmath>
#include <mutex>
#include <type_traits>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {


template <int HD>
struct AttnCfg {
  static constexpr int BM = 128;                  // rows per Q tile (TMEM lanes)
  static constexpr int BN = HD == 64 ? 128 : 64;  // keys per tile
  // Q tiles per CTA (both share every K/V tile) and CTAs per SM.  One tile
  // per CTA with two CTAs per SM (2-stage ring) measured 32% slower at head
  // dim 64: each CTA fetches its own K/V and the shallow ring exposes latency.
  static constexpr int NQ = 2;
  static constexpr int CTAS_PER_SM = 1;
  static constexpr int ROWS = NQ * BM;
  // warps: 4 NQ softmax, then the TMA producer, then NQ UMMA issuers
  static constexpr int PRODUCER_WARP = 4 * NQ;
  static constexpr int THREADS = (5 * NQ + 1) * 32;
  static constexpr int STAGES = HD == 64 ? 5 : 4;
  static constexpr int CB = HD / 64;              // 64-column slices of the head dim
  static constexpr int Q_BYTES = BM * HD * 2;     // one Q tile
  static constexpr int KV_BYTES = BN * HD * 2;    // K or V of one key tile
  static constexpr int OFF_K = NQ * Q_BYTES;
  static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + STAGES * KV_BYTES;
  static constexpr int SMEM = OFF_BAR + 256 + 1024;  // + barriers + alignment slack
  // TMEM columns: S of tile t at t*BN (fp32), P of tile t at P_COL + t*BN/2
  // (fp16 pairs), O of tile t at O_COL + t*HD (fp32)
  static constexpr uint32_t P_COL = NQ * BN;
  static constexpr uint32_t O_COL = NQ * BN + NQ * BN / 2;
  static constexpr uint32_t TMEM_COLS = NQ == 2 ? 512 : 256;
  static_assert(O_COL + NQ * HD <= TMEM_COLS, "S, P and O of every tile fit in TMEM");
  static_assert(TMEM_COLS * CTAS_PER_SM <= 512, "TMEM of the CTAs sharing an SM");
  static_assert(3 * STAGES * 8 + 5 * NQ * 8 <= 256, "barriers");
  static_assert((SMEM + 1024) * CTAS_PER_SM <= 233472, "shared memory of the CTAs sharing an SM");
};

// kind::f16 instruction descriptor: fp32 D, A/B fp16 (or bf16), A K-major,
// B K-major or MN-major (bit 16), N >> 3 at bit 17, M >> 4 at bit 24.
template <bool F16>
__host__ __device__ constexpr uint32_t idesc_attn(int m, int n, bool b_mn_major) {
  return (1u << 4) | (F16 ? 0u : (1u << 7) | (1u << 10)) | (b_mn_major ? (1u << 16) : 0u) |
         (static_cast<uint32_t>(n >> 3) << 17) | (static_cast<uint32_t>(m >> 4) << 24);
}

// MN-major operand with 128-byte swizzle: 8 K-rows of 128 bytes (64 MN
// elements) form an atom; LBO = byte stride between 64-element MN atoms,
// SBO = byte stride between 8-row K groups.
__device__ __forceinline__ uint64_t sdesc_mn_sw128(uint32_t saddr, uint32_t lbo_bytes) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo_bytes >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>(1024 >> 4) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  d |= static_cast<uint64_t>(2) << 61;
  return d;
}

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Packed fp32 pairs (two registers as one 64-bit operand) for the f32x2 FMA
// and add of the softmax: half the instructions of scalar fp32.
__device__ __forceinline__ uint64_t f2_pack(float lo, float hi) {
  uint64_t r;
  asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
  return r;
}

__device__ __forceinline__ void f2_unpack(uint64_t r, float& lo, float& hi) {
  asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(r));
}

__device__ __forceinline__ uint64_t f2_fma(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

__device__ __forceinline__ uint64_t f2_add(uint64_t a, uint64_t b) {
  uint64_t d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}

// max(a, b, c) in one instruction
__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Bounded wait that also gives up at once when another thread of the CTA
// already timed out (abort flag), so a failure cannot chain into long waits.
__device__ __forceinline__ bool wait_bar(uint64_t* bar, uint32_t parity, int32_t* status,
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

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Threads: warps 0-3 and 4-7 are the softmax warpgroups of Q tiles 0 and 1
// (thread = row of its tile, whole rows of S), warp 8 is the TMA producer and
// TMEM owner, warps 9 and 10 issue the UMMAs of Q tiles 0 and 1.  Both Q tiles
// share every K/V tile.
template <int HD, bool F16>
__global__ void __launch_bounds__(AttnCfg<HD>::THREADS, AttnCfg<HD>::CTAS_PER_SM) attn_tc_kernel(
    const uint16_t* __restrict__ q, const int32_t* __restrict__ pos, int n, int hq, int hkv,
    const int32_t* __restrict__ table, int64_t n_logical,
    const __grid_constant__ CUtensorMap pool_run, const __grid_constant__ CUtensorMap pool_blk,
    int64_t pool_blocks,
    uint16_t* __restrict__ out, float* __restrict__ part_o, float* __restrict__ part_lse,
    int keys_per_split, int n_splits, float scale_log2, int32_t* status,
    const int32_t* __restrict__ flags, long long flag_wait_cycles,
    const uint16_t* __restrict__ host_pool, int64_t host_blocks) {
  using C = AttnCfg<HD>;
  constexpr int BN = C::BN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sQ = smem;  // [NQ tiles]
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* k_full = bars;                    // [STAGES]
  uint64_t* v_full = bars + C::STAGES;        // [STAGES]
  uint64_t* kv_empty = bars + 2 * C::STAGES;  // [STAGES]
  uint64_t* s_full = bars + 3 * C::STAGES;    // [NQ tiles] S(j) in TMEM
  uint64_t* s_free = s_full + C::NQ;          // [NQ tiles] S(j) read into registers
  uint64_t* p_full = s_free + C::NQ;          // [NQ tiles] P(j) in TMEM
  uint64_t* p_free = p_full + C::NQ;          // [NQ tiles] P(j) V(j) done
  uint64_t* drain = p_free + C::NQ;           // [NQ tiles] every UMMA of the tile's issuer done
  __shared__ uint32_t s_tmem;
  __shared__ int s_maxpos;
  __shared__ int s_abort;
  volatile int* abort_flag = &s_abort;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // grid: x = KV head, y = row tile counted from the last (the longest key
  // ranges are dispatched first, so the shortest fill the tail of the grid)
  const int g = blockIdx.x;
  const int group = hq / hkv;
  const int R = n * group;
  const int r0 = (gridDim.y - 1 - blockIdx.y) * C::ROWS;
  const int split = blockIdx.z;
  // Q tiles holding at least one real row: a trailing tile of padding rows
  // (the last row tile of a short row set) gets no UMMAs and no softmax
  const int nq = min(C::NQ, (R - r0 + C::BM - 1) / C::BM);

  if (tid == 0) {
    for (int s = 0; s < C::STAGES; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&kv_empty[s], nq);  // every active Q tile's P V done
    }
    for (int t = 0; t < C::NQ; ++t) {
      mbar_init(&s_full[t], 1);
      mbar_init(&s_free[t], 4);  // one arrival per softmax warp of the tile
      mbar_init(&p_full[t], 4);
      mbar_init(&p_free[t], 1);
      mbar_init(&drain[t], 1);
    }
    fence_barrier_init();
    s_maxpos = -1;
    s_abort = 0;
    tma_prefetch_desc(&pool_run);
    tma_prefetch_desc(&pool_blk);
  }
  if (warp == C::PRODUCER_WARP) {
    tmem_alloc(&s_tmem, C::TMEM_COLS);
    tc_fence_before();  // the TMEM address, read by the other warps after the barrier below
  }
  // the prologue above touches no memory another kernel writes
  pdl_enter();

  // the producer finds the key range itself (the largest position of the
  // CTA's rows) and reads the first key tile's block-table entries while the
  // softmax warps load Q, so the first K/V fetch does not wait for Q
  int prod_kv_len = 0;
  int32_t prod_tab0 = -1;
  if (warp == C::PRODUCER_WARP) {
    const int t_lo = r0 / group, t_hi = (min(R, r0 + C::ROWS) - 1) / group;
    int mp = -1;
    for (int t = t_lo + lane; t <= t_hi; t += 32) mp = max(mp, pos[t]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) mp = max(mp, __shfl_xor_sync(0xffffffffu, mp, off));
    prod_kv_len = mp + 1;
    const int64_t blk0 = static_cast<int64_t>(split * keys_per_split) / 16 + lane;
    if (lane < BN / 16 && blk0 < n_logical) prod_tab0 = table[blk0];
  }

  // softmax threads: tile and row; the Q tiles in the UMMA K-major layout
  const int qt = tid >> 7;  // Q tile of the softmax warps
  const int row = tid & 127;
  const int rr = r0 + qt * C::BM + row;
  int row_pos = -1;
  if (warp < C::PRODUCER_WARP) {
    const int t = rr / group, h = g * group + rr % group;
    if (rr < R) row_pos = pos[t];
    uint8_t* q_tile = sQ + qt * C::Q_BYTES;
#pragma unroll
    for (int c = 0; c < HD / 8; ++c) {
      uint8_t* dst = q_tile + (c >> 3) * (C::BM * 128) + row * 128 + (((c & 7) ^ (row & 7)) << 4);
      if (rr < R)
        cp_async16(smem_u32(dst), q + (static_cast<int64_t>(t) * hq + h) * HD + c * 8);
      else
        *reinterpret_cast<uint4*>(dst) = make_uint4(0, 0, 0, 0);
    }
    cp_async_commit();
  }
  __syncthreads();  // barriers initialised, TMEM allocated
  int kv_len = prod_kv_len;
  if (warp != C::PRODUCER_WARP) {
    if (row_pos >= 0) atomicMax(&s_maxpos, row_pos);
    if (warp < C::PRODUCER_WARP) {
      cp_async_wait<0>();
      fence_async_smem();  // Q (generic-proxy writes) visible to the tensor core
    }
    tc_fence_before();
    // the softmax and UMMA warps only: Q loaded and every row position seen
    asm volatile("bar.sync 1, %0;" ::"n"(C::THREADS - 32) : "memory");
    kv_len = s_maxpos + 1;
  }
  tc_fence_after();
  const uint32_t tmem = s_tmem;
  const int k_begin = split * keys_per_split;
  const int k_end = min(kv_len, k_begin + keys_per_split);
  const int T = k_end > k_begin ? (k_end - k_begin + BN - 1) / BN : 0;

  if (warp == C::PRODUCER_WARP) {
    if (T > 0) {
      // ---- TMA producer (whole warp): lane b looks up block b of a key tile,
      // one tile ahead of its use, so the table reads overlap the copies ----
      constexpr int NB = BN / 16;
      constexpr int32_t kPast = INT32_MIN;  // block past the key range
      const int32_t yk = g * 16, yv = (hkv + g) * 16;
      auto lookup = [&](int j) -> int32_t {
        const int key0 = k_begin + j * BN + lane * 16;
        if (lane >= NB || key0 >= k_end) return kPast;
        const int64_t blk = key0 >> 4;
        return blk < n_logical ? table[blk] : -1;
      };
      // residency flags (restore copies in flight): a lane's block must have
      // landed before its keys are fetched.  The flag of the next tile's block
      // is loaded once this tile's copies are issued (its table entry has
      // arrived by then), so a flag that is already set costs no wait.
      auto flag_of = [&](int32_t pb) -> int32_t {
        return (flags == nullptr || pb < 0 || pb >= pool_blocks) ? 1 : ld_acquire_gpu(flags + pb);
      };
      // tile 0's entries were read before the barrier
      int32_t p_cur = (lane >= NB || k_begin + lane * 16 >= k_end) ? kPast : prod_tab0;
      int32_t f_cur = flag_of(p_cur);
      int issued = 0;
      for (int j = 0; j < T; ++j) {
        const int s = j % C::STAGES;
        const int32_t p_nxt = j + 1 < T ? lookup(j + 1) : kPast;
        int32_t p = p_cur;
        // a swapped block read in place: entry -2 - slot of the pinned store
        const bool host = host_pool != nullptr && p != kPast && p <= -2 &&
                          -static_cast<int64_t>(p) - 2 < host_blocks;
        if (p != kPast && !host && (p < 0 || p >= pool_blocks)) {
          set_status(status, kStatusDevice);  // its keys read another block
          p = kPast;
        }
        const bool valid = p != kPast && !host;  // fetched by TMA from the pool
        const unsigned host_lanes = __ballot_sync(0xffffffffu, host);
        const int32_t first_raw = __shfl_sync(0xffffffffu, p, 0);
        const int32_t first = first_raw < 0 ? 0 : first_raw;
        // the tile's blocks are consecutive in the pool: one box per operand slice
        // (blocks past the key range are read too; their keys are masked)
        const bool run = host_lanes == 0 && __all_sync(0xffffffffu, !valid || p == first + lane);
        const int32_t mine = valid ? p : first;
        bool ok = true;
        if (lane == 0 && j >= C::STAGES)
          ok = wait_bar(&kv_empty[s], ((j / C::STAGES) - 1) & 1, status, abort_flag);
        if (!__shfl_sync(0xffffffffu, ok, 0)) break;
        if (flags != nullptr) {
          bool rdy = !valid || f_cur != 0;
          if (!__all_sync(0xffffffffu, rdy)) {
            const long long t0 = clock64();
            while (true) {
              if (!rdy) rdy = ld_acquire_gpu(flags + p) != 0;
              if (__all_sync(0xffffffffu, rdy)) break;
              // give up at the limit, or at once when another thread of this CTA
              // or another CTA has timed out already (the status word says so)
              if (__any_sync(0xffffffffu, *abort_flag != 0 || clock64() - t0 > flag_wait_cycles ||
                                              (status != nullptr &&
                                               *reinterpret_cast<volatile int32_t*>(status) == kStatusTimeout))) {
                if (lane == 0) {
                  set_status(status, kStatusTimeout);
                  *abort_flag = 1;
                }
                ok = false;
                break;
              }
              __nanosleep(128);
            }
            if (!__all_sync(0xffffffffu, ok)) break;
          }
          fence_proxy_async_global();  // the TMA reads come after the flags were seen
        }
        uint32_t tma_bytes = C::KV_BYTES;
        if (host_lanes != 0) {
          // blocks held in pinned host memory: the warp copies their K and V
          // rows over the host link with 16-byte cp.async (plain loads, no
          // TMA) into the places the per-block TMA boxes would fill (128-byte
          // swizzle), and each lane registers its copies on the stage's
          // barriers before lane 0 arrives, so no phase completes early
          constexpr int CPR = HD / 8;  // 16-byte chunks per row
          for (unsigned hm = host_lanes; hm != 0; hm &= hm - 1) {
            const int hl = __ffs(hm) - 1;
            const int64_t hb = -static_cast<int64_t>(__shfl_sync(0xffffffffu, p, hl)) - 2;
            const uint16_t* src = host_pool + hb * (2LL * hkv * 16 * HD);
#pragma unroll 1
            for (int ci = lane; ci < 16 * CPR; ci += 32) {
              const int r = ci / CPR, cc = ci % CPR, c = cc >> 3, u = cc & 7;
              const uint32_t off = c * (BN * 128) + hl * 16 * 128 + r * 128 + ((u ^ (r & 7)) << 4);
              cp_async16(smem_u32(sK + s * C::KV_BYTES + off), src + (static_cast<int64_t>(yk + r)) * HD + cc * 8);
            }
          }
          cp_async_mbar_arrive(&k_full[s]);
          for (unsigned hm = host_lanes; hm != 0; hm &= hm - 1) {
            const int hl = __ffs(hm) - 1;
            const int64_t hb = -static_cast<int64_t>(__shfl_sync(0xffffffffu, p, hl)) - 2;
            const uint16_t* src = host_pool + hb * (2LL * hkv * 16 * HD);
#pragma unroll 1
            for (int ci = lane; ci < 16 * CPR; ci += 32) {
              const int r = ci / CPR, cc = ci % CPR, c = cc >> 3, u = cc & 7;
              const uint32_t off = c * (BN * 128) + hl * 16 * 128 + r * 128 + ((u ^ (r & 7)) << 4);
              cp_async16(smem_u32(sV + s * C::KV_BYTES + off), src + (static_cast<int64_t>(yv + r)) * HD + cc * 8);
            }
          }
          cp_async_mbar_arrive(&v_full[s]);
          tma_bytes = (NB - __popc(host_lanes)) * 16 * 128 * C::CB;
          __syncwarp();
        }
        if (lane == 0) {
          mbar_arrive_expect_tx(&k_full[s], tma_bytes);
          mbar_arrive_expect_tx(&v_full[s], tma_bytes);
        }
        __syncwarp();
        if (run) {
          if (lane == 0) {
#pragma unroll
            for (int c = 0; c < C::CB; ++c) {
              tma_load_3d(sK + s * C::KV_BYTES + c * (BN * 128), &pool_run, &k_full[s], c * 64, yk, first);
              tma_load_3d(sV + s * C::KV_BYTES + c * (BN * 128), &pool_run, &v_full[s], c * 64, yv, first);
            }
          }
        } else if (lane < NB && !host) {
#pragma unroll
          for (int c = 0; c < C::CB; ++c) {
            tma_load_3d(sK + s * C::KV_BYTES + c * (BN * 128) + lane * 16 * 128, &pool_blk, &k_full[s],
                        c * 64, yk, mine);
            tma_load_3d(sV + s * C::KV_BYTES + c * (BN * 128) + lane * 16 * 128, &pool_blk, &v_full[s],
                        c * 64, yv, mine);
          }
        }
        issued = j + 1;
        p_cur = p_nxt;
        if (flags != nullptr) f_cur = flag_of(p_cur);
      }
      // drain: every fill issued has landed before shared memory is released
      // (a bounded wait without the abort shortcut: after an abort the copies
      // already issued still land)
      if (lane == 0) {
        for (int j = issued - C::STAGES < 0 ? 0 : issued - C::STAGES; j < issued; ++j) {
          mbar_wait(&k_full[j % C::STAGES], (j / C::STAGES) & 1, status);
          mbar_wait(&v_full[j % C::STAGES], (j / C::STAGES) & 1, status);
        }
      }
    }
  } else if (warp > C::PRODUCER_WARP) {
    // ---- UMMA issuers, one per Q tile t: S_t(j+1), then P_t V(j) ----
    const int t = warp - C::PRODUCER_WARP - 1;
    if (lane == 0 && T > 0 && t < nq) {
      constexpr uint32_t id_s = idesc_attn<F16>(128, BN, false);
      constexpr uint32_t id_o = idesc_attn<F16>(128, HD, true);
      const uint32_t q_base = smem_u32(sQ + t * C::Q_BYTES);
      const uint32_t k_base = smem_u32(sK), v_base = smem_u32(sV);
      const uint32_t s_tm = tmem + t * BN, p_tm = tmem + C::P_COL + t * (BN / 2);
      const uint32_t o_tm = tmem + C::O_COL + t * HD;
      auto issue_s = [&](int j) {
        const uint32_t kst = k_base + (j % C::STAGES) * C::KV_BYTES;
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const int cb = kk >> 2, w = kk & 3;
          umma_f16(s_tm, sdesc_k_sw128(q_base + cb * (C::BM * 128) + w * 32),
                   sdesc_k_sw128(kst + cb * (BN * 128) + w * 32), id_s, kk > 0 ? 1u : 0u);
        }
        umma_commit(&s_full[t]);
      };
      auto issue_pv = [&](int j) {
        const int s = j % C::STAGES;
        const uint32_t vst = v_base + s * C::KV_BYTES;
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk)
          umma_f16_ts(o_tm, p_tm + kk * 8, sdesc_mn_sw128(vst + kk * 16 * 128, BN * 128), id_o,
                      (j > 0 || kk > 0) ? 1u : 0u);
        umma_commit(&p_free[t]);
        umma_commit(&kv_empty[s]);
      };
      bool ok = wait_bar(&k_full[0], 0, status, abort_flag);
      if (ok) {
        tc_fence_after();
        if (host_pool != nullptr) fence_async_smem();
        issue_s(0);
      }
      for (int j = 0; ok && j < T; ++j) {
        const uint32_t ph = j & 1;
        if (j + 1 < T) {
          // the next S runs while the softmax exponentiates S(j)
          if (!wait_bar(&k_full[(j + 1) % C::STAGES], ((j + 1) / C::STAGES) & 1, status, abort_flag)) break;
          if (!wait_bar(&s_free[t], ph, status, abort_flag)) break;
          tc_fence_after();
          if (host_pool != nullptr) fence_async_smem();  // cp.async-written K before the UMMA reads it
          issue_s(j + 1);
        }
        if (!wait_bar(&v_full[j % C::STAGES], (j / C::STAGES) & 1, status, abort_flag)) break;
        if (!wait_bar(&p_full[t], ph, status, abort_flag)) break;
        tc_fence_after();
        if (host_pool != nullptr) fence_async_smem();  // ... and V
        issue_pv(j);
      }
      // every UMMA this thread issued has completed before TMEM is released
      // (after an abort the softmax warps do not wait for the last ones)
      umma_commit(&drain[t]);
      mbar_wait(&drain[t], 0, status);
    }
  } else {
    // ---- softmax: thread = row of Q tile qt, all BN columns ----
    const uint32_t trow = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
    const uint32_t s_col = qt * BN, p_col = C::P_COL + qt * (BN / 2), o_col = C::O_COL + qt * HD;
    float m_ref = -INFINITY, l = 0.0f;
    bool ok = true;
    const int Tq = qt < nq ? T : 0;  // key tiles this Q tile processes
    for (int j = 0; j < Tq && ok; ++j) {
      const uint32_t ph = j & 1;
      const int kb = k_begin + j * BN;
      ok = wait_bar(&s_full[qt], ph, status, abort_flag);
      __syncwarp();
      if (!__all_sync(0xffffffffu, ok)) {
        ok = false;
        break;
      }
      tc_fence_after();
      float v[BN];
      float hmax = -INFINITY;  // the row's maximum, reduced by the TMEM loads
#pragma unroll
      for (int c = 0; c < BN; c += 64) {
        float h;
        tmem_ld64w_max(trow + s_col + c, v + c, h);
        hmax = fmaxf(hmax, h);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[qt]);
      const bool full = __all_sync(0xffffffffu, (kb + BN - 1 <= row_pos) && (kb + BN <= k_end));
      float tmax;
      if (full) {
        tmax = hmax * scale_log2;
      } else {
        // diagonal or ragged tile: mask, then reduce in registers
#pragma unroll
        for (int i = 0; i < BN; ++i) {
          const int key = kb + i;
          if (!(key <= row_pos && key < k_end)) v[i] = -INFINITY;
        }
        float mx[8];
#pragma unroll
        for (int a = 0; a < 8; ++a) mx[a] = fmaxf(v[2 * a], v[2 * a + 1]);
#pragma unroll
        for (int i = 16; i < BN; i += 16) {
#pragma unroll
          for (int a = 0; a < 8; ++a) mx[a] = fmax3(mx[a], v[i + 2 * a], v[i + 2 * a + 1]);
        }
        tmax = fmax3(fmax3(mx[0], mx[1], mx[2]), fmax3(mx[3], mx[4], mx[5]), fmaxf(mx[6], mx[7])) *
               scale_log2;
      }
      const float m_new = fmaxf(m_ref, tmax);
      const bool need = m_new > m_ref + 8.0f;
      const float m_old = m_ref;
      if (need) m_ref = m_new;
      const float nbase = m_ref == -INFINITY ? 0.0f : -m_ref;
      // P(j) goes to registers first, so the exponentials run while P(j-1) V(j-1)
      // still reads the P buffer
      uint32_t pk[BN / 2];
      const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nb2 = f2_pack(nbase, nbase);
      uint64_t ls2[2] = {f2_pack(0.f, 0.f), f2_pack(0.f, 0.f)};
#pragma unroll
      for (int i = 0; i < BN / 2; ++i) {
        float x0, x1;
        f2_unpack(f2_fma(f2_pack(v[2 * i], v[2 * i + 1]), sc2, nb2), x0, x1);
        const float p0 = ex2(x0), p1 = ex2(x1);
        ls2[i & 1] = f2_add(ls2[i & 1], f2_pack(p0, p1));
        pk[i] = pack2<F16>(p0, p1);
      }
      // P(j-1) V(j-1) must be done before O is rebased or P is overwritten
      if (j > 0) {
        ok = wait_bar(&p_free[qt], (j - 1) & 1, status, abort_flag);
        __syncwarp();
        if (!__all_sync(0xffffffffu, ok)) {
          ok = false;
          break;
        }
        tc_fence_after();
        if (__any_sync(0xffffffffu, need)) {
          const float alpha = need ? ex2(m_old - m_ref) : 1.0f;
#pragma unroll 1
          for (int c = 0; c < HD; c += 32) {
            float o[32];
            tmem_ld32w(trow + o_col + c, o);
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32w(trow + o_col + c, o);
          }
          l *= alpha;
        }
      }
      {
        float a0, a1, b0, b1;
        f2_unpack(ls2[0], a0, a1);
        f2_unpack(ls2[1], b0, b1);
        l += (a0 + a1) + (b0 + b1);
      }
      if constexpr (BN == 128) {
        tmem_st64w_u32(trow + p_col, pk);
      } else {
        tmem_st32w_u32(trow + p_col, pk);
      }
      tc_fence_before();  // P in TMEM before the issuer's P V
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[qt]);
    }
    // ---- epilogue: O / l ----
    bool have_o = false;
    if (ok && Tq > 0) {
      ok = wait_bar(&p_free[qt], (Tq - 1) & 1, status, abort_flag);
      __syncwarp();
      have_o = __all_sync(0xffffffffu, ok);
      tc_fence_after();
    }
    const float o_scale = l > 0.0f ? 1.0f / l : 0.0f;
    const int t = rr / group, h = g * group + rr % group;
    const int64_t orow = static_cast<int64_t>(t) * hq + h;
    // At head dim 128 the warp's 32 rows go through its quarter of the
    // tile's Q shared memory (every UMMA that reads it has completed: S(Tq-1)
    // before the softmax loaded it), HD x 2 bytes a row per pass, 16-byte
    // units XOR-swizzled by row; then each store instruction writes whole
    // rows, where a thread storing its own row touches 32 rows per
    // instruction (measured 1-3% faster at head dim 128, 2% slower at 64,
    // whose kernel is short of registers).  After an abort the tile's UMMAs
    // may still read Q, and nothing is written.
    constexpr int U = HD / 8;  // 16-byte units of a staged row
    uint4* stg = reinterpret_cast<uint4*>(sQ + qt * C::Q_BYTES) + (warp & 3) * 32 * U;
    const int wr0 = r0 + qt * C::BM + (warp & 3) * 32;  // tile row of lane 0
    const bool write_rows = Tq == 0 || have_o;
    auto store_rows = [&](auto dst_row) {
      __syncwarp();
#pragma unroll 4
      for (int it = 0; it < U; ++it) {
        const int k = it * 32 + lane, rw = k / U, un = k % U;
        const int rrw = wr0 + rw;
        if (rrw < R) {
          const int64_t orw = static_cast<int64_t>(rrw / group) * hq + g * group + rrw % group;
          dst_row(orw)[un] = stg[rw * U + (un ^ (rw & (U - 1)))];
        }
      }
      __syncwarp();
    };
    if (HD == 64 && write_rows) {
#pragma unroll
      for (int c = 0; c < HD; c += 64) {
        float o[64];
        if (have_o) {
          tmem_ld64w(trow + o_col + c, o);
        } else {
#pragma unroll
          for (int i = 0; i < 64; ++i) o[i] = 0.0f;
        }
        if (rr < R) {
          if (n_splits == 1) {
            uint4* dst = reinterpret_cast<uint4*>(out + orow * HD + c);
#pragma unroll
            for (int u = 0; u < 8; ++u)
              dst[u] = make_uint4(pack2<true>(o[8 * u] * o_scale, o[8 * u + 1] * o_scale),
                                  pack2<true>(o[8 * u + 2] * o_scale, o[8 * u + 3] * o_scale),
                                  pack2<true>(o[8 * u + 4] * o_scale, o[8 * u + 5] * o_scale),
                                  pack2<true>(o[8 * u + 6] * o_scale, o[8 * u + 7] * o_scale));
          } else {
            float4* dst = reinterpret_cast<float4*>(
                part_o + (static_cast<int64_t>(split) * n * hq + orow) * HD + c);
#pragma unroll
            for (int u = 0; u < 16; ++u)
              dst[u] = make_float4(o[4 * u] * o_scale, o[4 * u + 1] * o_scale,
                                   o[4 * u + 2] * o_scale, o[4 * u + 3] * o_scale);
          }
        }
      }
    } else if (write_rows && n_splits == 1) {
#pragma unroll
      for (int c = 0; c < HD; c += 64) {
        float o[64];
        if (have_o) {
          tmem_ld64w(trow + o_col + c, o);
        } else {
#pragma unroll
          for (int i = 0; i < 64; ++i) o[i] = 0.0f;
        }
#pragma unroll
        for (int u = 0; u < 8; ++u)
          stg[lane * U + ((c / 8 + u) ^ (lane & (U - 1)))] =
              make_uint4(pack2<true>(o[8 * u] * o_scale, o[8 * u + 1] * o_scale),
                         pack2<true>(o[8 * u + 2] * o_scale, o[8 * u + 3] * o_scale),
                         pack2<true>(o[8 * u + 4] * o_scale, o[8 * u + 5] * o_scale),
                         pack2<true>(o[8 * u + 6] * o_scale, o[8 * u + 7] * o_scale));
      }
      store_rows([&](int64_t orw) { return reinterpret_cast<uint4*>(out + orw * HD); });
    } else if (write_rows) {
      // fp32 partials: two passes of HD/2 columns
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        float o[HD / 2];
        if (have_o) {
          if constexpr (HD == 128) {
            tmem_ld64w(trow + o_col + half * 64, o);
          } else {
            tmem_ld32w(trow + o_col + half * 32, o);  // not reached: head dim 64 stores directly
          }
        } else {
#pragma unroll
          for (int i = 0; i < HD / 2; ++i) o[i] = 0.0f;
        }
#pragma unroll
        for (int u = 0; u < U; ++u)
          stg[lane * U + (u ^ (lane & (U - 1)))] = make_uint4(
              __float_as_uint(o[4 * u] * o_scale), __float_as_uint(o[4 * u + 1] * o_scale),
              __float_as_uint(o[4 * u + 2] * o_scale), __float_as_uint(o[4 * u + 3] * o_scale));
        store_rows([&](int64_t orw) {
          return reinterpret_cast<uint4*>(part_o + (static_cast<int64_t>(split) * n * hq + orw) * HD +
                                          half * (HD / 2));
        });
      }
    }
    if (write_rows && rr < R && n_splits > 1)
      part_lse[static_cast<int64_t>(split) * n * hq + orow] = l > 0.0f ? m_ref + log2f(l) : -INFINITY;
  }

  tc_fence_before();
  __syncthreads();
  if (warp == C::PRODUCER_WARP) {
    __syncwarp();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// out[row] = sum_s 2^(lse_s - lse_max) o_s / sum_s 2^(lse_s - lse_max); one warp per row.
// Lane s holds split s's log-sum-exp and weight (n_splits <= 64: two per lane),
// and the partial rows are read eight splits at a time, so the loads of the
// splits overlap instead of queueing one after another.
template <int HD>
__global__ void attn_combine_kernel(const float* __restrict__ part_o,
                                    const float* __restrict__ part_lse, int64_t rows, int n_splits,
                                    uint16_t* __restrict__ out) {
  pdl_enter();
  const int64_t row = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const float l0 = lane < n_splits ? part_lse[lane * rows + row] : -INFINITY;
  const float l1 = lane + 32 < n_splits ? part_lse[(lane + 32) * rows + row] : -INFINITY;
  float mx = fmaxf(l0, l1);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  const float w0 = (l0 == -INFINITY) ? 0.0f : exp2f(l0 - mx);  // mx is finite when any l is
  const float w1 = (l1 == -INFINITY) ? 0.0f : exp2f(l1 - mx);
  float wsum = w0 + w1;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) wsum += __shfl_xor_sync(0xffffffffu, wsum, off);
  constexpr int PER = HD / 32;
  using Vec = typename std::conditional<PER == 4, float4, float2>::type;
  float acc[PER];
#pragma unroll
  for (int j = 0; j < PER; ++j) acc[j] = 0.0f;
  // eight splits' rows are loaded before any is used, so their loads overlap;
  // an empty split has weight 0 and rows of zeros
  for (int s0 = 0; s0 < n_splits; s0 += 8) {
    Vec v[8];
    float w[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int s = s0 + j;
      const bool in = s < n_splits;  // uniform over the warp
      w[j] = in ? __shfl_sync(0xffffffffu, s < 32 ? w0 : w1, s & 31) : 0.0f;
      if (in) {
        v[j] = *reinterpret_cast<const Vec*>(part_o + (s * rows + row) * HD + lane * PER);
      } else {
        float* z = reinterpret_cast<float*>(&v[j]);
#pragma unroll
        for (int e = 0; e < PER; ++e) z[e] = 0.0f;
      }
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const float* f = reinterpret_cast<const float*>(&v[j]);
#pragma unroll
      for (int e = 0; e < PER; ++e) acc[e] = fmaf(w[j], f[e], acc[e]);
    }
  }
  const float inv = wsum > 0.0f ? 1.0f / wsum : 0.0f;
  uint16_t* dst = out + row * HD + lane * PER;
#pragma unroll
  for (int j = 0; j < PER; j += 2)
    *reinterpret_cast<uint32_t*>(dst + j) = pack2<true>(acc[j] * inv, acc[j + 1] * inv);
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
    cudaDriverEntryPointQueryResult qr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &qr) == cudaSuccess &&
        qr == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

// The pool as a 3-D tensor of 16-bit elements: [pool_blocks][2 * hkv * 16 rows][hd]
// (K rows of every head, then V rows), read in boxes of `depth` blocks x 16 rows
// (one head) x 64 columns with 128-byte swizzle.
bool make_pool_map(CUtensorMap* map, const void* pool, int64_t pool_blocks, int hkv, int hd,
                   int depth) {
  EncodeFn fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t rows = static_cast<cuuint64_t>(2) * hkv * 16;
  cuuint64_t dims[3] = {static_cast<cuuint64_t>(hd), rows, static_cast<cuuint64_t>(pool_blocks)};
  cuuint64_t strides[2] = {static_cast<cuuint64_t>(hd) * 2, rows * hd * 2};
  cuuint32_t box[3] = {64, 16, static_cast<cuuint32_t>(depth)};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_UINT16, 3, const_cast<void*>(pool), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int HD, bool F16>
cudaError_t launch_hd(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq, int32_t hkv,
                      const int32_t* table, int64_t n_logical, const void* pool,
                      int64_t pool_blocks, uint16_t* out, float* part_o, float* part_lse,
                      int n_splits, int keys_per_split, int32_t* status, const int32_t* flags,
                      long long flag_wait, const uint16_t* host_pool, int64_t host_blocks,
                      cudaStream_t st) {
  using C = AttnCfg<HD>;
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    attr_err = cudaFuncSetAttribute(attn_tc_kernel<HD, F16>,
                                    cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  });
  if (attr_err != cudaSuccess) return attr_err;
  CUtensorMap run_map, blk_map;
  if (!make_pool_map(&run_map, pool, pool_blocks, hkv, HD, C::BN / 16) ||
      !make_pool_map(&blk_map, pool, pool_blocks, hkv, HD, 1))
    return cudaErrorInvalidValue;
  const int group = hq / hkv;
  const int64_t R = n * group;
  const int64_t row_tiles = (R + C::ROWS - 1) / C::ROWS;
  if (row_tiles > 65535) return cudaErrorInvalidValue;
  dim3 grid(static_cast<unsigned>(hkv), static_cast<unsigned>(row_tiles), static_cast<unsigned>(n_splits));
  const float scale_log2 =
      static_cast<float>(1.0 / std::sqrt(static_cast<double>(HD)) * 1.4426950408889634);
  launch_k(attn_tc_kernel<HD, F16>, dim3(grid), dim3(C::THREADS), C::SMEM, st,
      q, pos, static_cast<int>(n), hq, hkv, table, n_logical, run_map, blk_map, pool_blocks, out, part_o,
      part_lse, keys_per_split, n_splits, scale_log2, status, flags, flag_wait, host_pool, host_blocks);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess || n_splits == 1) return e;
  const int64_t rows = n * hq;
  launch_k(attn_combine_kernel<HD>, dim3(static_cast<unsigned>((rows + 7) / 8)), dim3(256), 0, st,
      part_o, part_lse, rows, n_splits, out);
  return cudaGetLastError();
}

}  // namespace

void attention_split(int64_t n, int32_t hq, int32_t hkv, int32_t hd, int64_t max_keys, int num_sms,
                     int* n_splits, int* keys_per_split) {
  if (attention_decode_applies(n, hq, hkv, hd)) {
    attention_decode_split(hkv, max_keys, num_sms, n_splits, keys_per_split);
    return;
  }
  const int rows_per_cta = hd == 64 ? AttnCfg<64>::ROWS : AttnCfg<128>::ROWS;
  const int slots = num_sms * (hd == 64 ? AttnCfg<64>::CTAS_PER_SM : AttnCfg<128>::CTAS_PER_SM);
  const int64_t ctas = ((n * (hq / hkv) + rows_per_cta - 1) / rows_per_cta) * hkv;
  int s = 1;
  if (ctas < slots && max_keys > 1024) {
    // fewer CTAs than resident slots: more splits fill the waves better, but
    // each split writes a partial output and log-sum-exp that the combine
    // reads back, and a split of ~512 keys is mostly that fixed cost.  So a
    // larger split count is taken only when its waves are at least 10%
    // fuller, with at least 1024 keys per split.  (Taking every tie toward
    // more splits once turned 144 CTAs into 19 splits of 512 keys for a 5%
    // fuller wave: the 3B f = 0.75 step with 1536 recomputed rows went from
    // 13.0 to 20.8 ms.)
    const int64_t max_s = std::min<int64_t>(64, (max_keys + 1023) / 1024);
    double best = 0.0;
    for (int64_t c = 1; c <= max_s; ++c) {
      const int64_t total = ctas * c;
      const int64_t waves = (total + slots - 1) / slots;
      const double eff = static_cast<double>(total) / static_cast<double>(waves * slots);
      if (c == 1 || eff > best * 1.1) {
        best = eff;
        s = static_cast<int>(c);
      }
      if (waves > 1 && eff < best) break;
    }
  }
  int64_t per = (max_keys + s - 1) / s;
  per = (per + 127) / 128 * 128;  // whole key tiles of either head size
  if (per < 128) per = 128;
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
                             int64_t max_keys, int num_sms, int32_t* status, cudaStream_t st,
                             const int32_t* flags, int64_t flag_wait_cycles, const void* host_pool,
                             int64_t host_blocks) {
  if (n <= 0) return cudaSuccess;
  const long long fw = flag_wait_cycles > 0 ? flag_wait_cycles : kWaitCycles;
  int s = 1, per = 0;
  attention_split(n, hq, hkv, hd, max_keys, num_sms, &s, &per);
  // the combine reads the partials as 8- or 16-byte vectors
  if (s > 1 && (scratch == nullptr || scratch_bytes < attention_scratch_bytes(n, hq, hd, s) ||
                reinterpret_cast<uintptr_t>(scratch) % 16 != 0)) {
    s = 1;
    per = static_cast<int>((max_keys + 127) / 128 * 128);  // whole 16-token blocks too
  }
  float* part_o = static_cast<float*>(scratch);
  float* part_lse = s > 1 ? part_o + static_cast<int64_t>(s) * n * hq * hd : nullptr;
  (void)kv_dtype;  // the pool is fp16-encoded for both KV types: q, K, P, V are fp16
  if (attention_decode_applies(n, hq, hkv, hd)) {
    cudaError_t e = launch_attention_decode(q, pos, n, hq, hkv, hd, table, n_logical, pool, pool_blocks, out,
                                            part_o, part_lse, s, per, status, flags, fw,
                                            static_cast<const uint16_t*>(host_pool), host_blocks, st);
    if (e != cudaSuccess || s == 1) return e;
    const int64_t rows = n * hq;
    if (hd == 64)
      launch_k(attn_combine_kernel<64>, dim3(static_cast<unsigned>((rows + 7) / 8)), dim3(256), 0, st, part_o, part_lse, rows, s, out);
    else
      launch_k(attn_combine_kernel<128>, dim3(static_cast<unsigned>((rows + 7) / 8)), dim3(256), 0, st, part_o, part_lse, rows, s, out);
    return cudaGetLastError();
  }
  if (hd == 64)
    return launch_hd<64, true>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks, out,
                               part_o, part_lse, s, per, status, flags, fw,
                               static_cast<const uint16_t*>(host_pool), host_blocks, st);
  if (hd == 128)
    return launch_hd<128, true>(q, pos, n, hq, hkv, table, n_logical, pool, pool_blocks, out,
                                part_o, part_lse, s, per, status, flags, fw,
                                static_cast<const uint16_t*>(host_pool), host_blocks, st);
  return cudaErrorInvalidValue;
}

}  // namespace mzc
