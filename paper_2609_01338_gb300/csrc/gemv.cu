// Projections of one to four rows (decode steps): out[m][n] = epilogue(sum_k
// A[m][k] W[n][k]) with the weight matrix streamed once from HBM.  At these
// row counts the product is bound by the weight bytes; the tensor-core GEMM
// would pad every row to a 128-row tile and keep only its ring of weight
// tiles in flight per SM.  Here one warp owns one output row of W (SwiGLU:
// the gate and up rows of one output column), reads it with 16-byte
// non-caching loads, several in flight per lane, and reduces with shuffles;
// the few activation rows come through L1.  fp32 accumulation; the
// epilogues are the GEMM's (fp16 store, fp32 residual add, SwiGLU).
//
// Folded RMSNorm for one row (RowNorm; decode steps and the last layer's
// logits row): the residual-add form (NORM = 1) also writes h = fp16(x * g)
// for its outputs and one partial sum of x^2 per CTA (its outputs summed in
// slot order) at ss[blockIdx.x]; the fp16-store and SwiGLU forms (NORM = 2)
// load the producer's nt partials at their start (at most kGemvNormMax), sum
// them after the main loop in a fixed order (per thread, then a shuffle tree,
// then the warps in order; every CTA gets the same bits) and scale their
// outputs by rsqrt(sum / d + eps).
#include <cuda_fp16.h>

#include "kernels.hpp"
#include "ptx.cuh"

namespace mzc {

namespace {

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float dot8(const uint4& w, const uint4& a) {
  const __half2* wh = reinterpret_cast<const __half2*>(&w);
  const __half2* ah = reinterpret_cast<const __half2*>(&a);
  float s = 0.0f;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 wf = __half22float2(wh[i]), af = __half22float2(ah[i]);
    s = fmaf(wf.x, af.x, s);
    s = fmaf(wf.y, af.y, s);
  }
  return s;
}

__device__ __forceinline__ float silu_g(float g) { return g / (1.0f + __expf(-g)); }

// R weight rows per output (2 for SwiGLU), MR activation rows (m <= MR), and
// KS warps per output, each over a contiguous 1/KS of K: a CTA of 8 warps holds
// 8 / KS outputs, and the KS partial sums meet in shared memory, added in
// warp order (the same sum on every run).  Splitting K keeps each warp's chain
// of dependent load rounds short and puts more weight bytes in flight.
template <int EPI, int MR, int KS, int NORM = 0>
__global__ void __launch_bounds__(256) gemv_kernel(const uint16_t* __restrict__ a,
                                                   const uint16_t* __restrict__ w,
                                                   void* __restrict__ out, int m, int n, int k,
                                                   int32_t* status, const RowNorm rn) {
  pdl_enter();
  constexpr int R = EPI == EPI_SWIGLU_BF16 ? 2 : 1;
  constexpr int OUTS = 8 / KS;  // outputs per CTA
  static_assert(NORM == 0 || MR == 1, "the folded norm is for one row");
  constexpr int NQ = kGemvNormMax / 256;  // partials per thread (consumer)
  __shared__ float part[8][R][MR];
  __shared__ float s_norm[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float pv[NORM == 2 ? NQ : 1];
  if constexpr (NORM == 2) {
    // the producer's partial sums of squares, loaded now, summed after the
    // main loop (their latency hides under the weight stream)
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
      const int idx = threadIdx.x + 256 * q;
      pv[q] = idx < rn.nt ? rn.ss[idx] : 0.0f;
    }
  }
  const int slot = warp / KS, ks = warp % KS;
  const int j = blockIdx.x * OUTS + slot;
  const int n_out = EPI == EPI_SWIGLU_BF16 ? n / 2 : n;
  const bool valid = j < n_out;
  int rows[R];
  if constexpr (EPI == EPI_SWIGLU_BF16) {
    rows[0] = (j / kSwigluGroup) * 2 * kSwigluGroup + j % kSwigluGroup;  // gate
    rows[1] = rows[0] + kSwigluGroup;                                    // up
  } else {
    rows[0] = j;
  }
  float acc[R][MR];
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int i = 0; i < MR; ++i) acc[r][i] = 0.0f;
  const int chunks = k / 8;  // 16-byte chunks per row
  const int c_begin = static_cast<int>(static_cast<int64_t>(ks) * chunks / KS);
  const int c_end = valid ? static_cast<int>(static_cast<int64_t>(ks + 1) * chunks / KS) : c_begin;
  constexpr int U = 4;  // chunks in flight per lane and row
  for (int c0 = c_begin + lane; c0 < c_end; c0 += 32 * U) {
    uint4 wv[R][U];
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int c = c0 + 32 * u;
        wv[r][u] = c < c_end ? ld_stream(reinterpret_cast<const uint4*>(w + static_cast<int64_t>(rows[r]) * k) + c)
                             : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int c = c0 + 32 * u;
      if (c >= c_end) break;
#pragma unroll
      for (int i = 0; i < MR; ++i) {
        if (i >= m) break;
        const uint4 av = __ldg(reinterpret_cast<const uint4*>(a + static_cast<int64_t>(i) * k) + c);
#pragma unroll
        for (int r = 0; r < R; ++r) acc[r][i] += dot8(wv[r][u], av);
      }
    }
  }
#pragma unroll
  for (int r = 0; r < R; ++r)
#pragma unroll
    for (int i = 0; i < MR; ++i)
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) acc[r][i] += __shfl_xor_sync(0xffffffffu, acc[r][i], o);
  if constexpr (NORM == 2) {
    float t = 0.0f;
#pragma unroll
    for (int q = 0; q < NQ; ++q) t += pv[q];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) s_norm[warp] = t;
    __syncthreads();
    float sum = 0.0f;
#pragma unroll
    for (int q = 0; q < 8; ++q) sum += s_norm[q];
    const float rs = rsqrtf(sum / rn.d + rn.eps);
#pragma unroll
    for (int r = 0; r < R; ++r) acc[r][0] *= rs;  // the per-warp K parts scale alike
  }
  if constexpr (NORM == 1) {
    // residual add with the folded norm's outputs: every thread reaches the
    // CTA barrier below, so no thread leaves early
    if constexpr (KS > 1) {
      if (lane == 0) part[warp][0][0] = acc[0][0];
      __syncthreads();
    }
    const bool writer = ks == 0 && lane == 0;
    float ysq = 0.0f;
    if (writer && valid) {
      float t = acc[0][0];
#pragma unroll
      for (int q = 1; q < KS; ++q) t += part[warp + q][0][0];
      float* o = static_cast<float*>(out) + j;
      const float y = *o + t;
      *o = y;
      const float hv = y * rn.g[j];
      if (fabsf(hv) >= kF16Overflow) set_status(status, kStatusOverflow);
      reinterpret_cast<__half*>(rn.h)[j] = __float2half_rn(hv);
      ysq = y * y;
    }
    if (writer) s_norm[slot] = ysq;
    __syncthreads();
    if (threadIdx.x == 0) {
      float sum = 0.0f;
#pragma unroll
      for (int q = 0; q < OUTS; ++q) sum += s_norm[q];
      rn.ss[blockIdx.x] = sum;
    }
    return;
  }
  if constexpr (KS > 1) {
    if (lane == 0) {
#pragma unroll
      for (int r = 0; r < R; ++r)
#pragma unroll
        for (int i = 0; i < MR; ++i) part[warp][r][i] = acc[r][i];
    }
    __syncthreads();
    if (ks != 0 || lane != 0) return;
#pragma unroll
    for (int r = 0; r < R; ++r)
#pragma unroll
      for (int i = 0; i < MR; ++i) {
        float t = part[warp][r][i];
#pragma unroll
        for (int q = 1; q < KS; ++q) t += part[warp + q][r][i];
        acc[r][i] = t;
      }
  } else {
    if (lane != 0) return;
  }
  if (!valid) return;
#pragma unroll
  for (int i = 0; i < MR; ++i) {
    if (i >= m) break;
    if constexpr (EPI == EPI_STORE_BF16) {
      if (fabsf(acc[0][i]) >= kF16Overflow) set_status(status, kStatusOverflow);
      static_cast<__half*>(out)[static_cast<int64_t>(i) * n + j] = __float2half_rn(acc[0][i]);
    } else if constexpr (EPI == EPI_ADD_F32) {
      static_cast<float*>(out)[static_cast<int64_t>(i) * n + j] += acc[0][i];
    } else {
      const float y = silu_g(acc[0][i]) * acc[1][i];
      if (fabsf(y) >= kF16Overflow) set_status(status, kStatusOverflow);
      static_cast<__half*>(out)[static_cast<int64_t>(i) * n_out + j] = __float2half_rn(y);
    }
  }
}

template <int EPI, int MR, int KS, int NORM = 0>
cudaError_t launch_mrk(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                       int64_t k, int32_t* status, cudaStream_t st, const RowNorm& rn) {
  const int64_t n_out = EPI == EPI_SWIGLU_BF16 ? n / 2 : n;
  constexpr int OUTS = 8 / KS;
  launch_k(gemv_kernel<EPI, MR, KS, NORM>, dim3(static_cast<unsigned>((n_out + OUTS - 1) / OUTS)), dim3(256), 0,
           st, a, w, out, static_cast<int>(m), static_cast<int>(n), static_cast<int>(k), status, rn);
  return cudaGetLastError();
}

// K split per output: outputs of 6 KB of weights and more take two warps
// (3B decode step: 2.68 -> 2.58 ms on one box; four warps for the 16 KB down
// rows measured 2.64).
int gemv_ks(int64_t k, int epilogue) {
  const int64_t bytes = k * 2 * (epilogue == EPI_SWIGLU_BF16 ? 2 : 1);  // weight bytes of one output
  return bytes >= 6144 ? 2 : 1;
}

template <int EPI, int MR, int NORM = 0>
cudaError_t launch_mr(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                      int64_t k, int32_t* status, cudaStream_t st, const RowNorm& rn) {
  if (gemv_ks(k, EPI) == 2) return launch_mrk<EPI, MR, 2, NORM>(a, w, out, m, n, k, status, st, rn);
  return launch_mrk<EPI, MR, 1, NORM>(a, w, out, m, n, k, status, st, rn);
}

template <int EPI>
cudaError_t launch_epi(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                       int64_t k, int32_t* status, cudaStream_t st, const RowNorm* rn) {
  if (rn != nullptr) {
    // one row, with the folded norm: producer (residual add) or consumer
    if constexpr (EPI == EPI_ADD_F32) return launch_mr<EPI, 1, 1>(a, w, out, m, n, k, status, st, *rn);
    else return launch_mr<EPI, 1, 2>(a, w, out, m, n, k, status, st, *rn);
  }
  const RowNorm none{};
  return m == 1 ? launch_mr<EPI, 1>(a, w, out, m, n, k, status, st, none)
                : launch_mr<EPI, 4>(a, w, out, m, n, k, status, st, none);
}

}  // namespace

int64_t gemv_norm_tiles(int64_t n, int64_t k) {
  return (n + 8 / gemv_ks(k, EPI_ADD_F32) - 1) / (8 / gemv_ks(k, EPI_ADD_F32));
}

cudaError_t launch_gemv(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                        int64_t k, int epilogue, int32_t* status, cudaStream_t st, const RowNorm* rn) {
  if (m <= 0) return cudaSuccess;
  if (m > kGemvMaxRows || k % 8 != 0) return cudaErrorInvalidValue;
  if (rn != nullptr) {
    // the folded norm takes one row; the producer's partials are one per CTA
    if (m != 1 || rn->ss == nullptr || rn->nt <= 0 || rn->nt > kGemvNormMax) return cudaErrorInvalidValue;
    if (epilogue == EPI_ADD_F32 && (rn->h == nullptr || rn->g == nullptr || rn->nt != gemv_norm_tiles(n, k)))
      return cudaErrorInvalidValue;
  }
  switch (epilogue) {
    case EPI_STORE_BF16:
      return launch_epi<EPI_STORE_BF16>(a, w, out, m, n, k, status, st, rn);
    case EPI_ADD_F32:
      return launch_epi<EPI_ADD_F32>(a, w, out, m, n, k, status, st, rn);
    case EPI_SWIGLU_BF16:
      return launch_epi<EPI_SWIGLU_BF16>(a, w, out, m, n, k, status, st, rn);
    default:
      return cudaErrorInvalidValue;
  }
}

}  // namespace mzc
