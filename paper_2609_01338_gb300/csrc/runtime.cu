// libmzc runtime: the C ABI of include/mzc.h.
//
// A ctx owns, on one device:
//   - the weights, one contiguous slot per layer (QKV rows q|k|v, O, gate/up
//     interleaved in groups of 64 rows, down padded to a multiple of 64
//     features), so that evicting or restoring a layer's weights is one copy
//     (the paper's per-layer weight unit, Sec. 4.2);
//   - the KV block pool: physical block b holds one layer's K [hkv][16][hd]
//     then V [hkv][16][hd] for 16 positions; the per-layer block tables map
//     logical blocks to physical ones (the chunk-pointer array, Sec. 4.2);
//   - activations for max_rows rows, split-KV scratch, rotary tables;
//   - a compute stream and a copy stream, with per-layer events recorded by
//     the restore on the copy stream; each layer's attention waits only on
//     its own layer's event (zero-wait, Sec. 4.4);
//   - the pinned swap store (allocated on the first COPY eviction) and the
//     pinned master copies of evicted layer weights.
// Host bookkeeping (residency, allocation, restore planning) is state.cpp.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "kernels.hpp"
#include "mzc.h"
#include "state.hpp"

using mzc::ceil_div;

namespace {

thread_local std::string g_create_error;

struct LayerDev {
  uint8_t* base = nullptr;  // slot start (device)
  size_t bytes = 0;
  uint16_t *wqkv = nullptr, *wo = nullptr, *w13 = nullptr, *w2 = nullptr;
  float *attn_norm = nullptr, *ffn_norm = nullptr;
  mzc::GemmWeight tm_qkv, tm_o, tm_13, tm_2;
  uint8_t* host_master = nullptr;  // pinned, allocated on first eviction
};

size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

mzc_profile default_profile() {
  mzc_profile p;
  p.h2d_gbs = 200.0;
  p.gemm_us_128 = 110.0;
  p.gemm_us_512 = 260.0;
  p.gemm_us_2048 = 700.0;
  p.attn_tflops = 800.0;
  p.attn_row_ns = 2000.0;
  p.attn_prompt_tflops = 500.0;
  p.row_ns = 150.0;
  p.layer_us = 15.0;
  return p;
}

}  // namespace

struct mzc_ctx {
  mzc::State st;
  mzc_model_shape shape{};
  mzc_options opt{};
  int num_sms = 0;
  int64_t f_pad = 0, qkv_dim = 0, max_rows = 0, nblk = 0, block_bytes = 0;
  cudaStream_t cs = nullptr, xs = nullptr;
  std::vector<LayerDev> layers;
  uint8_t* d_weights = nullptr;
  uint16_t *d_embed = nullptr, *d_lm = nullptr;
  float* d_fnorm = nullptr;
  // folded RMSNorm of row sets of 5-256 rows: resident copies of the layers'
  // norm weights ([L][attn, ffn][d]; a producer GEMM reads the next layer's
  // before that layer's streamed weights are waited for) and the per-row,
  // per-128-column-tile sums of squares [256][d / 128]
  float* d_gnorm = nullptr;
  float* d_ss = nullptr;
  uint8_t* d_pool = nullptr;
  float *d_cos = nullptr, *d_sin = nullptr;
  float* d_x = nullptr;
  uint16_t *d_h = nullptr, *d_qkv = nullptr, *d_q = nullptr, *d_attn = nullptr, *d_act = nullptr;
  CUtensorMap tm_h, tm_attn, tm_act;
  uint8_t* d_meta = nullptr;  // tokens | pos | block tables
  uint8_t* h_meta = nullptr;
  uint8_t* h_meta_dev = nullptr;  // device view of the mapped h_meta
  size_t meta_bytes = 0;
  float* d_logits = nullptr;
  float* h_logits = nullptr;
  int32_t* h_status = nullptr;  // inside h_logits' allocation, after the vocab floats
  void* d_scratch = nullptr;
  int64_t scratch_bytes = 0;
  int32_t* d_status = nullptr;
  uint8_t* h_store = nullptr;
  uint16_t* h_store_dev = nullptr;  // device view of the mapped store (read_swapped)
  uint8_t* d_staging = nullptr;
  int32_t* d_list = nullptr;
  int32_t* h_list = nullptr;
  uint8_t* h_staging = nullptr;  // pinned, one layer of blocks (reads)
  std::vector<cudaEvent_t> ev_kv, ev_w;
  // swap codec: compressed slots; restores land in a staging buffer (two,
  // alternating by layer) and a decode stream writes the pool
  int32_t codec = MZC_CODEC_NONE;
  int64_t slot_bytes = 0;
  cudaStream_t ds = nullptr;
  std::vector<cudaEvent_t> ev_h2d, ev_dec;
  uint8_t* d_rstage[2] = {nullptr, nullptr};
  cudaEvent_t ev_t0 = nullptr, ev_t1 = nullptr, ev_c0 = nullptr, ev_c1 = nullptr,
              ev_l0 = nullptr, ev_l1 = nullptr;
  // streams passed in through mzc_options belong to the caller
  bool own_cs = true, own_xs = true;
  // MZC_WAIT_BLOCK_FLAG: a residency flag per physical block (non-zero = data
  // present), cleared for a restore's destination blocks on the compute
  // stream and set by the copy engine after each copied run (from h_ones)
  int32_t* d_flags = nullptr;
  int32_t* h_ones = nullptr;
  // order flags of the residual-add GEMMs whose last wave is split over k
  mzc::GemmSplit gsplit;
  cudaEvent_t ev_clear = nullptr;
  bool restore_issued = false, lm_timed = false, ttft_from_copy = false;
  // per-class launch counts and optional CUDA-event timing
  int32_t ktime_mask = 0;
  mzc_kernel_stat kstat[MZC_K_NCLASS] = {};
  struct KEv {
    int cls;
    cudaEvent_t a, b;
    double flops, bytes;
  };
  std::vector<cudaEvent_t> ev_pool;
  std::vector<KEv> kev;
  size_t ev_next = 0;
  std::vector<int32_t> tokens;
  int32_t policy = MZC_POLICY_COPY;
  mzc_profile prof = default_profile();
  mzc_stats_t last{};
  std::string err;

  mzc_status fail(mzc_status s, const std::string& m) {
    err = m;
    return s;
  }
  mzc_status from_state(mzc_status s) {
    if (s != MZC_OK) err = st.error();
    return s;
  }
};

#define CK(call)                                                                          \
  do {                                                                                    \
    cudaError_t e_ = (call);                                                              \
    if (e_ != cudaSuccess)                                                                \
      return ctx->fail(MZC_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_)); \
  } while (0)

namespace {

mzc_status destroy_impl(mzc_ctx* ctx) {
  if (!ctx) return MZC_ERR_INVALID;
  cudaSetDevice(ctx->opt.device);
  if (ctx->cs) cudaStreamSynchronize(ctx->cs);
  if (ctx->xs) cudaStreamSynchronize(ctx->xs);
  if (ctx->ds) cudaStreamSynchronize(ctx->ds);
  for (auto& L : ctx->layers)
    if (L.host_master) cudaFreeHost(L.host_master);
  void* dev[] = {ctx->d_weights, ctx->d_embed, ctx->d_lm,      ctx->d_fnorm,   ctx->d_pool,
                 ctx->d_cos,     ctx->d_sin,   ctx->d_x,       ctx->d_h,       ctx->d_qkv,
                 ctx->d_q,       ctx->d_attn,  ctx->d_act,     ctx->d_meta,    ctx->d_logits,
                 ctx->d_scratch, ctx->d_status, ctx->d_staging, ctx->d_list,
                 ctx->d_rstage[0], ctx->d_rstage[1], ctx->d_flags, ctx->gsplit.flags,
                 ctx->d_gnorm,   ctx->d_ss};
  for (void* p : dev)
    if (p) cudaFree(p);
  void* host[] = {ctx->h_meta, ctx->h_logits, ctx->h_store, ctx->h_list, ctx->h_staging, ctx->h_ones};
  for (void* p : host)
    if (p) cudaFreeHost(p);
  for (auto e : ctx->ev_pool) cudaEventDestroy(e);
  for (auto e : ctx->ev_kv) cudaEventDestroy(e);
  for (auto e : ctx->ev_w) cudaEventDestroy(e);
  for (auto e : ctx->ev_h2d) cudaEventDestroy(e);
  for (auto e : ctx->ev_dec) cudaEventDestroy(e);
  cudaEvent_t evs[] = {ctx->ev_t0, ctx->ev_t1, ctx->ev_c0, ctx->ev_c1, ctx->ev_l0, ctx->ev_l1,
                       ctx->ev_clear};
  for (auto e : evs)
    if (e) cudaEventDestroy(e);
  if (ctx->cs && ctx->own_cs) cudaStreamDestroy(ctx->cs);
  if (ctx->xs && ctx->own_xs) cudaStreamDestroy(ctx->xs);
  if (ctx->ds) cudaStreamDestroy(ctx->ds);
  delete ctx;
  return MZC_OK;
}

// bf16 weights -> fp16 GEMM operands (round to nearest even).  Exact for
// every bf16 value in [2^-14, 65504]; smaller magnitudes round to fp16
// subnormals (absolute error <= 2^-25).  Returns false if a value would
// overflow fp16.
bool bf16_to_f16(const uint16_t* src, uint16_t* dst, int64_t n) {
  bool ok = true;
  for (int64_t i = 0; i < n; ++i) {
    uint32_t u = static_cast<uint32_t>(src[i]) << 16;
    float f;
    std::memcpy(&f, &u, 4);
    if (!(std::fabs(f) <= 65504.0f)) ok = false;
    __half h = __float2half_rn(f);
    dst[i] = __half_as_ushort(h);
  }
  return ok;
}

// Converts one layer's canonical bf16 weights into its packed fp16 host image.
bool pack_layer(const mzc_model_shape& s, int64_t f_pad, const mzc_layer_weights& w,
                std::vector<uint8_t>& img, const LayerDev& L) {
  const int64_t d = s.d_model, hq = s.n_q_heads, hkv = s.n_kv_heads, hd = s.head_dim, f = s.ffn_dim;
  std::fill(img.begin(), img.end(), 0);
  auto off = [&](const void* dev) { return static_cast<size_t>(static_cast<const uint8_t*>(dev) - L.base); };
  bool ok = true;
  uint16_t* qkv = reinterpret_cast<uint16_t*>(img.data() + off(L.wqkv));
  ok &= bf16_to_f16(w.wq, qkv, hq * hd * d);
  ok &= bf16_to_f16(w.wk, qkv + hq * hd * d, hkv * hd * d);
  ok &= bf16_to_f16(w.wv, qkv + (hq + hkv) * hd * d, hkv * hd * d);
  ok &= bf16_to_f16(w.wo, reinterpret_cast<uint16_t*>(img.data() + off(L.wo)), d * hq * hd);
  uint16_t* w13 = reinterpret_cast<uint16_t*>(img.data() + off(L.w13));
  const int64_t G = mzc::kSwigluGroup;
  for (int64_t j = 0; j < f; ++j) {
    const int64_t grp = j / G, r = j % G;
    ok &= bf16_to_f16(w.w_gate + j * d, w13 + (grp * 2 * G + r) * d, d);
    ok &= bf16_to_f16(w.w_up + j * d, w13 + (grp * 2 * G + G + r) * d, d);
  }
  uint16_t* w2 = reinterpret_cast<uint16_t*>(img.data() + off(L.w2));
  for (int64_t r = 0; r < d; ++r) ok &= bf16_to_f16(w.w_down + r * f, w2 + r * f_pad, f);
  std::memcpy(img.data() + off(L.attn_norm), w.attn_norm, sizeof(float) * d);
  std::memcpy(img.data() + off(L.ffn_norm), w.ffn_norm, sizeof(float) * d);
  return ok;
}

mzc_status create_impl(const mzc_model_shape* shape, const mzc_options* options,
                       const mzc_weights* weights, mzc_ctx* ctx) {
  const mzc_model_shape& s = *shape;
  ctx->shape = s;
  ctx->opt = options ? *options : mzc_options{};
  if (!options) ctx->opt.overlap = 1;
  if (s.head_dim != 64 && s.head_dim != 128)
    return ctx->fail(MZC_ERR_INVALID, "head_dim must be 64 or 128");
  if (s.d_model % 64 != 0) return ctx->fail(MZC_ERR_INVALID, "d_model must be a multiple of 64");
  if ((static_cast<int64_t>(s.n_q_heads) * s.head_dim) % 64 != 0)
    return ctx->fail(MZC_ERR_INVALID, "n_q_heads*head_dim must be a multiple of 64");
  if (ctx->opt.swap_codec != MZC_CODEC_NONE && ctx->opt.swap_codec != MZC_CODEC_Q8)
    return ctx->fail(MZC_ERR_INVALID, "unknown swap_codec");
  if (ctx->opt.wait_mode != MZC_WAIT_LAYER_EVENT && ctx->opt.wait_mode != MZC_WAIT_BLOCK_FLAG)
    return ctx->fail(MZC_ERR_INVALID, "unknown wait_mode");
  // with the 8-bit store, kernels (not the copy engine) write the restored
  // blocks; a flag they set could wait behind attention CTAs that spin on it
  if (ctx->opt.wait_mode == MZC_WAIT_BLOCK_FLAG && ctx->opt.swap_codec != MZC_CODEC_NONE)
    return ctx->fail(MZC_ERR_INVALID, "MZC_WAIT_BLOCK_FLAG needs swap_codec MZC_CODEC_NONE");
  if (ctx->opt.debug_checks != 0 && ctx->opt.debug_checks != 1)
    return ctx->fail(MZC_ERR_INVALID, "debug_checks must be 0 or 1");
  if (ctx->opt.read_swapped != 0 && ctx->opt.read_swapped != 1)
    return ctx->fail(MZC_ERR_INVALID, "read_swapped must be 0 or 1");
  // in-place reads need the blocks as stored (not 8-bit codes)
  if (ctx->opt.read_swapped && ctx->opt.swap_codec != MZC_CODEC_NONE)
    return ctx->fail(MZC_ERR_INVALID, "read_swapped needs swap_codec MZC_CODEC_NONE");
  ctx->codec = ctx->opt.swap_codec;
  {
    const int64_t block_elems = 2LL * s.n_kv_heads * 16 * s.head_dim;
    ctx->slot_bytes = ctx->codec == MZC_CODEC_Q8 ? mzc::q8_block_bytes(block_elems) : 2 * block_elems;
  }
  mzc_status ss = ctx->st.init(s, ctx->opt.pool_blocks, ctx->opt.host_store_bytes, ctx->slot_bytes);
  if (ss != MZC_OK) return ctx->fail(ss, ctx->st.error());
  ctx->st.set_read_swapped(ctx->opt.read_swapped != 0);
  if (!weights || !weights->embed || !weights->lm_head || !weights->final_norm || !weights->layers)
    return ctx->fail(MZC_ERR_INVALID, "weights are incomplete");
  CK(cudaSetDevice(ctx->opt.device));
  CK(cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->opt.device));
  const int64_t d = s.d_model, hq = s.n_q_heads, hkv = s.n_kv_heads, hd = s.head_dim;
  const int64_t L = s.n_layers, V = s.vocab;
  ctx->f_pad = align_up(s.ffn_dim, mzc::kSwigluGroup);
  ctx->qkv_dim = (hq + 2 * hkv) * hd;
  ctx->max_rows = ctx->opt.max_rows > 0 ? ctx->opt.max_rows : s.max_ctx;
  ctx->nblk = ctx->st.nblk_max();
  ctx->block_bytes = ctx->st.block_bytes();
  const int64_t R = ctx->max_rows, F2 = 2 * ctx->f_pad;

  if (ctx->opt.compute_stream) {
    ctx->cs = static_cast<cudaStream_t>(ctx->opt.compute_stream);
    ctx->own_cs = false;
  } else {
    CK(cudaStreamCreateWithFlags(&ctx->cs, cudaStreamNonBlocking));
  }
  if (ctx->opt.copy_stream) {
    ctx->xs = static_cast<cudaStream_t>(ctx->opt.copy_stream);
    ctx->own_xs = false;
  } else {
    CK(cudaStreamCreateWithFlags(&ctx->xs, cudaStreamNonBlocking));
  }
  if (ctx->codec != MZC_CODEC_NONE) {
    CK(cudaStreamCreateWithFlags(&ctx->ds, cudaStreamNonBlocking));
    ctx->ev_h2d.assign(L, nullptr);
    ctx->ev_dec.assign(L, nullptr);
    for (int64_t l = 0; l < L; ++l) {
      CK(cudaEventCreateWithFlags(&ctx->ev_h2d[l], cudaEventDisableTiming));
      CK(cudaEventCreateWithFlags(&ctx->ev_dec[l], cudaEventDisableTiming));
    }
  }
  ctx->ev_kv.assign(L, nullptr);
  ctx->ev_w.assign(L, nullptr);
  for (int64_t l = 0; l < L; ++l) {
    CK(cudaEventCreateWithFlags(&ctx->ev_kv[l], cudaEventDisableTiming));
    CK(cudaEventCreateWithFlags(&ctx->ev_w[l], cudaEventDisableTiming));
  }
  cudaEvent_t* timed[] = {&ctx->ev_t0, &ctx->ev_t1, &ctx->ev_c0, &ctx->ev_c1, &ctx->ev_l0, &ctx->ev_l1};
  for (auto e : timed) CK(cudaEventCreate(e));

  // ---- weights: one slot per layer ----
  size_t o = 0;
  const size_t sz_qkv = align_up(ctx->qkv_dim * d * 2, 1024), sz_o = align_up(d * hq * hd * 2, 1024);
  const size_t sz_13 = align_up(F2 * d * 2, 1024), sz_2 = align_up(d * ctx->f_pad * 2, 1024);
  const size_t sz_n = align_up(d * 4, 1024);
  const size_t slot = sz_qkv + sz_o + sz_13 + sz_2 + 2 * sz_n;
  CK(cudaMalloc(&ctx->d_weights, slot * L));
  ctx->layers.assign(L, LayerDev{});
  std::vector<uint8_t> img(slot);
  for (int64_t l = 0; l < L; ++l) {
    LayerDev& Ld = ctx->layers[l];
    Ld.base = ctx->d_weights + slot * l;
    Ld.bytes = slot;
    o = 0;
    Ld.wqkv = reinterpret_cast<uint16_t*>(Ld.base + o); o += sz_qkv;
    Ld.wo = reinterpret_cast<uint16_t*>(Ld.base + o); o += sz_o;
    Ld.w13 = reinterpret_cast<uint16_t*>(Ld.base + o); o += sz_13;
    Ld.w2 = reinterpret_cast<uint16_t*>(Ld.base + o); o += sz_2;
    Ld.attn_norm = reinterpret_cast<float*>(Ld.base + o); o += sz_n;
    Ld.ffn_norm = reinterpret_cast<float*>(Ld.base + o); o += sz_n;
    const mzc_layer_weights& w = weights->layers[l];
    if (!w.wq || !w.wk || !w.wv || !w.wo || !w.w_gate || !w.w_up || !w.w_down || !w.attn_norm || !w.ffn_norm)
      return ctx->fail(MZC_ERR_INVALID, "layer weights are incomplete");
    if (!pack_layer(s, ctx->f_pad, w, img, Ld))
      return ctx->fail(MZC_ERR_INVALID, "a projection weight is outside the fp16 range");
    CK(cudaMemcpy(Ld.base, img.data(), slot, cudaMemcpyHostToDevice));
  }
  CK(cudaMalloc(&ctx->d_embed, V * d * 2));
  CK(cudaMalloc(&ctx->d_lm, V * d * 2));
  CK(cudaMalloc(&ctx->d_fnorm, d * 4));
  CK(cudaMemcpy(ctx->d_embed, weights->embed, V * d * 2, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(ctx->d_lm, weights->lm_head, V * d * 2, cudaMemcpyHostToDevice));
  CK(cudaMemcpy(ctx->d_fnorm, weights->final_norm, d * 4, cudaMemcpyHostToDevice));
  if (d % 128 == 0) {
    CK(cudaMalloc(&ctx->d_gnorm, static_cast<size_t>(L) * 2 * d * 4));
    CK(cudaMalloc(&ctx->d_ss, static_cast<size_t>(256) * (d / 128) * 4));
    for (int64_t l = 0; l < L; ++l) {
      CK(cudaMemcpy(ctx->d_gnorm + (2 * l) * d, weights->layers[l].attn_norm, d * 4, cudaMemcpyHostToDevice));
      CK(cudaMemcpy(ctx->d_gnorm + (2 * l + 1) * d, weights->layers[l].ffn_norm, d * 4, cudaMemcpyHostToDevice));
    }
  }

  // ---- KV pool (zeroed: never-written slots hold finite values) ----
  const size_t pool_bytes = static_cast<size_t>(ctx->st.pool_blocks()) * ctx->block_bytes;
  CK(cudaMalloc(&ctx->d_pool, pool_bytes));
  CK(cudaMemset(ctx->d_pool, 0, pool_bytes));

  // ---- rotary tables: angle(pos, i) = pos * theta^(-2i/hd) in double ----
  {
    const int64_t P = s.max_ctx, half = hd / 2;
    std::vector<float> c(P * half), sn(P * half);
    for (int64_t i = 0; i < half; ++i) {
      const double inv = std::pow(static_cast<double>(s.rope_theta), -2.0 * static_cast<double>(i) / static_cast<double>(hd));
      for (int64_t p = 0; p < P; ++p) {
        const double a = static_cast<double>(p) * inv;
        c[p * half + i] = static_cast<float>(std::cos(a));
        sn[p * half + i] = static_cast<float>(std::sin(a));
      }
    }
    CK(cudaMalloc(&ctx->d_cos, P * half * 4));
    CK(cudaMalloc(&ctx->d_sin, P * half * 4));
    CK(cudaMemcpy(ctx->d_cos, c.data(), P * half * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(ctx->d_sin, sn.data(), P * half * 4, cudaMemcpyHostToDevice));
  }

  // ---- activations ----
  CK(cudaMalloc(&ctx->d_x, R * d * 4));
  CK(cudaMalloc(&ctx->d_h, R * d * 2));
  CK(cudaMalloc(&ctx->d_qkv, R * ctx->qkv_dim * 2));
  CK(cudaMalloc(&ctx->d_q, R * hq * hd * 2));
  CK(cudaMalloc(&ctx->d_attn, R * hq * hd * 2));
  CK(cudaMalloc(&ctx->d_act, R * ctx->f_pad * 2));
  CK(cudaMemset(ctx->d_h, 0, R * d * 2));
  CK(cudaMemset(ctx->d_attn, 0, R * hq * hd * 2));
  CK(cudaMemset(ctx->d_act, 0, R * ctx->f_pad * 2));
  // A operands: box 128 rows of 64 columns
  bool ok = mzc::make_tmap_f16(&ctx->tm_h, ctx->d_h, R, d, 128) &&
            mzc::make_tmap_f16(&ctx->tm_attn, ctx->d_attn, R, hq * hd, 128) &&
            mzc::make_tmap_f16(&ctx->tm_act, ctx->d_act, R, ctx->f_pad, 128);
  for (int64_t l = 0; l < L && ok; ++l) {
    LayerDev& Ld = ctx->layers[l];
    ok = mzc::make_gemm_weight(&Ld.tm_qkv, Ld.wqkv, ctx->qkv_dim, d) &&
         mzc::make_gemm_weight(&Ld.tm_o, Ld.wo, d, hq * hd) &&
         mzc::make_gemm_weight(&Ld.tm_13, Ld.w13, F2, d) &&
         mzc::make_gemm_weight(&Ld.tm_2, Ld.w2, d, ctx->f_pad);
  }
  if (!ok) return ctx->fail(MZC_ERR_CUDA, "cuTensorMapEncodeTiled failed");

  // ---- per-call metadata, logits, scratch, status ----
  ctx->meta_bytes = align_up(static_cast<size_t>(s.max_ctx) * 8 + static_cast<size_t>(L) * ctx->nblk * 4, 16);
  CK(cudaMalloc(&ctx->d_meta, ctx->meta_bytes));
  // mapped: the prefill pulls its metadata in with a kernel, so the upload never
  // queues behind restore copies on the host-to-device copy engine
  CK(cudaHostAlloc(&ctx->h_meta, ctx->meta_bytes, cudaHostAllocMapped));
  CK(cudaHostGetDevicePointer(reinterpret_cast<void**>(&ctx->h_meta_dev), ctx->h_meta, 0));
  CK(cudaMalloc(&ctx->d_logits, V * 4));
  // the logits, then one word for the status read back with each step
  CK(cudaHostAlloc(&ctx->h_logits, V * 4 + 16, cudaHostAllocDefault));
  ctx->h_status = reinterpret_cast<int32_t*>(ctx->h_logits + V);
  *ctx->h_status = 0;
  int64_t scratch = 0;
  for (int64_t n = 1; n <= std::min<int64_t>(R, 8192); ++n) {
    int sp = 1, per = 0;
    mzc::attention_split(n, s.n_q_heads, s.n_kv_heads, s.head_dim, s.max_ctx, ctx->num_sms, &sp, &per);
    scratch = std::max(scratch, mzc::attention_scratch_bytes(n, s.n_q_heads, s.head_dim, sp));
  }
  ctx->scratch_bytes = scratch;
  if (scratch > 0) CK(cudaMalloc(&ctx->d_scratch, scratch));
  CK(cudaMalloc(&ctx->d_status, 4));
  CK(cudaMemset(ctx->d_status, 0, 4));
  ctx->gsplit.n_flags = std::max(ctx->num_sms, 256);
  CK(cudaMalloc(&ctx->gsplit.flags, ctx->gsplit.n_flags * 8));
  CK(cudaMemset(ctx->gsplit.flags, 0, ctx->gsplit.n_flags * 8));
  CK(cudaMalloc(&ctx->d_staging, ctx->nblk * ctx->block_bytes));
  if (ctx->codec != MZC_CODEC_NONE)
    for (auto& b : ctx->d_rstage) CK(cudaMalloc(&b, ctx->nblk * ctx->slot_bytes));
  CK(cudaMalloc(&ctx->d_list, L * ctx->nblk * 4));
  CK(cudaHostAlloc(&ctx->h_list, L * ctx->nblk * 4, cudaHostAllocDefault));
  CK(cudaHostAlloc(&ctx->h_staging, ctx->nblk * ctx->block_bytes, cudaHostAllocDefault));
  if (ctx->opt.wait_mode == MZC_WAIT_BLOCK_FLAG) {
    CK(cudaMalloc(&ctx->d_flags, ctx->st.pool_blocks() * 4));
    CK(cudaMemset(ctx->d_flags, 1, ctx->st.pool_blocks() * 4));  // every block present
    CK(cudaHostAlloc(&ctx->h_ones, ctx->nblk * 4, cudaHostAllocDefault));
    for (int64_t i = 0; i < ctx->nblk; ++i) ctx->h_ones[i] = 1;
    CK(cudaEventCreateWithFlags(&ctx->ev_clear, cudaEventDisableTiming));
  }
  CK(cudaDeviceSynchronize());
  return MZC_OK;
}

// debug_checks: every resident or in-flight (layer, block) maps to a physical
// block inside the pool, and no two map to the same one.
mzc_status debug_check_tables(mzc_ctx* ctx) {
  std::vector<uint8_t> used(static_cast<size_t>(ctx->st.pool_blocks()), 0);
  for (int32_t l = 0; l < ctx->shape.n_layers; ++l)
    for (int64_t b = 0; b < ctx->nblk; ++b) {
      const mzc::BlockEntry& e = ctx->st.at(l, b);
      if (e.phys < 0) continue;
      if (e.phys >= ctx->st.pool_blocks())
        return ctx->fail(MZC_ERR_STATE, "debug check: layer " + std::to_string(l) + " block " +
                                            std::to_string(b) + " maps outside the pool");
      if (used[e.phys]++)
        return ctx->fail(MZC_ERR_STATE, "debug check: physical block " + std::to_string(e.phys) +
                                            " is mapped twice");
    }
  return MZC_OK;
}

// Moves `moves` (COPY eviction) out to the pinned store, then poisons the
// freed physical blocks (largest finite KV value) so that a read that does
// not wait for its restore shows up in the results.
mzc_status copy_out(mzc_ctx* ctx, const std::vector<mzc::EvictMove>& moves) {
  int64_t total = 0;
  for (auto& mv : moves) {
    std::memcpy(ctx->h_list + total, mv.phys.data(), mv.phys.size() * 4);
    total += static_cast<int64_t>(mv.phys.size());
  }
  if (total == 0) return MZC_OK;
  CK(cudaMemcpyAsync(ctx->d_list, ctx->h_list, total * 4, cudaMemcpyHostToDevice, ctx->cs));
  int64_t at = 0;
  for (auto& mv : moves) {
    const int64_t nb = static_cast<int64_t>(mv.phys.size());
    if (ctx->codec == MZC_CODEC_Q8)
      CK(mzc::launch_q8_encode(ctx->d_pool, ctx->d_list + at, nb, ctx->block_bytes / 2, ctx->d_staging, ctx->cs));
    else
      CK(mzc::launch_gather_blocks(ctx->d_pool, ctx->d_list + at, nb, ctx->block_bytes, ctx->d_staging, ctx->cs));
    CK(cudaMemcpyAsync(ctx->h_store + mv.host_off, ctx->d_staging, nb * ctx->slot_bytes,
                       cudaMemcpyDeviceToHost, ctx->cs));
    at += nb;
  }
  CK(mzc::launch_poison_blocks(ctx->d_pool, ctx->d_list, total, ctx->block_bytes, ctx->shape.kv_dtype, ctx->cs));
  CK(cudaStreamSynchronize(ctx->cs));
  return MZC_OK;
}

mzc_status poison(mzc_ctx* ctx, const std::vector<int32_t>& phys) {
  if (phys.empty()) return MZC_OK;
  std::memcpy(ctx->h_list, phys.data(), phys.size() * 4);
  CK(cudaMemcpyAsync(ctx->d_list, ctx->h_list, phys.size() * 4, cudaMemcpyHostToDevice, ctx->cs));
  CK(mzc::launch_poison_blocks(ctx->d_pool, ctx->d_list, static_cast<int64_t>(phys.size()), ctx->block_bytes, ctx->shape.kv_dtype, ctx->cs));
  CK(cudaStreamSynchronize(ctx->cs));
  return MZC_OK;
}

mzc_status ensure_store(mzc_ctx* ctx) {
  if (ctx->h_store) return MZC_OK;
  if (ctx->opt.read_swapped) {
    // mapped, so the attention kernels can read swapped blocks in place
    CK(cudaHostAlloc(&ctx->h_store, ctx->st.host_store_bytes(), cudaHostAllocMapped));
    CK(cudaHostGetDevicePointer(reinterpret_cast<void**>(&ctx->h_store_dev), ctx->h_store, 0));
  } else {
    CK(cudaHostAlloc(&ctx->h_store, ctx->st.host_store_bytes(), cudaHostAllocDefault));
  }
  return MZC_OK;
}

mzc_status check_status(mzc_ctx* ctx, const std::string& where = std::string()) {
  int32_t s = 0;
  CK(cudaMemcpy(&s, ctx->d_status, 4, cudaMemcpyDeviceToHost));
  if (s != 0) {
    CK(cudaMemset(ctx->d_status, 0, 4));
    const char* what = s == MZC_ERR_TIMEOUT    ? "a device wait timed out"
                       : s == MZC_ERR_OVERFLOW ? "an fp16 activation or K/V value overflowed (|x| >= 65520)"
                                               : "a device bounds check failed";
    return ctx->fail(static_cast<mzc_status>(s), where + what);
  }
  return MZC_OK;
}

cudaEvent_t next_event(mzc_ctx* ctx) {
  if (ctx->ev_next == ctx->ev_pool.size()) {
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    ctx->ev_pool.push_back(e);
  }
  return ctx->ev_pool[ctx->ev_next++];
}

// Launches one kernel of class `cls` (n_kernels launches, algorithmic work
// flops / bytes), bracketed by CUDA events on the compute stream when kernel
// timing is on.
template <class F>
cudaError_t klaunch(mzc_ctx* ctx, int cls, double flops, double bytes, int n_kernels, F&& fn) {
  mzc_kernel_stat& k = ctx->kstat[cls];
  k.launches += n_kernels;
  k.flops += flops;
  k.bytes += bytes;
  if (!((ctx->ktime_mask >> cls) & 1)) return fn();
  cudaEvent_t a = next_event(ctx), b = next_event(ctx);
  if (!a || !b) return cudaErrorMemoryAllocation;
  cudaError_t e = cudaEventRecord(a, ctx->cs);
  if (e != cudaSuccess) return e;
  e = fn();
  if (e != cudaSuccess) return e;
  e = cudaEventRecord(b, ctx->cs);
  ctx->kev.push_back(mzc_ctx::KEv{cls, a, b, flops, bytes});
  return e;
}

mzc_status run_prefill(mzc_ctx* ctx, const int32_t* tokens, int64_t n, float* logits_out) {
  const mzc_model_shape& s = ctx->shape;
  const int64_t d = s.d_model, hq = s.n_q_heads, hkv = s.n_kv_heads, hd = s.head_dim, L = s.n_layers;
  for (int64_t i = 0; i < n; ++i)
    if (tokens[i] < 0 || tokens[i] >= s.vocab) return ctx->fail(MZC_ERR_INVALID, "token id outside the vocabulary");
  mzc::PrefillPlan P;
  mzc_status ss = ctx->st.prepare_prefill(n, ctx->max_rows, &P);
  if (ss != MZC_OK) return ctx->from_state(ss);
  if (ctx->opt.debug_checks) {
    mzc_status e = debug_check_tables(ctx);
    if (e != MZC_OK) {
      ctx->st.abort_prefill(P);
      return e;
    }
  }
  // per-block waits: the attention reads a block once its flag is set, so no
  // layer event is waited on for the keys a restore copies in
  const int32_t* flags = (ctx->d_flags && ctx->opt.overlap && ctx->restore_issued) ? ctx->d_flags : nullptr;
  const int64_t nrec = P.rec_end - P.rec_begin, rows = nrec + n;
  if (rows == 0) {
    ctx->st.complete(0);
    return MZC_OK;
  }
  // metadata: tokens | positions | block tables
  int32_t* htok = reinterpret_cast<int32_t*>(ctx->h_meta);
  int32_t* hpos = htok + rows;
  int32_t* htab = hpos + rows;
  for (int64_t i = 0; i < nrec; ++i) {
    htok[i] = ctx->tokens[P.rec_begin + i];
    hpos[i] = static_cast<int32_t>(P.rec_begin + i);
  }
  for (int64_t i = 0; i < n; ++i) {
    htok[nrec + i] = tokens[i];
    hpos[nrec + i] = static_cast<int32_t>(P.prompt_begin + i);
  }
  ctx->st.block_table_into(htab, ctx->opt.read_swapped != 0);
  const size_t tab_entries = static_cast<size_t>(ctx->st.table_entries());
  // swapped blocks this prefill reads in place from the mapped store
  const void* host_pool = ctx->opt.read_swapped ? ctx->h_store_dev : nullptr;
  const int64_t host_blocks = host_pool ? ctx->st.host_slots() : 0;
  const size_t mbytes = static_cast<size_t>(rows) * 8 + tab_entries * 4;
  int32_t* dtok = reinterpret_cast<int32_t*>(ctx->d_meta);
  int32_t* dpos = dtok + rows;
  int32_t* dtab = dpos + rows;
  cudaStream_t cs = ctx->cs;
  auto bail = [&](mzc_status e) {
    cudaStreamSynchronize(cs);
    ctx->st.abort_prefill(P);
    return e;
  };
#define CKP(call)                                                                             \
  do {                                                                                        \
    cudaError_t e_ = (call);                                                                  \
    if (e_ != cudaSuccess)                                                                    \
      return bail(ctx->fail(MZC_ERR_CUDA, std::string(#call) + ": " + cudaGetErrorString(e_))); \
  } while (0)
  CKP(cudaEventRecord(ctx->ev_t0, cs));
  ctx->ttft_from_copy = ctx->restore_issued;
  CKP(mzc::launch_copy16(ctx->h_meta_dev, ctx->d_meta, static_cast<int64_t>(mbytes), cs));
  if (!ctx->opt.overlap && ctx->restore_issued) CKP(cudaStreamWaitEvent(cs, ctx->ev_c1, 0));
  ctx->ev_next = 0;
  ctx->kev.clear();
  const double kvb = s.kv_dtype == MZC_KV_FP16 ? 2.0 : 2.0;  // bytes per stored K/V element
  // algorithmic attention work of rows [r0, r0 + nr)
  auto attn_work = [&](int64_t r0, int64_t nr, double* fl, double* by) {
    double pairs = 0.0;
    int64_t mx = 0;
    for (int64_t i = r0; i < r0 + nr; ++i) {
      pairs += static_cast<double>(hpos[i]) + 1.0;
      mx = std::max<int64_t>(mx, hpos[i] + 1);
    }
    *fl = 4.0 * hd * hq * pairs;
    *by = 2.0 * hkv * hd * kvb * mx + 2.0 * nr * hq * hd * 2.0;
  };
  const double dd = static_cast<double>(d);
  // Rows run in causal chunks of at most max_rows: every row of a chunk
  // attends only to positions written by this chunk or an earlier one, and a
  // chunk goes through all layers before the next starts.  The prompt rows
  // come last, so the last chunk holds the row whose logits are returned.
  const int64_t chunk = ctx->max_rows;
  int64_t last_rows = 0;
  const bool want_logits = n > 0 && logits_out != nullptr;
  for (int64_t c0 = 0; c0 < rows; c0 += chunk) {
    const int64_t c1 = std::min(rows, c0 + chunk), cr = c1 - c0;
    const int64_t rec_hi = std::min(c1, nrec);          // recompute rows [c0, rec_hi)
    const int64_t n_rec_c = std::max<int64_t>(0, rec_hi - c0);
    const int64_t n_prm_c = cr - n_rec_c;                // prompt rows of this chunk
    const int64_t max_keys = static_cast<int64_t>(hpos[c1 - 1]) + 1;
    const double R = static_cast<double>(cr);
    int32_t* ctok = dtok + c0;
    int32_t* cpos = dpos + c0;
    CKP(klaunch(ctx, MZC_K_EMBED, 0.0, R * dd * 6.0, 1, [&] {
      return mzc::launch_embed(ctok, cr, ctx->d_embed, static_cast<int32_t>(d), s.vocab, ctx->d_x, ctx->d_status, cs);
    }));
    // RMSNorm folded into the projections: each residual-add projection also
    // writes x * g of the next norm and partial sums of squares of x, and the
    // next QKV or gate/up projection scales its rows by rstd, so no norm runs
    // as its own launch but the first layer's attention norm (after the
    // embedding).  Row sets of 5-256 rows: the split-K kernels, one partial
    // per row and 128-column tile.  One row (decode steps, and the last
    // layer's logits row of every prefill): the GEMV kernels, one partial per
    // producer CTA.
    const bool fold_rows = !ctx->opt.separate_norm && ctx->d_ss != nullptr && cr > mzc::kGemvMaxRows &&
                           cr <= 256 && mzc::gemm_splitk_launches(cr, d, hq * hd, mzc::EPI_ADD_F32, ctx->num_sms) &&
                           mzc::gemm_splitk_launches(cr, d, ctx->f_pad, mzc::EPI_ADD_F32, ctx->num_sms);
    const int64_t np_o = mzc::gemv_norm_tiles(d, hq * hd), np_d = mzc::gemv_norm_tiles(d, ctx->f_pad);
    const bool fold_one = !ctx->opt.separate_norm && ctx->d_ss != nullptr && np_o <= mzc::kGemvNormMax &&
                          np_d <= mzc::kGemvNormMax;
    const bool fold = fold_rows || (cr == 1 && fold_one);
    mzc::RowNorm rn_qkv;  // consumer of the previous layer's down projection
    rn_qkv.ss = ctx->d_ss;
    rn_qkv.nt = static_cast<int>(fold_rows ? d / 128 : np_d);
    rn_qkv.d = static_cast<float>(d);
    rn_qkv.eps = s.rms_eps;
    mzc::RowNorm rn_mlp = rn_qkv;  // consumer of the O projection
    rn_mlp.nt = static_cast<int>(fold_rows ? d / 128 : np_o);
    mzc::RowNorm rn_o = rn_mlp, rn_down = rn_qkv;  // producers: write h and the sums
    rn_o.h = rn_down.h = ctx->d_h;
    // Option fused_rope: the rotary embedding and KV-block write inside the
    // QKV projection's split-K reduction for row sets of 5-256 rows (no rotary
    // launch, no fp16 QKV round trip), unless the layer's writes must wait for
    // a copy.
    const bool rope_rows = ctx->opt.fused_rope && cr > mzc::kGemvMaxRows && cr <= 256 &&
                           (hd == 64 || hd == 128) &&
                           mzc::gemm_splitk_launches(cr, ctx->qkv_dim, d, mzc::EPI_QKV_ROPE, ctx->num_sms);
    mzc::RopeKV rk;
    rk.pos = cpos;
    rk.cos_t = ctx->d_cos;
    rk.sin_t = ctx->d_sin;
    rk.n_logical = ctx->nblk;
    rk.pool = reinterpret_cast<uint16_t*>(ctx->d_pool);
    rk.pool_blocks = ctx->st.pool_blocks();
    rk.q_out = ctx->d_q;
    rk.hq = static_cast<int>(hq);
    rk.hkv = static_cast<int>(hkv);
    rk.hd = static_cast<int>(hd);
    rk.f16kv = s.kv_dtype == MZC_KV_FP16 ? 1 : 0;
    auto gemm = [&](const CUtensorMap& ta, const void* a_ptr, const mzc::GemmWeight& w, void* out,
                    int64_t N, int64_t K, int epi, const mzc::RowNorm* rn = nullptr) {
      double out_b = epi == mzc::EPI_ADD_F32 ? R * N * 8.0 : (epi == mzc::EPI_SWIGLU_BF16 ? R * N : R * N * 2.0);
      if (rn != nullptr) out_b += epi == mzc::EPI_ADD_F32 ? R * N * 2.0 : R * (N / 128) * 4.0;
      return klaunch(ctx, MZC_K_GEMM, 2.0 * R * N * K, 2.0 * (R * K + static_cast<double>(N) * K) + out_b, 1,
                     [&] {
                       return mzc::launch_gemm(ta, w, out, cr, N, K, epi, ctx->d_status, cs,
                                               static_cast<const uint16_t*>(a_ptr), &ctx->gsplit, rn);
                     });
    };
    // attention of chunk rows [r0, r0 + nr) (r0 relative to the chunk)
    auto attention = [&](int64_t r0, int64_t nr, int64_t mk, const int32_t* ltab,
                         const int32_t* wait_flags = nullptr) {
      double fl, by;
      attn_work(c0 + r0, nr, &fl, &by);
      int sp = 1, per = 0;
      mzc::attention_split(nr, s.n_q_heads, s.n_kv_heads, s.head_dim, mk, ctx->num_sms, &sp, &per);
      const bool fits = sp == 1 || ctx->scratch_bytes >= mzc::attention_scratch_bytes(nr, s.n_q_heads, s.head_dim, sp);
      return klaunch(ctx, MZC_K_ATTENTION, fl, by, (sp > 1 && fits) ? 2 : 1, [&] {
        return mzc::launch_attention(ctx->d_q + r0 * hq * hd, cpos + r0, nr, s.n_q_heads, s.n_kv_heads,
                                     s.head_dim, ltab, ctx->nblk, ctx->d_pool, ctx->st.pool_blocks(),
                                     s.kv_dtype, ctx->d_attn + r0 * hq * hd, ctx->d_scratch,
                                     ctx->scratch_bytes, mk, ctx->num_sms, ctx->d_status, cs, wait_flags, 0,
                                     host_pool, host_blocks);
      });
    };
    const double norm_bytes = R * dd * 6.0 + dd * 4.0;
    const double rope_bytes = R * (hq + 2.0 * hkv) * hd * 4.0 + R * hd * 4.0;
    for (int64_t l = 0; l < L; ++l) {
      const LayerDev& W = ctx->layers[l];
      const int32_t* ltab = dtab + l * ctx->nblk;
      if (P.w_wait[l]) CKP(cudaStreamWaitEvent(cs, ctx->ev_w[l], 0));
      const bool fold_in = fold && l > 0;  // h and the sums come from layer l-1's down projection
      if (!fold_in)
        CKP(klaunch(ctx, MZC_K_RMSNORM, 0.0, norm_bytes, 1, [&] {
          return mzc::launch_rmsnorm(ctx->d_x, W.attn_norm, cr, static_cast<int32_t>(d), s.rms_eps, ctx->d_h, cs,
                                     ctx->d_status);
        }));
      const bool kv_wait = P.kv_wait_write[l] && n_prm_c > 0;
      if (rope_rows && !kv_wait) {
        rk.table = ltab;
        bool launched = false;
        const double qn = static_cast<double>(ctx->qkv_dim);
        CKP(klaunch(ctx, MZC_K_GEMM, 2.0 * R * qn * dd, 2.0 * (R * dd + qn * dd) + rope_bytes / 2.0, 1, [&] {
          return mzc::launch_gemm_splitk(ctx->tm_h, W.tm_qkv, ctx->d_qkv, cr, ctx->qkv_dim, d, mzc::EPI_QKV_ROPE,
                                         ctx->num_sms, ctx->d_status, cs, &launched, fold_in ? &rn_qkv : nullptr,
                                         &rk);
        }));
        if (!launched)
          return bail(ctx->fail(MZC_ERR_CUDA, "the QKV projection with the rotary write did not launch"));
      } else {
        CKP(gemm(ctx->tm_h, ctx->d_h, W.tm_qkv, ctx->d_qkv, ctx->qkv_dim, d, mzc::EPI_STORE_BF16,
                 fold_in ? &rn_qkv : nullptr));
        if (kv_wait) CKP(cudaStreamWaitEvent(cs, ctx->ev_kv[l], 0));
        CKP(klaunch(ctx, MZC_K_ROPE_KV, 0.0, rope_bytes, 1, [&] {
          return mzc::launch_rope_kv_write(ctx->d_qkv, cpos, cr, s.n_q_heads, s.n_kv_heads, s.head_dim,
                                           ctx->d_cos, ctx->d_sin, ltab, ctx->nblk, ctx->d_pool,
                                           ctx->st.pool_blocks(), s.kv_dtype, ctx->d_q, ctx->d_status, cs);
        }));
      }
      const bool wait_rec = n_rec_c > 0 && P.kv_wait_rec[l];
      const bool wait_prm = n_prm_c > 0 && P.kv_wait_prompt[l];
      if (l == L - 1) {
        // Every row's K/V of the last layer are written above.  The layer's
        // output (attention, O, MLP) feeds only the logits, i.e. the call's
        // last row: the other rows stop here, and without logits all do.
        if (want_logits && c1 == rows) {
          const int64_t r = cr - 1;
          const double f = static_cast<double>(hq) * hd;
          if (flags && wait_prm) {
            CKP(attention(r, 1, max_keys, ltab, flags));
          } else {
            if (wait_prm) CKP(cudaStreamWaitEvent(cs, ctx->ev_kv[l], 0));
            CKP(attention(r, 1, max_keys, ltab));
          }
          auto row_gemm = [&](const void* a_row, const mzc::GemmWeight& w, void* out_row, int64_t N, int64_t K,
                              int epi, const mzc::RowNorm* rn = nullptr) {
            const double out_b = epi == mzc::EPI_ADD_F32 ? N * 8.0 : (epi == mzc::EPI_SWIGLU_BF16 ? N * 1.0 : N * 2.0);
            return klaunch(ctx, MZC_K_GEMM, 2.0 * N * K, 2.0 * (K + static_cast<double>(N) * K) + out_b, 1, [&] {
              return mzc::launch_gemm(ctx->tm_h, w, out_row, 1, N, K, epi, ctx->d_status, cs,
                                      static_cast<const uint16_t*>(a_row), nullptr, rn);
            });
          };
          // the row's MLP norm folded into its O and gate/up GEMVs
          mzc::RowNorm rn_o1 = rn_o, rn_m1 = rn_mlp;
          rn_o1.nt = rn_m1.nt = static_cast<int>(np_o);
          rn_o1.h = ctx->d_h + r * d;
          rn_o1.g = ctx->d_gnorm != nullptr ? ctx->d_gnorm + (2 * l + 1) * d : nullptr;
          CKP(row_gemm(ctx->d_attn + r * hq * hd, W.tm_o, ctx->d_x + r * d, d, static_cast<int64_t>(f),
                       mzc::EPI_ADD_F32, fold_one ? &rn_o1 : nullptr));
          if (!fold_one)
            CKP(klaunch(ctx, MZC_K_RMSNORM, 0.0, dd * 10.0, 1, [&] {
              return mzc::launch_rmsnorm(ctx->d_x + r * d, W.ffn_norm, 1, static_cast<int32_t>(d), s.rms_eps,
                                         ctx->d_h + r * d, cs, ctx->d_status);
            }));
          CKP(row_gemm(ctx->d_h + r * d, W.tm_13, ctx->d_act + r * ctx->f_pad, 2 * ctx->f_pad, d,
                       mzc::EPI_SWIGLU_BF16, fold_one ? &rn_m1 : nullptr));
          CKP(row_gemm(ctx->d_act + r * ctx->f_pad, W.tm_2, ctx->d_x + r * d, d, ctx->f_pad, mzc::EPI_ADD_F32));
        }
        if (ctx->opt.debug_checks) {
          CKP(cudaStreamSynchronize(cs));
          mzc_status e = check_status(ctx, "layer " + std::to_string(l) + " (rows " + std::to_string(c0) +
                                               ".." + std::to_string(c1) + "): ");
          if (e != MZC_OK) return bail(e);
        }
        continue;
      }
      if (flags && n_rec_c > 0 && n_prm_c > 0 && wait_prm && !wait_rec) {
        // recomputed rows read only resident keys: their own launch, with no
        // flags, ahead of the prompt rows (in one launch the prompt rows' CTAs,
        // dispatched first, would hold the SMs while they wait on the copies)
        CKP(attention(0, n_rec_c, static_cast<int64_t>(hpos[c0 + n_rec_c - 1]) + 1, ltab));
        CKP(attention(n_rec_c, n_prm_c, max_keys, ltab, flags));
      } else if (flags && (wait_rec || wait_prm)) {
        CKP(attention(0, cr, max_keys, ltab, flags));
      } else if (n_rec_c > 0 && n_prm_c > 0 && wait_prm && !wait_rec) {
        // recompute rows read only resident keys: they run before the copy lands
        CKP(attention(0, n_rec_c, static_cast<int64_t>(hpos[c0 + n_rec_c - 1]) + 1, ltab));
        CKP(cudaStreamWaitEvent(cs, ctx->ev_kv[l], 0));
        CKP(attention(n_rec_c, n_prm_c, max_keys, ltab));
      } else {
        if (wait_rec || wait_prm) CKP(cudaStreamWaitEvent(cs, ctx->ev_kv[l], 0));
        CKP(attention(0, cr, max_keys, ltab));
      }
      if (fold) {
        rn_o.g = ctx->d_gnorm + (2 * l + 1) * d;  // this layer's MLP norm
        CKP(gemm(ctx->tm_attn, ctx->d_attn, W.tm_o, ctx->d_x, d, hq * hd, mzc::EPI_ADD_F32, &rn_o));
      } else {
        CKP(gemm(ctx->tm_attn, ctx->d_attn, W.tm_o, ctx->d_x, d, hq * hd, mzc::EPI_ADD_F32));
        CKP(klaunch(ctx, MZC_K_RMSNORM, 0.0, norm_bytes, 1, [&] {
          return mzc::launch_rmsnorm(ctx->d_x, W.ffn_norm, cr, static_cast<int32_t>(d), s.rms_eps, ctx->d_h, cs,
                                     ctx->d_status);
        }));
      }
      CKP(gemm(ctx->tm_h, ctx->d_h, W.tm_13, ctx->d_act, 2 * ctx->f_pad, d, mzc::EPI_SWIGLU_BF16,
               fold ? &rn_mlp : nullptr));
      if (fold) rn_down.g = ctx->d_gnorm + (2 * (l + 1)) * d;  // the next layer's attention norm
      CKP(gemm(ctx->tm_act, ctx->d_act, W.tm_2, ctx->d_x, d, ctx->f_pad, mzc::EPI_ADD_F32,
               fold ? &rn_down : nullptr));
      if (ctx->opt.debug_checks) {
        // name the first layer whose kernels recorded a device error
        CKP(cudaStreamSynchronize(cs));
        mzc_status e = check_status(ctx, "layer " + std::to_string(l) + " (rows " + std::to_string(c0) +
                                             ".." + std::to_string(c1) + "): ");
        if (e != MZC_OK) return bail(e);
      }
    }
    last_rows = cr;
  }
  ctx->lm_timed = false;
  if (n > 0 && logits_out) {
    CKP(cudaEventRecord(ctx->ev_l0, cs));
    CKP(klaunch(ctx, MZC_K_LM_HEAD, 2.0 * s.vocab * dd, s.vocab * dd * 2.0 + s.vocab * 4.0 + dd * 8.0, 1, [&] {
      return mzc::launch_lm_head(ctx->d_x + (last_rows - 1) * d, ctx->d_fnorm, static_cast<int32_t>(d), s.rms_eps,
                                 ctx->d_lm, s.vocab, ctx->d_logits, ctx->num_sms, cs);
    }));
    CKP(cudaEventRecord(ctx->ev_l1, cs));
    CKP(cudaMemcpyAsync(ctx->h_logits, ctx->d_logits, static_cast<size_t>(s.vocab) * 4, cudaMemcpyDeviceToHost, cs));
    ctx->lm_timed = true;
  }
  CKP(cudaEventRecord(ctx->ev_t1, cs));
  // the status word comes back with the step (after the copy stream's work
  // too), so a clean step costs no extra round trip to read it
  if (ctx->restore_issued) CKP(cudaStreamWaitEvent(cs, ctx->ev_c1, 0));
  CKP(cudaMemcpyAsync(ctx->h_status, ctx->d_status, 4, cudaMemcpyDeviceToHost, cs));
  // the host side of the restore's completion runs while the device works:
  // nothing reads the table before this call returns, and both streams are
  // synchronised below (a failed step still leaves the copied blocks valid)
  ctx->st.complete_restore();
  CKP(cudaStreamSynchronize(cs));
  if (ctx->restore_issued) CKP(cudaStreamSynchronize(ctx->xs));
#undef CKP
  for (const auto& ke : ctx->kev) {
    float ms = 0.0f;
    if (cudaEventElapsedTime(&ms, ke.a, ke.b) == cudaSuccess) ctx->kstat[ke.cls].ms += ms;
  }
  ctx->kev.clear();
  mzc_status st = *ctx->h_status == 0 ? MZC_OK : check_status(ctx);
  if (st != MZC_OK) {
    ctx->st.abort_prefill(P);
    return st;
  }
  if (n > 0 && logits_out) std::memcpy(logits_out, ctx->h_logits, static_cast<size_t>(s.vocab) * 4);
  ctx->st.complete(n);
  ctx->tokens.insert(ctx->tokens.end(), tokens, tokens + n);
  ctx->last.rows_last = rows;
  ctx->last.recompute_rows_last = nrec;
  ctx->restore_issued = false;
  return MZC_OK;
}

// Per-layer algorithmic sizes of a shape.
struct CostModelShape {
  double layer_weight_bytes, linear_flops_row, attn_flops_pair, qkv_frac;
  explicit CostModelShape(const mzc_model_shape& s) {
    const double d = s.d_model, hq = s.n_q_heads, hkv = s.n_kv_heads, hd = s.head_dim, f = s.ffn_dim;
    const double params = d * (hq + 2 * hkv) * hd + hq * hd * d + 3.0 * d * f;
    layer_weight_bytes = 2.0 * params;
    linear_flops_row = 2.0 * params;
    attn_flops_pair = 4.0 * hd * hq;
    qkv_frac = d * (hq + 2 * hkv) * hd / params;
  }
};

// Per-unit cost model of the two restore paths (Sec. 4.3: per-unit times
// from offline profiling, total time linear in the number of units).
// Copy: evicted blocks x bytes / host-link rate, layer after layer.  Compute
// of the fused rows (recomputed tail + prompt), per layer: the projections
// interpolated from their measured times at 128 / 512 / 2048 rows, attention
// pairs at the measured rates of recompute-like and prompt-like rows (the
// recompute rate reached linearly from the prompt rate between 128 and 2048
// recomputed rows), per-row memory-bound kernels and a fixed per-layer cost.  The two paths overlap
// layer by layer: the part of a layer before the attention that reads copied
// keys (QKV projection, rotary/KV write, attention of the recomputed rows)
// never waits; the rest starts once that layer's copy has landed.
struct CostModel : CostModelShape {
  mzc_model_shape s;
  mzc_profile p;
  CostModel(const mzc_model_shape& s_, const mzc_profile& p_) : CostModelShape(s_), s(s_), p(p_) {}
  double copy_s(int64_t tokens) const {
    const double blocks = static_cast<double>(ceil_div(tokens, 16));
    const double bytes = blocks * s.n_layers * 2.0 * s.n_kv_heads * 16 * s.head_dim * 2;
    return bytes / (p.h2d_gbs * 1e9);
  }
  double gemm_s(double rows) const {
    double us;
    if (rows <= 128) us = p.gemm_us_128;
    else if (rows <= 512) us = p.gemm_us_128 + (rows - 128) * (p.gemm_us_512 - p.gemm_us_128) / 384.0;
    else us = p.gemm_us_512 + (rows - 512) * (p.gemm_us_2048 - p.gemm_us_512) / 1536.0;
    return us * 1e-6;
  }
  // one layer's compute, split at the wait for copied keys: *pre never waits
  double layer_s(int64_t p0, int64_t s1, int64_t n_ctx, int64_t n_prompt, double* pre = nullptr) const {
    const double rows = static_cast<double>(s1 - p0 + n_prompt);
    if (pre) *pre = 0.0;
    if (rows <= 0) return 0.0;
    auto tri = [](double a, double b) { return (b * (b + 1) - a * (a + 1)) / 2.0; };
    const double rec_pairs = tri(static_cast<double>(p0), static_cast<double>(s1));
    const double prm_pairs = tri(static_cast<double>(n_ctx), static_cast<double>(n_ctx + n_prompt));
    // a few hundred recomputed rows fill few CTAs and run near the prompt
    // rate; the recompute rate holds from 2048 rows on
    const double nrec = static_cast<double>(s1 - p0);
    const double w = std::min(1.0, std::max(0.0, (nrec - 128.0) / 1920.0));
    const double rec_rate = p.attn_prompt_tflops + (p.attn_tflops - p.attn_prompt_tflops) * w;
    const double rec_attn = rec_pairs * attn_flops_pair / (rec_rate * 1e12) + nrec * p.attn_row_ns * 1e-9;
    const double prm_attn = prm_pairs * attn_flops_pair / (p.attn_prompt_tflops * 1e12);
    const double g = gemm_s(rows), rw = rows * p.row_ns * 1e-9, fixed = p.layer_us * 1e-6;
    if (pre) *pre = g * qkv_frac + rec_attn + rw * (2.0 / 3.0) + fixed * 0.5;
    return g + rec_attn + prm_attn + rw + fixed;
  }
  // one KV unit (16 rows, every layer) recomputed at the rear of an n_ctx
  // context: the rows at the 2048-row projection rate, their attention over
  // the whole context at the recompute rate, per-row kernels (the eviction
  // policy's t_rec_kv, Algorithm 1)
  double rec_unit_s(int64_t n_ctx) const {
    const double per_row = gemm_s(2048.0) / 2048.0 +
                           static_cast<double>(n_ctx) * attn_flops_pair / (p.attn_tflops * 1e12) +
                           (p.attn_row_ns + p.row_ns) * 1e-9;
    return 16.0 * per_row * s.n_layers;
  }
  // predicted TTFT when [p0, s1) is recomputed and [s1, n_ctx) copied
  double ttft_s(int64_t p0, int64_t s1, int64_t n_ctx, int64_t n_prompt) const {
    double pre = 0.0;
    const double layer = layer_s(p0, s1, n_ctx, n_prompt, &pre);
    const double copy = copy_s(n_ctx - s1);
    if (copy <= 0.0) return s.n_layers * layer;
    const double per_copy = copy / s.n_layers;
    double t = 0.0;
    for (int l = 0; l < s.n_layers; ++l) t = std::max(t + pre, (l + 1) * per_copy) + (layer - pre);
    return t;
  }
};

}  // namespace

extern "C" {

mzc_status mzc_create(const mzc_model_shape* shape, const mzc_options* options,
                      const mzc_weights* weights, mzc_ctx** out) {
  if (!out) return MZC_ERR_INVALID;
  *out = nullptr;
  if (!shape) {
    g_create_error = "shape is NULL";
    return MZC_ERR_INVALID;
  }
  mzc_ctx* ctx = new mzc_ctx();
  mzc_status s = create_impl(shape, options, weights, ctx);
  if (s != MZC_OK) {
    g_create_error = ctx->err;
    destroy_impl(ctx);
    return s;
  }
  *out = ctx;
  return MZC_OK;
}

mzc_status mzc_destroy(mzc_ctx* ctx) { return destroy_impl(ctx); }

mzc_status mzc_prefill(mzc_ctx* ctx, const int32_t* tokens, int64_t n, float* logits_out) {
  if (!ctx) return MZC_ERR_INVALID;
  if (n < 0 || (n > 0 && !tokens)) return ctx->fail(MZC_ERR_INVALID, "bad token buffer");
  CK(cudaSetDevice(ctx->opt.device));
  return run_prefill(ctx, tokens, n, logits_out);
}

mzc_status mzc_evict(mzc_ctx* ctx, int32_t l0, int32_t l1, int64_t t0, int64_t t1, int32_t mode) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  if (mode == MZC_AUTO) {
    if (l0 != 0 || l1 != ctx->shape.n_layers)
      return ctx->fail(MZC_ERR_INVALID, "AUTO eviction covers every layer");
    const int64_t n_ctx = ctx->st.n_ctx();
    if (t0 < 0 || t0 >= n_ctx) return ctx->fail(MZC_ERR_RANGE, "token range outside the context");
    const int64_t p = t0 / 16 * 16;
    int64_t split = n_ctx;
    if (ctx->policy == MZC_POLICY_COPY) split = p;
    else if (ctx->policy == MZC_POLICY_HYBRID) {
      mzc_status e = mzc_plan_split_ctx(ctx, p, 0, &split);
      if (e != MZC_OK) return ctx->fail(e, "hybrid split failed");
    }
    if (split > p) {
      mzc_status e = mzc_evict(ctx, 0, l1, p, split, MZC_DROP);
      if (e != MZC_OK) return e;
    }
    if (split < n_ctx) return mzc_evict(ctx, 0, l1, split, n_ctx, MZC_COPY);
    return MZC_OK;
  }
  std::vector<int32_t> freed;
  if (mode == MZC_DROP && t0 >= 0 && t1 <= ctx->st.n_ctx() && t0 < t1 && l0 >= 0 && l1 <= ctx->shape.n_layers) {
    for (int32_t l = l0; l < l1; ++l)
      for (int64_t b = t0 / 16; b < ceil_div(t1, 16); ++b)
        if (ctx->st.at(l, b).phys >= 0) freed.push_back(ctx->st.at(l, b).phys);
  }
  if (mode == MZC_COPY) {
    mzc_status e = ensure_store(ctx);
    if (e != MZC_OK) return e;
  }
  std::vector<mzc::EvictMove> moves;
  mzc_status s = ctx->st.evict_range(l0, l1, t0, t1, mode, &moves);
  if (s != MZC_OK) return ctx->from_state(s);
  if (mode == MZC_COPY) return copy_out(ctx, moves);
  return poison(ctx, freed);
}

mzc_status mzc_evict_blocks(mzc_ctx* ctx, const int32_t* layer, const int64_t* blk, int64_t n, int32_t mode) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  if (mode == MZC_COPY) {
    mzc_status e = ensure_store(ctx);
    if (e != MZC_OK) return e;
  }
  std::vector<mzc::EvictMove> moves;
  mzc_status s = ctx->st.evict_blocks(layer, blk, n, mode, &moves);
  if (s != MZC_OK) return ctx->from_state(s);
  return copy_out(ctx, moves);
}

mzc_status mzc_evict_weights(mzc_ctx* ctx, int32_t l0, int32_t l1) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  mzc_status s = ctx->st.evict_weights(l0, l1);
  if (s != MZC_OK) return ctx->from_state(s);
  for (int32_t l = l0; l < l1; ++l) {
    LayerDev& Ld = ctx->layers[l];
    if (!Ld.host_master) CK(cudaHostAlloc(&Ld.host_master, Ld.bytes, cudaHostAllocDefault));
    CK(cudaMemcpyAsync(Ld.host_master, Ld.base, Ld.bytes, cudaMemcpyDeviceToHost, ctx->cs));
    CK(cudaMemsetAsync(Ld.base, 0xFF, Ld.bytes, ctx->cs));  // NaN until restored
  }
  CK(cudaStreamSynchronize(ctx->cs));
  return MZC_OK;
}

mzc_status mzc_restore_async(mzc_ctx* ctx) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  std::vector<mzc_copy_run> runs;
  std::vector<int32_t> wl;
  // per-block flags: the destination blocks read as absent from here on (their
  // flags are cleared on the compute stream, ahead of any attention of the
  // next prefill); the copy stream sets each run's flags after its data
  const bool set_flags = ctx->d_flags && ctx->opt.overlap && ctx->codec == MZC_CODEC_NONE;
  // The plan is made a layer at a time, each layer's copies issued before the
  // next layer is planned, so the first copy leaves as soon as its layer is
  // planned.  With per-block flags every destination is planned first: the
  // flags are cleared before any copy.
  bool any = false;
  mzc_status s = set_flags ? ctx->st.plan_restore(&runs, &wl) : ctx->st.begin_restore(&any);
  if (s != MZC_OK) return ctx->from_state(s);
  if (!ctx->st.restore_in_flight()) return MZC_OK;
  cudaStream_t xs = ctx->xs;
  CK(cudaEventRecord(ctx->ev_c0, xs));
  if (set_flags && !runs.empty()) {
    for (const mzc_copy_run& r : runs)
      CK(cudaMemsetAsync(ctx->d_flags + r.phys_begin, 0, static_cast<size_t>(r.n_blocks) * 4, ctx->cs));
    CK(cudaEventRecord(ctx->ev_clear, ctx->cs));
    CK(cudaStreamWaitEvent(xs, ctx->ev_clear, 0));
  }
  size_t ri = 0, wi = 0;
  int64_t bytes = 0, copies = 0;
  for (int32_t l = 0; l < ctx->shape.n_layers; ++l) {
    if (!set_flags) {
      bool w = false;
      ctx->st.plan_restore_layer(l, &runs, &w);
      if (w) wl.push_back(l);
    }
    if (wi < wl.size() && wl[wi] == l) {
      const LayerDev& Ld = ctx->layers[l];
      CK(cudaMemcpyAsync(Ld.base, Ld.host_master, Ld.bytes, cudaMemcpyHostToDevice, xs));
      bytes += static_cast<int64_t>(Ld.bytes);
      ++copies;
      ++wi;
    }
    CK(cudaEventRecord(ctx->ev_w[l], xs));
    if (ctx->codec == MZC_CODEC_NONE) {
      while (ri < runs.size() && runs[ri].layer == l) {
        const mzc_copy_run& r = runs[ri++];
        const int64_t nb = static_cast<int64_t>(r.n_blocks) * ctx->block_bytes;
        CK(cudaMemcpyAsync(ctx->d_pool + r.phys_begin * ctx->block_bytes, ctx->h_store + r.host_off,
                           nb, cudaMemcpyHostToDevice, xs));
        if (set_flags)
          CK(cudaMemcpyAsync(ctx->d_flags + r.phys_begin, ctx->h_ones, static_cast<size_t>(r.n_blocks) * 4,
                             cudaMemcpyHostToDevice, xs));
        bytes += nb;
        ++copies;
      }
      CK(cudaEventRecord(ctx->ev_kv[l], xs));
      continue;
    }
    // compressed: the layer's runs land packed in staging buffer l % 2 (free
    // once layer l - 2 is decoded), then the decode stream writes the pool
    const size_t r0 = ri;
    uint8_t* stage = ctx->d_rstage[l & 1];
    if (l >= 2) CK(cudaStreamWaitEvent(xs, ctx->ev_dec[l - 2], 0));
    int64_t at = 0;
    while (ri < runs.size() && runs[ri].layer == l) {
      const mzc_copy_run& r = runs[ri++];
      const int64_t nb = static_cast<int64_t>(r.n_blocks) * ctx->slot_bytes;
      CK(cudaMemcpyAsync(stage + at, ctx->h_store + r.host_off, nb, cudaMemcpyHostToDevice, xs));
      at += nb;
      bytes += nb;
      ++copies;
    }
    CK(cudaEventRecord(ctx->ev_h2d[l], xs));
    CK(cudaStreamWaitEvent(ctx->ds, ctx->ev_h2d[l], 0));
    at = 0;
    for (size_t k = r0; k < ri; ++k) {
      const mzc_copy_run& r = runs[k];
      CK(mzc::launch_q8_decode(stage + at, r.n_blocks, ctx->block_bytes / 2, nullptr, r.phys_begin,
                               ctx->shape.kv_dtype, ctx->d_pool, ctx->ds));
      at += static_cast<int64_t>(r.n_blocks) * ctx->slot_bytes;
    }
    CK(cudaEventRecord(ctx->ev_dec[l], ctx->ds));
    CK(cudaEventRecord(ctx->ev_kv[l], ctx->ds));
  }
  if (ctx->codec != MZC_CODEC_NONE) {
    // the copy stream's end event covers the decodes
    CK(cudaEventRecord(ctx->ev_dec[0], ctx->ds));
    CK(cudaStreamWaitEvent(xs, ctx->ev_dec[0], 0));
  }
  CK(cudaEventRecord(ctx->ev_c1, xs));
  ctx->restore_issued = true;
  ctx->last.bytes_h2d_last = bytes;
  ctx->last.copies_last = copies;
  return MZC_OK;
}

mzc_status mzc_recompute_tail(mzc_ctx* ctx, int64_t p, int64_t n) {
  if (!ctx) return MZC_ERR_INVALID;
  return ctx->from_state(ctx->st.recompute_tail(p, n));
}

mzc_status mzc_set_policy(mzc_ctx* ctx, int32_t policy, const mzc_profile* profile) {
  if (!ctx) return MZC_ERR_INVALID;
  if (policy < MZC_POLICY_COPY || policy > MZC_POLICY_HYBRID)
    return ctx->fail(MZC_ERR_INVALID, "unknown policy");
  ctx->policy = policy;
  if (profile) ctx->prof = *profile;
  return MZC_OK;
}

}  // extern "C"

namespace {

// The split s minimising the predicted TTFT among the block boundaries from p
// and n_ctx itself.  A split other than copy-only (s = p) must be predicted
// min_gain faster, and, when headroom < 1, keep the compute of a layer within
// headroom x the copy time of a layer: the layer-by-layer overlap then stays
// bound by the link, whose rate the model knows best, and an underestimate of
// the compute cannot turn the step compute-bound.
mzc_status plan_split_impl(const mzc_model_shape* shape, const mzc_profile* profile, int64_t p,
                           int64_t n_ctx, int64_t n_prompt, double min_gain, double headroom,
                           int64_t* s_out) {
  if (!shape || !s_out || p < 0 || n_ctx < p || n_prompt < 0) return MZC_ERR_INVALID;
  const mzc_profile prof = profile ? *profile : default_profile();
  if (prof.h2d_gbs <= 0 || prof.gemm_us_128 <= 0 || prof.gemm_us_512 <= 0 || prof.gemm_us_2048 <= 0 ||
      prof.attn_tflops <= 0 || prof.attn_row_ns < 0 || prof.attn_prompt_tflops <= 0 || prof.row_ns < 0 ||
      prof.layer_us < 0)
    return MZC_ERR_INVALID;
  CostModel cm(*shape, prof);
  const double copy_only = cm.ttft_s(p, p, n_ctx, n_prompt);
  int64_t best = p;
  double best_t = copy_only;
  for (int64_t s = p + 16;; s += 16) {
    const int64_t sc = std::min(s, n_ctx);
    const double t = cm.ttft_s(p, sc, n_ctx, n_prompt);
    bool fits = true;
    if (headroom < 1.0 && sc < n_ctx)
      fits = cm.layer_s(p, sc, n_ctx, n_prompt) <= headroom * cm.copy_s(n_ctx - sc) / shape->n_layers;
    if (fits && t < best_t) {
      best_t = t;
      best = sc;
    }
    if (sc >= n_ctx) break;
  }
  if (best_t > (1.0 - min_gain) * copy_only) best = p;
  *s_out = best;
  return MZC_OK;
}

}  // namespace

extern "C" {

// Raw store: a 1% predicted gain with every layer's compute within 95% of
// its copy (3B sweep: copy-only was kept at f <= 0.25 and beaten at f = 0.75
// and 1; a 1% margin without the headroom made f = 0.5 slower).
mzc_status mzc_plan_split(const mzc_model_shape* shape, const mzc_profile* profile, int64_t p,
                          int64_t n_ctx, int64_t n_prompt, int64_t* s_out) {
  return plan_split_impl(shape, profile, p, n_ctx, n_prompt, 0.01, 0.95, s_out);
}

mzc_status mzc_plan_split_ctx(mzc_ctx* ctx, int64_t p, int64_t n_prompt, int64_t* s_out) {
  if (!ctx || !s_out) return MZC_ERR_INVALID;
  // the model prices a copied block at its stored size over the link; a
  // compressed store moves slot_bytes per block.  Its decode kernels share the
  // SMs with the recompute, which the model does not price, so a compressed
  // store splits only for a predicted gain of 5%.
  mzc_profile pr = ctx->prof;
  pr.h2d_gbs *= static_cast<double>(ctx->block_bytes) / static_cast<double>(ctx->slot_bytes);
  const bool raw = ctx->codec == MZC_CODEC_NONE;
  mzc_status e = plan_split_impl(&ctx->shape, &pr, p, ctx->st.n_ctx(), n_prompt, raw ? 0.01 : 0.05,
                                 raw ? 0.95 : 1.0, s_out);
  return e == MZC_OK ? e : ctx->fail(e, "hybrid split failed");
}

mzc_status mzc_evict_size_plan(mzc_ctx* ctx, mzc_evict_plan* out) {
  if (!ctx || !out) return MZC_ERR_INVALID;
  const int32_t L = ctx->shape.n_layers;
  int64_t c0 = 0, r0 = 0;
  int32_t w0 = 0;
  if (ctx->st.evicted_layout(&c0, &r0, &w0) != MZC_OK)
    return ctx->fail(MZC_ERR_STATE, "evict_size needs the backward-out placement it makes (and no "
                                    "restore or recompute pending)");
  const double link = ctx->prof.h2d_gbs * 1e9;
  if (!(link > 0)) return ctx->fail(MZC_ERR_INVALID, "the profile has no host-link rate");
  mzc_evict_plan p{};
  p.t_copy_w = static_cast<double>(ctx->layers[0].bytes) / link;
  p.t_copy_kv = static_cast<double>(L) * static_cast<double>(ctx->slot_bytes) / link;
  p.t_rec_kv = CostModel(ctx->shape, ctx->prof).rec_unit_s(ctx->st.n_ctx());
  p.kv_total = ceil_div(ctx->st.n_ctx(), 16);
  p.w_total = L;
  p.w_evicted = w0;
  p.kv_copy = c0;
  p.kv_rec = r0;
  p.kv_bytes = static_cast<int64_t>(L) * ctx->block_bytes;
  p.w_bytes = static_cast<int64_t>(ctx->layers[0].bytes);
  *out = p;
  return MZC_OK;
}

mzc_status mzc_evict_size(mzc_ctx* ctx, int64_t bytes, int64_t* freed_out, int32_t* stage_out) {
  if (!ctx) return MZC_ERR_INVALID;
  const int32_t L = ctx->shape.n_layers;
  mzc_evict_plan p{};
  mzc_status e0 = mzc_evict_size_plan(ctx, &p);
  if (e0 != MZC_OK) return e0;
  const int64_t c0 = p.kv_copy, r0 = p.kv_rec;
  const int32_t w0 = p.w_evicted;
  int64_t freed = 0;
  int32_t stage = 0;
  mzc_status e = mzc_plan_evict_size(&p, bytes, &freed, &stage);
  if (e != MZC_OK) return ctx->fail(e, "invalid eviction request");
  mzc::EvictSizeSteps steps;
  mzc::evict_size_steps(ctx->st.n_ctx(), L, c0, r0, w0, p, &steps);
  if (steps.copy_t1 > steps.copy_t0) {
    e = mzc_evict(ctx, 0, L, steps.copy_t0, steps.copy_t1, MZC_COPY);
    if (e != MZC_OK) return e;
  }
  if (steps.drop_t1 > steps.drop_t0) {
    e = mzc_evict(ctx, 0, L, steps.drop_t0, steps.drop_t1, MZC_DROP);
    if (e != MZC_OK) return e;
  }
  if (steps.w1 > steps.w0) {
    e = mzc_evict_weights(ctx, steps.w0, steps.w1);
    if (e != MZC_OK) return e;
  }
  if (freed_out) *freed_out = freed;
  if (stage_out) *stage_out = stage;
  return MZC_OK;
}

mzc_status mzc_truncate(mzc_ctx* ctx, int64_t n_ctx) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  std::vector<int32_t> freed;
  if (n_ctx >= 0 && n_ctx <= ctx->st.n_ctx())
    for (int32_t l = 0; l < ctx->shape.n_layers; ++l)
      for (int64_t b = ceil_div(n_ctx, 16); b < ceil_div(ctx->st.n_ctx(), 16); ++b)
        if (ctx->st.at(l, b).st == MZC_RESIDENT && ctx->st.at(l, b).phys >= 0)
          freed.push_back(ctx->st.at(l, b).phys);
  mzc_status s = ctx->st.truncate(n_ctx);
  if (s != MZC_OK) return ctx->from_state(s);
  ctx->tokens.resize(static_cast<size_t>(n_ctx));
  return poison(ctx, freed);
}

mzc_status mzc_sync(mzc_ctx* ctx) {
  if (!ctx) return MZC_ERR_INVALID;
  CK(cudaSetDevice(ctx->opt.device));
  if (ctx->st.recompute_pending()) return run_prefill(ctx, nullptr, 0, nullptr);
  CK(cudaStreamSynchronize(ctx->cs));
  CK(cudaStreamSynchronize(ctx->xs));
  mzc_status s = check_status(ctx);
  if (s != MZC_OK) return s;
  if (ctx->st.restore_in_flight()) {
    ctx->st.complete(0);
    ctx->restore_issued = false;
  }
  return MZC_OK;
}

mzc_status mzc_query(mzc_ctx* ctx, int32_t layer, int64_t b, int32_t* state, int32_t* phys) {
  if (!ctx) return MZC_ERR_INVALID;
  if (layer < 0 || layer >= ctx->shape.n_layers || b < 0 || b >= ctx->nblk)
    return ctx->fail(MZC_ERR_RANGE, "index out of range");
  const mzc::BlockEntry& e = ctx->st.at(layer, b);
  if (state) *state = e.st;
  if (phys) *phys = e.phys;
  return MZC_OK;
}

mzc_status mzc_read_kv(mzc_ctx* ctx, int32_t layer, int64_t b, void* k_host, void* v_host) {
  if (!ctx || !k_host || !v_host) return MZC_ERR_INVALID;
  if (layer < 0 || layer >= ctx->shape.n_layers || b < 0 || b >= ceil_div(ctx->st.n_ctx(), 16))
    return ctx->fail(MZC_ERR_RANGE, "block outside the context");
  const mzc::BlockEntry& e = ctx->st.at(layer, b);
  if (e.st != MZC_RESIDENT) return ctx->fail(MZC_ERR_STATE, "block is not resident");
  CK(cudaSetDevice(ctx->opt.device));
  const int64_t half = ctx->block_bytes / 2;
  const uint8_t* src = ctx->d_pool + static_cast<int64_t>(e.phys) * ctx->block_bytes;
  CK(cudaMemcpy(k_host, src, half, cudaMemcpyDeviceToHost));
  CK(cudaMemcpy(v_host, src + half, half, cudaMemcpyDeviceToHost));
  return MZC_OK;
}

mzc_status mzc_read_kv_all(mzc_ctx* ctx, int64_t n, float* k_host, float* v_host) {
  if (!ctx || !k_host || !v_host) return MZC_ERR_INVALID;
  if (n < 0 || n > ctx->st.n_ctx()) return ctx->fail(MZC_ERR_RANGE, "n beyond the context");
  CK(cudaSetDevice(ctx->opt.device));
  const mzc_model_shape& s = ctx->shape;
  const int64_t hkv = s.n_kv_heads, hd = s.head_dim, nb = ceil_div(n, 16);
  for (int32_t l = 0; l < s.n_layers; ++l) {
    for (int64_t b = 0; b < nb; ++b) {
      const mzc::BlockEntry& e = ctx->st.at(l, b);
      if (e.st != MZC_RESIDENT) return ctx->fail(MZC_ERR_STATE, "block is not resident");
      ctx->h_list[b] = e.phys;
    }
    if (nb == 0) continue;
    CK(cudaMemcpyAsync(ctx->d_list, ctx->h_list, nb * 4, cudaMemcpyHostToDevice, ctx->cs));
    CK(mzc::launch_gather_blocks(ctx->d_pool, ctx->d_list, nb, ctx->block_bytes, ctx->d_staging, ctx->cs));
    CK(cudaMemcpyAsync(ctx->h_staging, ctx->d_staging, nb * ctx->block_bytes, cudaMemcpyDeviceToHost, ctx->cs));
    CK(cudaStreamSynchronize(ctx->cs));
    const uint16_t* blocks = reinterpret_cast<const uint16_t*>(ctx->h_staging);
    for (int64_t p = 0; p < n; ++p) {
      const int64_t b = p / 16, slot = p % 16;
      for (int64_t h = 0; h < hkv; ++h) {
        const uint16_t* kb = blocks + b * 2 * hkv * 16 * hd + (h * 16 + slot) * hd;
        const uint16_t* vb = kb + hkv * 16 * hd;
        float* ko = k_host + ((static_cast<int64_t>(l) * n + p) * hkv + h) * hd;
        float* vo = v_host + ((static_cast<int64_t>(l) * n + p) * hkv + h) * hd;
        for (int64_t c = 0; c < hd; ++c) {  // the pool is fp16-encoded for both KV types
          __half_raw rk, rv;
          rk.x = kb[c];
          rv.x = vb[c];
          ko[c] = __half2float(__half(rk));
          vo[c] = __half2float(__half(rv));
        }
      }
    }
  }
  return MZC_OK;
}

mzc_status mzc_stats(mzc_ctx* ctx, mzc_stats_t* out) {
  if (!ctx || !out) return MZC_ERR_INVALID;
  ctx->st.counts(out);
  out->bytes_h2d_last = ctx->last.bytes_h2d_last;
  out->copies_last = ctx->last.copies_last;
  out->rows_last = ctx->last.rows_last;
  out->recompute_rows_last = ctx->last.recompute_rows_last;
  return MZC_OK;
}

mzc_status mzc_last_times(mzc_ctx* ctx, float* ms3) {  // ms3 holds 4 floats
  if (!ctx || !ms3) return MZC_ERR_INVALID;
  ms3[0] = ms3[1] = ms3[2] = ms3[3] = 0.0f;
  if (cudaEventElapsedTime(&ms3[0], ctx->ev_t0, ctx->ev_t1) != cudaSuccess) ms3[0] = -1.0f;
  if (!ctx->ttft_from_copy || cudaEventElapsedTime(&ms3[1], ctx->ev_c0, ctx->ev_c1) != cudaSuccess) ms3[1] = -1.0f;
  if (!ctx->lm_timed || cudaEventElapsedTime(&ms3[2], ctx->ev_l0, ctx->ev_l1) != cudaSuccess) ms3[2] = -1.0f;
  if (cudaEventElapsedTime(&ms3[3], ctx->ttft_from_copy ? ctx->ev_c0 : ctx->ev_t0, ctx->ev_t1) != cudaSuccess)
    ms3[3] = -1.0f;
  cudaGetLastError();
  return MZC_OK;
}

mzc_status mzc_set_kernel_timing(mzc_ctx* ctx, int32_t class_mask) {
  if (!ctx) return MZC_ERR_INVALID;
  ctx->ktime_mask = class_mask;
  for (auto& k : ctx->kstat) k = mzc_kernel_stat{};
  return MZC_OK;
}

mzc_status mzc_kernel_stats(mzc_ctx* ctx, int32_t cls, mzc_kernel_stat* out) {
  if (!ctx || !out || cls < 0 || cls >= MZC_K_NCLASS) return MZC_ERR_INVALID;
  *out = ctx->kstat[cls];
  return MZC_OK;
}

const char* mzc_last_error(mzc_ctx* ctx) {
  if (!ctx) return g_create_error.c_str();
  return ctx->err.c_str();
}

mzc_status mzc_profile_measure(mzc_ctx* ctx, mzc_profile* out) {
  if (!ctx || !out) return MZC_ERR_INVALID;
  if (ctx->st.restore_in_flight() || ctx->st.recompute_pending())
    return ctx->fail(MZC_ERR_STATE, "profiling needs a ctx with no restore or recompute pending");
  CK(cudaSetDevice(ctx->opt.device));
  mzc_profile p = ctx->prof;
  cudaEvent_t a, b;
  CK(cudaEventCreate(&a));
  CK(cudaEventCreate(&b));
  float ms = 0.0f;
  // Host link: timed pinned -> device copies on the copy stream, into device
  // memory that holds no live KV -- the longest run of free pool blocks, which
  // is poisoned again afterwards like every freed block, or the ctx's staging
  // buffer, whichever is larger.  Resident blocks are never written.
  {
    int64_t run0 = 0;
    const int64_t run_n = ctx->st.largest_free_pool_run(&run0);
    const int64_t staging = ctx->nblk * ctx->block_bytes;
    const bool use_pool = run_n * ctx->block_bytes > staging;
    uint8_t* dst = use_pool ? ctx->d_pool + run0 * ctx->block_bytes : ctx->d_staging;
    const int64_t bytes = std::min<int64_t>(256LL << 20, use_pool ? run_n * ctx->block_bytes : staging);
    // about 1 GiB in all (4 to 64 copies), so small buffers still time steadily
    const int reps = static_cast<int>(std::min<int64_t>(64, std::max<int64_t>(4, (1LL << 30) / bytes)));
    uint8_t* h = nullptr;
    CK(cudaHostAlloc(&h, bytes, cudaHostAllocDefault));
    std::memset(h, 1, bytes);
    CK(cudaMemcpyAsync(dst, h, bytes, cudaMemcpyHostToDevice, ctx->xs));
    CK(cudaEventRecord(a, ctx->xs));
    for (int i = 0; i < reps; ++i) CK(cudaMemcpyAsync(dst, h, bytes, cudaMemcpyHostToDevice, ctx->xs));
    CK(cudaEventRecord(b, ctx->xs));
    CK(cudaEventSynchronize(b));
    CK(cudaEventElapsedTime(&ms, a, b));
    p.h2d_gbs = static_cast<double>(reps) * bytes / (ms * 1e-3) / 1e9;
    if (use_pool)
      CK(mzc::launch_poison_run(ctx->d_pool, run0, ceil_div(bytes, ctx->block_bytes), ctx->block_bytes, ctx->xs));
    CK(cudaStreamSynchronize(ctx->xs));
    CK(cudaFreeHost(h));
  }
  // A whole layer's four projections on scratch activations at 128, 512 and
  // 2048 rows (capped by max_rows).
  {
    const LayerDev& W = ctx->layers[0];
    const int64_t d = ctx->shape.d_model, hq = ctx->shape.n_q_heads, hd = ctx->shape.head_dim;
    auto layer_gemms = [&](int64_t m) -> cudaError_t {
      // (timing only: the activation buffers hold whatever the last prefill
      // left, so the GEMMs report nothing to the status word)
      cudaError_t e = mzc::launch_gemm(ctx->tm_h, W.tm_qkv, ctx->d_qkv, m, ctx->qkv_dim, d, mzc::EPI_STORE_BF16, nullptr, ctx->cs, nullptr, &ctx->gsplit);
      if (e == cudaSuccess) e = mzc::launch_gemm(ctx->tm_attn, W.tm_o, ctx->d_x, m, d, hq * hd, mzc::EPI_ADD_F32, nullptr, ctx->cs, nullptr, &ctx->gsplit);
      if (e == cudaSuccess) e = mzc::launch_gemm(ctx->tm_h, W.tm_13, ctx->d_act, m, 2 * ctx->f_pad, d, mzc::EPI_SWIGLU_BF16, nullptr, ctx->cs, nullptr, &ctx->gsplit);
      if (e == cudaSuccess) e = mzc::launch_gemm(ctx->tm_act, W.tm_2, ctx->d_x, m, d, ctx->f_pad, mzc::EPI_ADD_F32, nullptr, ctx->cs, nullptr, &ctx->gsplit);
      return e;
    };
    const int64_t sizes[3] = {128, 512, 2048};
    double* outs[3] = {&p.gemm_us_128, &p.gemm_us_512, &p.gemm_us_2048};
    for (int t = 0; t < 3; ++t) {
      const int64_t m = std::min<int64_t>(ctx->max_rows, sizes[t]);
      CK(layer_gemms(m));
      CK(cudaEventRecord(a, ctx->cs));
      for (int i = 0; i < 5; ++i) CK(layer_gemms(m));
      CK(cudaEventRecord(b, ctx->cs));
      CK(cudaEventSynchronize(b));
      CK(cudaEventElapsedTime(&ms, a, b));
      // rows beyond max_rows would run in chunks: scale linearly
      if (ms > 0) *outs[t] = ms * 1e3 / 5.0 * static_cast<double>(sizes[t]) / static_cast<double>(m);
    }
  }
  // attention over the resident context, when there is one: 1024
  // recompute-like rows (causal) starting at the middle and at the start of
  // the context -- two points that give a per-key rate and a per-row cost --
  // and 128 prompt-like rows at its end (split over the whole context)
  {
    const int64_t n_ctx = ctx->st.n_ctx();
    bool resident = n_ctx >= 2048;
    for (int32_t l = 0; l < ctx->shape.n_layers && resident; ++l)
      for (int64_t blk = 0; blk < ceil_div(n_ctx, 16) && resident; ++blk)
        resident = ctx->st.at(l, blk).st == MZC_RESIDENT;
    if (resident) {
      const mzc_model_shape& s = ctx->shape;
      std::vector<int32_t> tab;
      ctx->st.block_table(&tab);
      double t_sec[3] = {0, 0, 0}, pairs_k[3] = {0, 0, 0};
      int64_t rows_k[3] = {0, 0, 0};
      for (int kind = 0; kind < 3; ++kind) {
        const int64_t rows = std::min<int64_t>(ctx->max_rows, kind < 2 ? 1024 : 128);
        const int64_t first = kind == 0 ? n_ctx / 2 : (kind == 1 ? 0 : n_ctx - rows);
        int32_t* hp = reinterpret_cast<int32_t*>(ctx->h_meta);
        for (int64_t i = 0; i < rows; ++i) hp[i] = static_cast<int32_t>(first + i);
        std::memcpy(hp + rows, tab.data(), ctx->nblk * 4);
        int32_t* dp = reinterpret_cast<int32_t*>(ctx->d_meta);
        CK(cudaMemcpyAsync(dp, hp, (rows + ctx->nblk) * 4, cudaMemcpyHostToDevice, ctx->cs));
        const int64_t max_keys = first + rows;
        auto run = [&]() {
          return mzc::launch_attention(ctx->d_q, dp, rows, s.n_q_heads, s.n_kv_heads, s.head_dim, dp + rows,
                                       ctx->nblk, ctx->d_pool, ctx->st.pool_blocks(), s.kv_dtype,
                                       ctx->d_attn, ctx->d_scratch, ctx->scratch_bytes, max_keys,
                                       ctx->num_sms, ctx->d_status, ctx->cs);
        };
        CK(run());
        CK(cudaEventRecord(a, ctx->cs));
        for (int i = 0; i < 3; ++i) CK(run());
        CK(cudaEventRecord(b, ctx->cs));
        CK(cudaEventSynchronize(b));
        CK(cudaEventElapsedTime(&ms, a, b));
        for (int64_t i = 0; i < rows; ++i) pairs_k[kind] += static_cast<double>(first + i + 1);
        t_sec[kind] = ms * 1e-3 / 3.0;
        rows_k[kind] = rows;
      }
      const double fpp = 4.0 * s.head_dim * s.n_q_heads;
      if (t_sec[0] > t_sec[1] && pairs_k[0] > pairs_k[1] && rows_k[0] == rows_k[1]) {
        const double sec_per_pair = (t_sec[0] - t_sec[1]) / (pairs_k[0] - pairs_k[1]);
        p.attn_tflops = fpp / sec_per_pair / 1e12;
        p.attn_row_ns = std::max(0.0, (t_sec[1] - pairs_k[1] * sec_per_pair) / rows_k[1] * 1e9);
      } else if (t_sec[0] > 0) {
        p.attn_tflops = pairs_k[0] * fpp / t_sec[0] / 1e12;
        p.attn_row_ns = 0.0;
      }
      if (t_sec[2] > 0) p.attn_prompt_tflops = pairs_k[2] * fpp / t_sec[2] / 1e12;
    }
  }
  // memory-bound kernels per row (two RMSNorms and the rotary/KV write,
  // approximated by three norms): the per-row slope between a quarter and all
  // of up to 8192 rows (both large enough to stream), and the fixed per-layer
  // cost from the same launches at one row
  {
    auto norms = [&](int64_t rows) -> cudaError_t {
      cudaError_t e = cudaSuccess;
      for (int i = 0; i < 3 && e == cudaSuccess; ++i)
        e = mzc::launch_rmsnorm(ctx->d_x, ctx->layers[0].attn_norm, rows, ctx->shape.d_model, 1e-5f,
                                ctx->d_h, ctx->cs);
      return e;
    };
    const int64_t rows = std::min<int64_t>(ctx->max_rows, 8192);
    const int64_t sizes[3] = {1, std::max<int64_t>(1, rows / 4), rows};
    float ms[3] = {0.0f, 0.0f, 0.0f};
    for (int pass = 0; pass < 3; ++pass) {
      CK(norms(sizes[pass]));
      CK(cudaEventRecord(a, ctx->cs));
      for (int i = 0; i < 20; ++i) CK(norms(sizes[pass]));
      CK(cudaEventRecord(b, ctx->cs));
      CK(cudaEventSynchronize(b));
      CK(cudaEventElapsedTime(&ms[pass], a, b));
    }
    p.layer_us = ms[0] * 1e3 / 20.0 * (8.0 / 3.0);  // ~8 launches per layer
    p.row_ns = sizes[2] > sizes[1]
                   ? std::max(0.0, (static_cast<double>(ms[2]) - ms[1]) * 1e6 / 20.0 /
                                       static_cast<double>(sizes[2] - sizes[1]))
                   : 0.0;
  }
  CK(cudaEventDestroy(a));
  CK(cudaEventDestroy(b));
  mzc_status s = check_status(ctx);
  if (s != MZC_OK) return s;
  ctx->prof = p;
  *out = p;
  return MZC_OK;
}

// ---- single kernels ---------------------------------------------------------

static int sm_count() {
  static int n = 0;
  if (n == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
  }
  return n;
}

static mzc_status kernel_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return MZC_OK;
  g_create_error = std::string(what) + ": " + cudaGetErrorString(e);
  return MZC_ERR_CUDA;
}
#define KCK(expr) return kernel_status((expr), __func__)

mzc_status mzc_k_rmsnorm(const float* x, const float* g, int64_t n, int32_t d, float eps,
                         uint16_t* y, void* stream) {
  if (!x || !g || !y || d % 8 != 0 || n < 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_rmsnorm(x, g, n, d, eps, y, static_cast<cudaStream_t>(stream)));
}

mzc_status mzc_k_gemm(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                      int64_t k, int32_t epilogue, void* stream) {
  if (!a || !w || !out || m < 0 || n <= 0 || k <= 0 || k % 8 != 0 || n % 16 != 0)
    return MZC_ERR_INVALID;
  if (epilogue < 0 || epilogue > 2) return MZC_ERR_INVALID;
  if (epilogue == mzc::EPI_SWIGLU_BF16 && n % (2 * mzc::kSwigluGroup) != 0) return MZC_ERR_INVALID;
  if (m == 0) return MZC_OK;
  CUtensorMap ta;
  mzc::GemmWeight tw;
  if (!mzc::make_tmap_f16(&ta, a, static_cast<uint64_t>(m), static_cast<uint64_t>(k), 128) ||
      !mzc::make_gemm_weight(&tw, w, static_cast<uint64_t>(n), static_cast<uint64_t>(k)))
    return MZC_ERR_CUDA;
  KCK(mzc::launch_gemm(ta, tw, out, m, n, k, epilogue, nullptr, static_cast<cudaStream_t>(stream), a));
}

static int device_sms() {
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return 0;
  return sms;
}

mzc_status mzc_k_gemm_norm_out(const uint16_t* a, const uint16_t* w, float* x, int64_t m, int64_t n,
                               int64_t k, const float* g, uint16_t* h, float* ss, int32_t* status,
                               void* stream) {
  if (!a || !w || !x || !g || !h || !ss || m <= mzc::kGemvMaxRows || m > 256 || n <= 0 || n % 128 != 0 ||
      k <= 0 || k % 8 != 0)
    return MZC_ERR_INVALID;
  const int sms = device_sms();
  if (sms <= 0) return MZC_ERR_CUDA;
  if (!mzc::gemm_splitk_launches(m, n, k, mzc::EPI_ADD_F32, sms)) return MZC_ERR_INVALID;
  CUtensorMap ta;
  mzc::GemmWeight tw;
  if (!mzc::make_tmap_f16(&ta, a, static_cast<uint64_t>(m), static_cast<uint64_t>(k), 128) ||
      !mzc::make_gemm_weight(&tw, w, static_cast<uint64_t>(n), static_cast<uint64_t>(k)))
    return MZC_ERR_CUDA;
  mzc::RowNorm rn;
  rn.g = g;
  rn.h = h;
  rn.ss = ss;
  rn.nt = static_cast<int>(n / 128);
  rn.d = static_cast<float>(n);
  KCK(mzc::launch_gemm(ta, tw, x, m, n, k, mzc::EPI_ADD_F32, status, static_cast<cudaStream_t>(stream), a,
                       nullptr, &rn));
}

mzc_status mzc_k_gemm_norm_in(const uint16_t* h, const uint16_t* w, void* out, int64_t m, int64_t n,
                              int64_t k, int32_t epilogue, const float* ss, float eps, int32_t* status,
                              void* stream) {
  if (!h || !w || !out || !ss || m <= mzc::kGemvMaxRows || m > 256 || n <= 0 || n % 16 != 0 || k <= 0 ||
      k % 128 != 0)
    return MZC_ERR_INVALID;
  if (epilogue != mzc::EPI_STORE_BF16 && epilogue != mzc::EPI_SWIGLU_BF16) return MZC_ERR_INVALID;
  if (epilogue == mzc::EPI_SWIGLU_BF16 && n % (2 * mzc::kSwigluGroup) != 0) return MZC_ERR_INVALID;
  CUtensorMap ta;
  mzc::GemmWeight tw;
  if (!mzc::make_tmap_f16(&ta, h, static_cast<uint64_t>(m), static_cast<uint64_t>(k), 128) ||
      !mzc::make_gemm_weight(&tw, w, static_cast<uint64_t>(n), static_cast<uint64_t>(k)))
    return MZC_ERR_CUDA;
  mzc::RowNorm rn;
  rn.ss = const_cast<float*>(ss);
  rn.nt = static_cast<int>(k / 128);
  rn.d = static_cast<float>(k);
  rn.eps = eps;
  KCK(mzc::launch_gemm(ta, tw, out, m, n, k, epilogue, status, static_cast<cudaStream_t>(stream), h,
                       nullptr, &rn));
}

mzc_status mzc_k_gemm_split(const uint16_t* a, const uint16_t* w, float* out, int64_t m, int64_t n,
                            int64_t k, uint64_t* flags, int64_t n_flags, uint32_t epoch, int32_t* status,
                            int64_t* split_ctas, void* stream) {
  if (split_ctas) *split_ctas = 0;
  if (!a || !w || !out || !flags || m < 0 || n <= 0 || k <= 0 || k % 8 != 0 || n % 16 != 0 ||
      epoch == 0)
    return MZC_ERR_INVALID;
  int dev = 0, sms = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
    return MZC_ERR_CUDA;
  if (n_flags < sms) return MZC_ERR_INVALID;
  if (m == 0) return MZC_OK;
  CUtensorMap ta;
  mzc::GemmWeight tw;
  if (!mzc::make_tmap_f16(&ta, a, static_cast<uint64_t>(m), static_cast<uint64_t>(k), 128) ||
      !mzc::make_gemm_weight(&tw, w, static_cast<uint64_t>(n), static_cast<uint64_t>(k)))
    return MZC_ERR_CUDA;
  mzc::GemmSplit split;
  split.flags = flags;
  split.n_flags = n_flags;
  split.epoch = epoch - 1;  // the launch takes the next one: `epoch`
  const cudaError_t e = mzc::launch_gemm(ta, tw, out, m, n, k, mzc::EPI_ADD_F32, status,
                                         static_cast<cudaStream_t>(stream), a, &split);
  if (split_ctas) *split_ctas = split.last_ctas;
  KCK(e);
}

mzc_status mzc_k_swiglu_pack(const uint16_t* gate, const uint16_t* up, int64_t f, int64_t d,
                             uint16_t* out_host) {
  if (!gate || !up || !out_host || f <= 0 || d <= 0 || f % mzc::kSwigluGroup != 0) return MZC_ERR_INVALID;
  const int64_t G = mzc::kSwigluGroup;
  for (int64_t j = 0; j < f; ++j) {
    const int64_t grp = j / G, r = j % G;
    std::memcpy(out_host + (grp * 2 * G + r) * d, gate + j * d, sizeof(uint16_t) * d);
    std::memcpy(out_host + (grp * 2 * G + G + r) * d, up + j * d, sizeof(uint16_t) * d);
  }
  return MZC_OK;
}

mzc_status mzc_k_rope_kv_write(const uint16_t* qkv, const int32_t* pos, int64_t n, int32_t hq,
                               int32_t hkv, int32_t hd, const float* cos_t, const float* sin_t,
                               const int32_t* block_table, int64_t n_logical, void* pool,
                               int64_t pool_blocks, int32_t kv_dtype, uint16_t* q_out,
                               int32_t* status, void* stream) {
  if (!qkv || !pos || !cos_t || !sin_t || !block_table || !pool || !q_out || n < 0) return MZC_ERR_INVALID;
  if ((hd != 64 && hd != 128) || hkv <= 0 || hq % hkv != 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_rope_kv_write(qkv, pos, n, hq, hkv, hd, cos_t, sin_t, block_table, n_logical,
                                pool, pool_blocks, kv_dtype, q_out, status, static_cast<cudaStream_t>(stream)));
}

int64_t mzc_k_attention_scratch_bytes(int64_t n, int32_t hq, int32_t hkv, int32_t hd, int64_t max_keys) {
  if (n <= 0 || hkv <= 0) return 0;
  int sp = 1, per = 0;
  mzc::attention_split(n, hq, hkv, hd, max_keys, sm_count(), &sp, &per);
  return mzc::attention_scratch_bytes(n, hq, hd, sp);
}

mzc_status mzc_k_attention(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                           int32_t hkv, int32_t hd, const int32_t* block_table, int64_t n_logical,
                           const void* pool, int64_t pool_blocks, int32_t kv_dtype, uint16_t* out,
                           int64_t max_keys, void* scratch, int64_t scratch_bytes, int32_t* status,
                           void* stream) {
  if (!q || !pos || !block_table || !pool || !out || n < 0 || max_keys <= 0) return MZC_ERR_INVALID;
  if ((hd != 64 && hd != 128) || hkv <= 0 || hq % hkv != 0) return MZC_ERR_INVALID;
  if (reinterpret_cast<uintptr_t>(pool) % 16 != 0) return MZC_ERR_INVALID;  // TMA and bulk copies
  KCK(mzc::launch_attention(q, pos, n, hq, hkv, hd, block_table, n_logical, pool, pool_blocks,
                            kv_dtype, out, scratch, scratch_bytes, max_keys, sm_count(), status,
                            static_cast<cudaStream_t>(stream)));
}

mzc_status mzc_k_attention_wait(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                                int32_t hkv, int32_t hd, const int32_t* block_table, int64_t n_logical,
                                const void* pool, int64_t pool_blocks, int32_t kv_dtype, uint16_t* out,
                                int64_t max_keys, void* scratch, int64_t scratch_bytes,
                                const int32_t* block_flags, int64_t flag_wait_cycles, int32_t* status,
                                void* stream) {
  if (!q || !pos || !block_table || !pool || !out || !block_flags || n < 0 || max_keys <= 0 ||
      flag_wait_cycles < 0)
    return MZC_ERR_INVALID;
  if ((hd != 64 && hd != 128) || hkv <= 0 || hq % hkv != 0) return MZC_ERR_INVALID;
  if (reinterpret_cast<uintptr_t>(pool) % 16 != 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_attention(q, pos, n, hq, hkv, hd, block_table, n_logical, pool, pool_blocks,
                            kv_dtype, out, scratch, scratch_bytes, max_keys, sm_count(), status,
                            static_cast<cudaStream_t>(stream), block_flags, flag_wait_cycles));
}

mzc_status mzc_k_attention_noalloc(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                                   int32_t hkv, int32_t hd, const int32_t* block_table,
                                   int64_t n_logical, const void* pool, int64_t pool_blocks,
                                   int32_t kv_dtype, uint16_t* out, int64_t max_keys,
                                   int32_t* status, void* stream) {
  if (!q || !pos || !block_table || !pool || !out || n < 0 || max_keys <= 0) {
    g_create_error = "mzc_k_attention_noalloc: null pointer or negative size";
    return MZC_ERR_INVALID;
  }
  if ((hd != 64 && hd != 128) || hkv <= 0 || hq % hkv != 0) {
    g_create_error = "mzc_k_attention_noalloc: unsupported head shape";
    return MZC_ERR_INVALID;
  }
  if (reinterpret_cast<uintptr_t>(pool) % 16 != 0) {
    g_create_error = "mzc_k_attention_noalloc: pool not 16-byte aligned";
    return MZC_ERR_INVALID;
  }
  const int64_t need = mzc::attention_noalloc_need(n, hq, hkv, hd, max_keys, sm_count());
  if (need > mzc::kAttnNoallocScratchBytes) {
    g_create_error = "mzc_k_attention_noalloc: this call's split-KV partials need " +
                     std::to_string(need) + " bytes, more than the library's fixed " +
                     std::to_string(mzc::kAttnNoallocScratchBytes) +
                     "-byte array; use mzc_k_attention with caller scratch";
    return MZC_ERR_RANGE;
  }
  cudaError_t e = mzc::launch_attention_noalloc(q, pos, n, hq, hkv, hd, block_table, n_logical,
                                                pool, pool_blocks, kv_dtype, out, max_keys,
                                                sm_count(), status, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) {
    g_create_error = std::string("mzc_k_attention_noalloc: ") + cudaGetErrorString(e);
    return MZC_ERR_CUDA;
  }
  return MZC_OK;
}

mzc_status mzc_k_wait_probe(int32_t arrive, int64_t limit_cycles, int32_t* status, int32_t* completed,
                            void* stream) {
  if (!status || !completed || limit_cycles <= 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_wait_probe(arrive, limit_cycles, status, completed, static_cast<cudaStream_t>(stream)));
}

int64_t mzc_q8_block_bytes(int32_t hkv, int32_t hd) {
  if (hkv <= 0 || hd <= 0 || hd % 64 != 0) return 0;
  return mzc::q8_block_bytes(2LL * hkv * 16 * hd);
}

mzc_status mzc_k_q8_encode(const void* pool, const int32_t* phys, int64_t n, int32_t hkv, int32_t hd,
                           void* out, void* stream) {
  if (!pool || !phys || !out || n < 0 || hkv <= 0 || hd <= 0 || hd % 64 != 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_q8_encode(pool, phys, n, 2LL * hkv * 16 * hd, out, static_cast<cudaStream_t>(stream)));
}

mzc_status mzc_k_q8_decode(const void* in, int64_t n, int32_t hkv, int32_t hd, const int32_t* phys,
                           int64_t phys_begin, int32_t kv_dtype, void* pool, void* stream) {
  if (!in || !pool || n < 0 || hkv <= 0 || hd <= 0 || hd % 64 != 0 || phys_begin < 0 ||
      (kv_dtype != MZC_KV_BF16 && kv_dtype != MZC_KV_FP16))
    return MZC_ERR_INVALID;
  KCK(mzc::launch_q8_decode(in, n, 2LL * hkv * 16 * hd, phys, phys_begin, kv_dtype, pool,
                            static_cast<cudaStream_t>(stream)));
}

mzc_status mzc_k_lm_head(const float* x_row, const float* g, int32_t d, float eps,
                         const uint16_t* w, int64_t vocab, float* logits, void* stream) {
  if (!x_row || !g || !w || !logits || d % 8 != 0 || vocab <= 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_lm_head(x_row, g, d, eps, w, vocab, logits, sm_count(), static_cast<cudaStream_t>(stream)));
}

mzc_status mzc_k_embed(const int32_t* tokens, int64_t n, const uint16_t* embed, int32_t d,
                       int64_t vocab, float* x, int32_t* status, void* stream) {
  if (!tokens || !embed || !x || d % 8 != 0 || n < 0) return MZC_ERR_INVALID;
  KCK(mzc::launch_embed(tokens, n, embed, d, vocab, x, status, static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
