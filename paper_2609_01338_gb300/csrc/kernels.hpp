// Launchers of the prefill-path kernels (host side).  Each returns the
// cudaError_t of its launch; none synchronizes.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>
#include <utility>

namespace mzc {

// Programmatic dependent launch for the hot-path kernels (on unless the
// environment sets MZC_PDL=0 when the library loads): the next kernel of a
// stream is scheduled while the previous one finishes and waits in
// pdl_enter() for its results, hiding launch and CTA-scheduling latency.
bool pdl_enabled();

template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// The same with thread-block clusters of cluster_x CTAs along x.
template <typename... KArgs, typename... Args>
cudaError_t launch_k_cluster(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                             cudaStream_t st, unsigned cluster_x, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = cluster_x;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl_enabled() ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

enum GemmEpilogue { EPI_STORE_BF16 = 0, EPI_ADD_F32 = 1, EPI_SWIGLU_BF16 = 2, EPI_QKV_ROPE = 3 };

// EPI_QKV_ROPE (split-K GEMM only): the QKV projection's rows go straight to
// the rotary embedding and the KV-block write (as rope_kv_kernel, from the
// fp32 sums instead of fp16 outputs): q and k rotated (half-split pairs,
// fp32 tables), q to q_out [m][hq][hd] in fp16, K and V rounded to the KV
// precision into pool[table[pos / 16]] slot pos % 16 (K [hkv][16][hd], then V).
// Needs n = (hq + 2 hkv) hd a multiple of 128 and hd 64 or 128, so that a
// 128-column tile holds whole heads.
struct RopeKV {
  const int32_t* pos = nullptr;    // [m]
  const float* cos_t = nullptr;    // [positions][hd / 2]
  const float* sin_t = nullptr;
  const int32_t* table = nullptr;  // logical block -> physical block
  int64_t n_logical = 0;           // table entries: positions < n_logical * 16
  uint16_t* pool = nullptr;
  int64_t pool_blocks = 0;
  uint16_t* q_out = nullptr;
  int hq = 0, hkv = 0, hd = 0;
  int f16kv = 1;  // 0: K and V rounded to bf16 precision before the fp16 encoding
};

// Row group of the SwiGLU weight interleave: 64 gate rows, then the matching
// 64 up rows, repeated.  The fused epilogue needs both halves in one tile.
constexpr int kSwigluGroup = 64;

// A 2-D fp16 tensor map [rows][cols] (cols contiguous) with a box of
// 64 columns x box_rows rows and 128-byte swizzle (the UMMA K-major layout).
bool make_tmap_f16(CUtensorMap* map, const void* base, uint64_t rows, uint64_t cols,
                    uint32_t box_rows);

// A weight operand W [n][k] with one tensor map per tile width the GEMM may
// pick (box rows 64, 128 and 256).
struct GemmWeight {
  CUtensorMap box64, box128, box256;
  const uint16_t* ptr = nullptr;  // W itself, for the few-row GEMV
};
// RMSNorm folded into the projections of a short row set (RMSNorm(x) W^T =
// diag(rstd) ((x * g) W^T) for the decoder layer's pre-norms):
//   - producer, the split-K residual-add GEMM that finishes x (O or down):
//     besides x it writes h = fp16(x * g) and, per row r and 128-column tile
//     t of x, ss[r * nt + t] = the sum of x^2 over the tile's columns;
//   - consumer, the next projection (QKV or gate/up) with h as its A operand:
//     row r of its accumulator is scaled by
//     rstd_r = rsqrt((ss[r * nt + 0] + ... + ss[r * nt + nt - 1]) / d + eps),
//     summed in tile order, before its epilogue (fp16 store or SwiGLU).
struct RowNorm {
  const float* g = nullptr;  // producer: norm weights [d]
  uint16_t* h = nullptr;     // producer: fp16 x * g, [m][d]
  float* ss = nullptr;       // producer writes, consumer reads: [m][nt]
  int nt = 0;                // 128-column tiles of x (d / 128)
  float d = 0.0f, eps = 0.0f;
};

// Split-K GEMM over a thread-block cluster for m <= 256 (gemm_splitk.cu):
// launched (and *launched set) when n is a multiple of 128 and a cluster size
// of at least 2 fits the grid in one wave; otherwise nothing is launched.
// `rn`: as the producer (epilogue EPI_ADD_F32, rn->h set) or the consumer
// (EPI_STORE_BF16 / EPI_SWIGLU_BF16, rn->ss set) of a folded RMSNorm.
// `rk`: the rotary / KV-write targets of EPI_QKV_ROPE.
cudaError_t launch_gemm_splitk(const CUtensorMap& ta, const struct GemmWeight& w, void* out, int64_t m,
                               int64_t n, int64_t k, int epilogue, int num_sms, int32_t* status,
                               cudaStream_t st, bool* launched, const RowNorm* rn = nullptr,
                               const RopeKV* rk = nullptr);
// Whether launch_gemm_splitk launches for this shape (the same rule).
bool gemm_splitk_launches(int64_t m, int64_t n, int64_t k, int epilogue, int num_sms);
bool make_gemm_weight(GemmWeight* gw, const void* base, uint64_t n, uint64_t k);

// State for splitting the residual-add GEMM's last wave over k: a device
// array of n_flags uint64 (at least the number of SMs; any contents) and the
// epoch of the last split launch.  Launches that share it run in stream
// order; each split launch takes the next nonzero 32-bit epoch, so flag values
// left by earlier launches never match.
struct GemmSplit {
  uint64_t* flags = nullptr;
  int64_t n_flags = 0;
  uint32_t epoch = 0;
  int64_t last_ctas = 0;  // CTAs that shared the split tiles in the last launch (0: unsplit)
};
inline uint32_t next_split_epoch(GemmSplit* s) {
  if (++s->epoch == 0) s->epoch = 1;
  return s->epoch;
}

// C = A W^T; A map [>= m][k] with box rows 128.  The W map used is the one
// whose box matches the tile width gemm_box_n(m, n, epilogue) selects.  With
// `split`, the residual-add epilogue splits its last partial wave over k.
// With `rn` (a folded RMSNorm, m of kGemvMaxRows + 1 .. 256): the producer
// (EPI_ADD_F32) runs only as the split-K kernel (cudaErrorInvalidValue when
// gemm_splitk_launches says it would not); a consumer runs as the split-K
// kernel or the persistent kernel's row-scaled form.  For m = 1 with a_ptr,
// the GEMV's one-row form (launch_gemv); m of 2..4 with `rn` is refused.
uint32_t gemm_box_n(int64_t m, int64_t n, int epilogue);
cudaError_t launch_gemm(const CUtensorMap& ta, const GemmWeight& w, void* out, int64_t m,
                        int64_t n, int64_t k, int epilogue, int32_t* status, cudaStream_t st,
                        const uint16_t* a_ptr = nullptr, GemmSplit* split = nullptr,
                        const RowNorm* rn = nullptr);

// Few-row projections (decode steps; gemv.cu): A fp16 [m][k], W fp16 [n][k],
// same epilogues as the GEMM; launch_gemm takes this path for m <= kGemvMaxRows
// when it is given the activation pointer.  `rn`: the folded RMSNorm for one
// row (m = 1): the residual add writes h and one partial sum of squares per
// CTA (gemv_norm_tiles(n, k) of them, at most kGemvNormMax); the fp16-store or
// SwiGLU consumer sums rn->nt partials and scales its outputs by rstd.
constexpr int kGemvMaxRows = 4;
constexpr int kGemvNormMax = 2048;
int64_t gemv_norm_tiles(int64_t n, int64_t k);
cudaError_t launch_gemv(const uint16_t* a, const uint16_t* w, void* out, int64_t m, int64_t n,
                        int64_t k, int epilogue, int32_t* status, cudaStream_t st,
                        const RowNorm* rn = nullptr);

// 8-bit swap codec (codec.cu).  block_elems = 2 * hkv * 16 * hd.
int64_t q8_block_bytes(int64_t block_elems);
cudaError_t launch_q8_encode(const void* pool, const int32_t* phys, int64_t n_blocks,
                             int64_t block_elems, void* out, cudaStream_t st);
cudaError_t launch_q8_decode(const void* in, int64_t n_blocks, int64_t block_elems,
                             const int32_t* phys, int64_t phys_begin, int32_t kv_dtype, void* pool,
                             cudaStream_t st);

cudaError_t launch_wait_probe(int32_t arrive, int64_t limit_cycles, int32_t* status,
                              int32_t* completed, cudaStream_t st);

cudaError_t launch_embed(const int32_t* tokens, int64_t n, const uint16_t* embed, int32_t d,
                         int64_t vocab, float* x, int32_t* status, cudaStream_t st);
cudaError_t launch_rmsnorm(const float* x, const float* g, int64_t n, int32_t d, float eps,
                           uint16_t* y, cudaStream_t st, int32_t* status = nullptr);
cudaError_t launch_rope_kv_write(const uint16_t* qkv, const int32_t* pos, int64_t n, int32_t hq,
                                 int32_t hkv, int32_t hd, const float* cos_t, const float* sin_t,
                                 const int32_t* table, int64_t n_logical, void* pool,
                                 int64_t pool_blocks, int32_t kv_dtype, uint16_t* q_out,
                                 int32_t* status, cudaStream_t st);
// Split-KV plan: how many key splits a launch of n rows over at most
// max_keys keys uses, and the keys per split (a multiple of 64).
void attention_split(int64_t n, int32_t hq, int32_t hkv, int32_t hd, int64_t max_keys, int num_sms,
                     int* n_splits, int* keys_per_split);
int64_t attention_scratch_bytes(int64_t n, int32_t hq, int32_t hd, int n_splits);

// Decode attention (attention_decode.cu): at most kAttnDecodeMaxRows query rows
// per KV head (n tokens x hq/hkv heads; one decode token of a model with up to
// 4 query heads per KV head) take a CUDA-core kernel bound by the K/V read
// instead of the 128-row tensor tiles; same arguments, split-KV partials and
// combine as launch_attention, which dispatches to it.
constexpr int kAttnDecodeMaxRows = 4;
bool attention_decode_applies(int64_t n, int32_t hq, int32_t hkv, int32_t hd);
void attention_decode_split(int32_t hkv, int64_t max_keys, int num_sms, int* n_splits, int* keys_per_split);
cudaError_t launch_attention_decode(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq, int32_t hkv,
                                    int32_t hd, const int32_t* table, int64_t n_logical, const void* pool,
                                    int64_t pool_blocks, uint16_t* out, float* part_o, float* part_lse,
                                    int n_splits, int keys_per_split, int32_t* status,
                                    const int32_t* flags, long long flag_wait, const uint16_t* host_pool,
                                    int64_t host_blocks, cudaStream_t st);
// flags (may be null): int32 per physical block, non-zero once the block's
// data is in HBM; the kernels wait (bounded by flag_wait_cycles, 0 = the
// default limit) for the flag of every block they read before fetching it.
// host_pool (may be null): device-accessible base of pinned host memory
// holding host_blocks KV blocks in the pool's block layout; a block-table
// entry -2 - i names host block i, read in place with plain loads.
cudaError_t launch_attention(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                             int32_t hkv, int32_t hd, const int32_t* table, int64_t n_logical,
                             const void* pool, int64_t pool_blocks, int32_t kv_dtype,
                             uint16_t* out, void* scratch, int64_t scratch_bytes,
                             int64_t max_keys, int num_sms, int32_t* status, cudaStream_t st,
                             const int32_t* flags = nullptr, int64_t flag_wait_cycles = 0,
                             const void* host_pool = nullptr, int64_t host_blocks = 0);
// Attention whose split-KV partials use a fixed array inside the library
// (kAttnNoallocScratchBytes) instead of caller memory; no allocation.
constexpr int64_t kAttnNoallocScratchBytes = 8LL << 20;
int64_t attention_noalloc_need(int64_t n, int32_t hq, int32_t hkv, int32_t hd, int64_t max_keys,
                               int num_sms);
cudaError_t launch_attention_noalloc(const uint16_t* q, const int32_t* pos, int64_t n, int32_t hq,
                                     int32_t hkv, int32_t hd, const int32_t* table,
                                     int64_t n_logical, const void* pool, int64_t pool_blocks,
                                     int32_t kv_dtype, uint16_t* out, int64_t max_keys,
                                     int num_sms, int32_t* status, cudaStream_t st);
cudaError_t launch_lm_head(const float* x_row, const float* g, int32_t d, float eps,
                           const uint16_t* w, int64_t vocab, float* logits, int num_sms,
                           cudaStream_t st);
// Copies bytes (rounded up to 16) from src to dst with a kernel; src may be
// mapped pinned host memory (read by the SMs, not by a copy engine).
cudaError_t launch_copy16(const void* src, void* dst, int64_t bytes, cudaStream_t st);
// Copies blocks phys[i] (block_bytes each) of the pool to dst + i*block_bytes.
cudaError_t launch_gather_blocks(const void* pool, const int32_t* phys, int64_t n,
                                 int64_t block_bytes, void* dst, cudaStream_t st);
// Fills blocks phys[i] with the largest finite value of the KV type.
cudaError_t launch_poison_blocks(void* pool, const int32_t* phys, int64_t n, int64_t block_bytes,
                                 int32_t kv_dtype, cudaStream_t st);
// Poisons the contiguous physical blocks [phys_begin, phys_begin + n).
cudaError_t launch_poison_run(void* pool, int64_t phys_begin, int64_t n, int64_t block_bytes,
                              cudaStream_t st);

}  // namespace mzc
