// Host bookkeeping of the evictable LLM memory state: per-layer KV block
// tables (logical block -> physical block), residency of every (layer,
// block), the physical-block and pinned-store allocators, the dropped range
// awaiting recompute, and the forward-in restore planner.
//
// The paper partitions each layer's KV into fixed-size chunks addressed by an
// array of chunk pointers (Sec. 4.2) and evicts/restores them one unit at a
// time (Sec. 4.3, 4.4).  Here a chunk is a 16-token block; eviction either
// swaps a block to the pinned host store (restored by copy) or drops it
// (restored by recompute).  No CUDA call is made in this file.
#pragma once

#include <cstdint>
#include <map>
#include <string>
#include <vector>

#include "mzc.h"

namespace mzc {

// Free-range allocator over [0, capacity) (physical blocks or store bytes).
class RangeAlloc {
 public:
  void reset(int64_t capacity);
  int64_t free_total() const { return free_total_; }
  // One contiguous range of n at the lowest address that fits; -1 if none.
  int64_t alloc_contig(int64_t n);
  // n units as few ranges as possible: one contiguous range if one fits,
  // otherwise the lowest-addressed free ranges.  Empty if free_total < n.
  std::vector<std::pair<int64_t, int64_t>> alloc_runs(int64_t n);
  void release(int64_t start, int64_t n);
  // The longest free range: its length, and its start in *start (0 if none).
  int64_t largest_free(int64_t* start) const;

 private:
  std::map<int64_t, int64_t> free_;  // start -> length
  int64_t free_total_ = 0;
  int64_t capacity_ = 0;
};

struct BlockEntry {
  uint8_t st = MZC_EMPTY;
  int32_t phys = -1;
  int32_t region = -1;  // pinned-store region while SWAPPED / INFLIGHT
  int32_t idx = -1;     // slot within that region
};

struct Region {
  int32_t layer = 0;
  int64_t host_off = 0;
  int32_t n_slots = 0;
  int32_t live = 0;  // slots still holding a swapped or in-flight block
};

// One layer's part of a COPY eviction: which physical blocks to move (in
// slot order) to which pinned-store offset.
struct EvictMove {
  int32_t layer;
  int64_t host_off;
  std::vector<int32_t> phys;
};

// What a prefill has to compute, decided before any kernel runs.
struct PrefillPlan {
  int64_t rec_begin = 0, rec_end = 0;        // recompute positions [rec_begin, rec_end)
  int64_t prompt_begin = 0, prompt_end = 0;  // new positions
  // per layer: does any block the rows read arrive by copy in this restore?
  std::vector<uint8_t> kv_wait_prompt;   // blocks < prompt_end in flight
  std::vector<uint8_t> kv_wait_rec;      // blocks < rec_end in flight
  std::vector<uint8_t> kv_wait_write;    // a block the rows write into is in flight
  std::vector<uint8_t> w_wait;           // layer weights in flight
};

class State {
 public:
  // slot_bytes: pinned-store bytes per swapped block (0 = block_bytes, the
  // block as stored; less when the swap codec compresses it)
  mzc_status init(const mzc_model_shape& s, int64_t pool_blocks, int64_t host_store_bytes,
                  int64_t slot_bytes = 0);

  const mzc_model_shape& shape() const { return shape_; }
  int64_t n_ctx() const { return n_ctx_; }
  int64_t nblk_max() const { return nblk_max_; }
  int64_t block_bytes() const { return block_bytes_; }
  int64_t slot_bytes() const { return slot_bytes_; }
  int64_t pool_blocks() const { return pool_blocks_; }
  int64_t host_store_bytes() const { return host_bytes_; }
  const std::string& error() const { return err_; }

  BlockEntry& at(int32_t l, int64_t b) { return tab_[(size_t)l * nblk_max_ + b]; }
  const BlockEntry& at(int32_t l, int64_t b) const { return tab_[(size_t)l * nblk_max_ + b]; }
  const Region& region(int32_t r) const { return regions_[r]; }

  // Eviction. COPY fills `moves` (the caller copies those blocks out before
  // anything else allocates); DROP frees.  Validates everything first: on an
  // error nothing changes.
  mzc_status evict_range(int32_t l0, int32_t l1, int64_t t0, int64_t t1, int32_t mode,
                         std::vector<EvictMove>* moves);
  mzc_status evict_blocks(const int32_t* layer, const int64_t* blk, int64_t n, int32_t mode,
                          std::vector<EvictMove>* moves);
  mzc_status evict_weights(int32_t l0, int32_t l1);
  mzc_status recompute_tail(int64_t p, int64_t n);

  bool has_drop() const { return drop_t0_ >= 0; }
  int64_t drop_begin() const { return drop_t0_; }
  int64_t drop_end() const { return drop_t1_; }
  bool recompute_pending() const { return rec_pending_; }

  // Forward-in restore plan of every swapped block and weight unit; swapped
  // blocks become INFLIGHT with their destination physical block assigned.
  mzc_status plan_restore(std::vector<mzc_copy_run>* runs, std::vector<int32_t>* weight_layers);
  // The same plan a layer at a time, so that a caller can issue layer l's
  // copies before it plans layer l + 1: begin_restore validates the whole
  // restore (the pool holds every swapped block) and marks it in flight when
  // there is anything to restore (*any); then plan_restore_layer(l) for l = 0,
  // 1, ... appends layer l's runs and sets *weight when its weights come back.
  mzc_status begin_restore(bool* any);
  void plan_restore_layer(int32_t l, std::vector<mzc_copy_run>* runs, bool* weight);
  bool restore_in_flight() const { return inflight_; }

  // Validates a prefill of n_prompt new tokens and allocates the blocks its
  // rows write (the pending recompute range and the new positions).
  mzc_status prepare_prefill(int64_t n_prompt, int64_t max_rows, PrefillPlan* plan);
  // After the prefill (or a sync) completed on the device: in-flight and
  // recomputed blocks become RESIDENT, the context grows by the prompt.
  void complete(int64_t n_prompt);
  // The restore's part of complete(): in-flight blocks and weights become
  // RESIDENT and their host slots are released (no-op without a restore).
  // The runtime calls it once every copy of the restore has been enqueued
  // ahead of the work that waits for it, while the device still runs.
  void complete_restore();
  // Undo prepare_prefill's allocations when the launch failed.
  void abort_prefill(const PrefillPlan& plan);

  mzc_status truncate(int64_t n_ctx);

  int32_t weight_state(int32_t l) const { return w_state_[l]; }
  // The evicted state as the eviction policy leaves it (backward-out): the
  // last kv_rec blocks of every layer DROPPED, the kv_copy blocks before them
  // SWAPPED in every layer, everything before RESIDENT, and the weights of
  // the last w_evicted layers swapped.  MZC_ERR_STATE for any other shape, or
  // while a restore or recompute is pending.
  mzc_status evicted_layout(int64_t* kv_copy, int64_t* kv_rec, int32_t* w_evicted) const;
  // Longest run of free physical blocks (holds no live KV): length, start.
  int64_t largest_free_pool_run(int64_t* start) const { return pool_.largest_free(start); }
  void counts(mzc_stats_t* out) const;
  // Block table rows [L][nblk_max] (phys or -1) for the device.  With
  // host_slots, a SWAPPED block's entry is -2 - (its slot in the pinned store,
  // in units of slot_bytes), for kernels that read it in place.
  void block_table(std::vector<int32_t>* out, bool host_slots = false) const;
  // the same table written to out[0 .. n_layers * nblk_max) (e.g. a pinned staging buffer)
  void block_table_into(int32_t* out, bool host_slots = false) const;
  int64_t table_entries() const { return static_cast<int64_t>(tab_.size()); }
  // Whether a prefill may read SWAPPED blocks in place (no restore issued).
  void set_read_swapped(bool on) { read_swapped_ = on; }
  int64_t host_slots() const { return host_bytes_ / slot_bytes_; }

 private:
  mzc_status fail(mzc_status s, const std::string& msg) {
    err_ = msg;
    return s;
  }
  void drop_region_slot(int32_t r);

  mzc_model_shape shape_{};
  int64_t nblk_max_ = 0, block_bytes_ = 0, slot_bytes_ = 0, pool_blocks_ = 0, host_bytes_ = 0;
  int64_t n_ctx_ = 0;
  std::vector<BlockEntry> tab_;
  std::vector<Region> regions_;
  std::vector<uint8_t> w_state_;
  RangeAlloc pool_, host_;
  int64_t drop_t0_ = -1, drop_t1_ = -1;
  bool rec_pending_ = false;
  bool inflight_ = false;
  bool read_swapped_ = false;
  // false only once a scan found no SWAPPED block since the last eviction to
  // host: the per-step scans for swapped blocks are skipped while it is false
  bool maybe_swapped_ = false;
  std::string err_;
};

int64_t ceil_div(int64_t a, int64_t b);

// Algorithm 1's stages over the counts in *p (in/out) until at least `bytes`
// are freed or nothing is left; returns the last stage taken (MZC_STAGE_*)
// and the bytes freed in *freed.  Pure arithmetic.
int32_t plan_evict_size(mzc_evict_plan* p, int64_t bytes, int64_t* freed);

// The evictions that take a context of n_ctx positions from counts (c0, r0,
// w0) to plan's counts, in this order: COPY of token range [copy_t0,
// copy_t1) in every layer (blocks that were resident), DROP of [drop_t0,
// drop_t1) in every layer (resident or swapped blocks, adjacent to the
// dropped tail), weights of layers [w0, w1).  Empty ranges have t1 <= t0.
struct EvictSizeSteps {
  int64_t copy_t0 = 0, copy_t1 = 0, drop_t0 = 0, drop_t1 = 0;
  int32_t w0 = 0, w1 = 0;
};
void evict_size_steps(int64_t n_ctx, int32_t n_layers, int64_t c0, int64_t r0, int32_t w0,
                      const mzc_evict_plan& p, EvictSizeSteps* out);

}  // namespace mzc
