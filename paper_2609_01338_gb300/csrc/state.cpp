// Host bookkeeping of the evictable LLM memory state (see state.hpp).
#include "state.hpp"

#include <algorithm>
#include <cmath>
#include <cstring>

namespace mzc {

int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }

// ---- RangeAlloc ---------------------------------------------------------

void RangeAlloc::reset(int64_t capacity) {
  free_.clear();
  capacity_ = capacity;
  free_total_ = capacity;
  if (capacity > 0) free_[0] = capacity;
}

int64_t RangeAlloc::alloc_contig(int64_t n) {
  if (n <= 0) return -1;
  for (auto it = free_.begin(); it != free_.end(); ++it) {
    if (it->second >= n) {
      int64_t start = it->first, len = it->second;
      free_.erase(it);
      if (len > n) free_[start + n] = len - n;
      free_total_ -= n;
      return start;
    }
  }
  return -1;
}

std::vector<std::pair<int64_t, int64_t>> RangeAlloc::alloc_runs(int64_t n) {
  std::vector<std::pair<int64_t, int64_t>> out;
  if (n <= 0 || free_total_ < n) return out;
  int64_t s = alloc_contig(n);
  if (s >= 0) {
    out.emplace_back(s, n);
    return out;
  }
  int64_t need = n;
  while (need > 0) {
    auto it = free_.begin();
    int64_t start = it->first, len = it->second;
    int64_t take = std::min(len, need);
    free_.erase(it);
    if (len > take) free_[start + take] = len - take;
    free_total_ -= take;
    out.emplace_back(start, take);
    need -= take;
  }
  return out;
}

int64_t RangeAlloc::largest_free(int64_t* start) const {
  int64_t best = 0, at = 0;
  for (const auto& kv : free_)
    if (kv.second > best) {
      best = kv.second;
      at = kv.first;
    }
  if (start) *start = at;
  return best;
}

void RangeAlloc::release(int64_t start, int64_t n) {
  if (n <= 0) return;
  free_total_ += n;
  auto next = free_.lower_bound(start);
  if (next != free_.begin()) {
    auto prev = std::prev(next);
    if (prev->first + prev->second == start) {
      start = prev->first;
      n += prev->second;
      free_.erase(prev);
    }
  }
  next = free_.lower_bound(start);
  if (next != free_.end() && start + n == next->first) {
    n += next->second;
    free_.erase(next);
  }
  free_[start] = n;
}

// ---- State --------------------------------------------------------------

mzc_status State::init(const mzc_model_shape& s, int64_t pool_blocks, int64_t host_store_bytes,
                       int64_t slot_bytes) {
  if (s.n_layers <= 0 || s.d_model <= 0 || s.n_q_heads <= 0 || s.n_kv_heads <= 0 ||
      s.head_dim <= 0 || s.ffn_dim <= 0 || s.vocab <= 0 || s.max_ctx <= 0)
    return fail(MZC_ERR_INVALID, "shape fields must be positive");
  if (s.block_tokens != 16) return fail(MZC_ERR_INVALID, "block_tokens must be 16");
  if (s.n_q_heads % s.n_kv_heads != 0)
    return fail(MZC_ERR_INVALID, "n_q_heads must be a multiple of n_kv_heads");
  if (s.kv_dtype != MZC_KV_BF16 && s.kv_dtype != MZC_KV_FP16)
    return fail(MZC_ERR_INVALID, "kv_dtype must be MZC_KV_BF16 or MZC_KV_FP16");
  shape_ = s;
  nblk_max_ = ceil_div(s.max_ctx, 16);
  block_bytes_ = 2LL * s.n_kv_heads * 16 * s.head_dim * 2;
  slot_bytes_ = slot_bytes > 0 ? slot_bytes : block_bytes_;
  pool_blocks_ = pool_blocks > 0 ? pool_blocks : 2LL * s.n_layers * nblk_max_;
  if (pool_blocks_ >= (1LL << 31)) return fail(MZC_ERR_INVALID, "pool_blocks too large");
  host_bytes_ = host_store_bytes > 0 ? host_store_bytes : (int64_t)s.n_layers * nblk_max_ * slot_bytes_;
  tab_.assign((size_t)s.n_layers * nblk_max_, BlockEntry{});
  regions_.clear();
  w_state_.assign(s.n_layers, MZC_RESIDENT);
  pool_.reset(pool_blocks_);
  host_.reset(host_bytes_);
  n_ctx_ = 0;
  drop_t0_ = drop_t1_ = -1;
  rec_pending_ = inflight_ = false;
  return MZC_OK;
}

void State::drop_region_slot(int32_t r) {
  Region& R = regions_[r];
  if (--R.live == 0) {
    host_.release(R.host_off, (int64_t)R.n_slots * slot_bytes_);
    R.n_slots = 0;
  }
}

mzc_status State::evict_range(int32_t l0, int32_t l1, int64_t t0, int64_t t1, int32_t mode,
                              std::vector<EvictMove>* moves) {
  const int32_t L = shape_.n_layers;
  if (mode != MZC_COPY && mode != MZC_DROP) return fail(MZC_ERR_INVALID, "mode must be COPY or DROP");
  if (l0 < 0 || l1 > L || l0 >= l1) return fail(MZC_ERR_RANGE, "layer range out of bounds");
  if (t0 < 0 || t1 > n_ctx_ || t0 >= t1) return fail(MZC_ERR_RANGE, "token range outside the context");
  if (inflight_ || rec_pending_) return fail(MZC_ERR_STATE, "a restore or recompute is pending");
  const int64_t b0 = t0 / 16, b1 = ceil_div(t1, 16);
  // DROP may also take SWAPPED blocks (their host copies are discarded): the
  // eviction policy can move a unit from the copy path to the recompute path
  for (int32_t l = l0; l < l1; ++l)
    for (int64_t b = b0; b < b1; ++b) {
      const uint8_t st = at(l, b).st;
      if (st != MZC_RESIDENT && !(mode == MZC_DROP && st == MZC_SWAPPED))
        return fail(MZC_ERR_STATE, "block " + std::to_string(b) + " of layer " + std::to_string(l) +
                                       (mode == MZC_DROP ? " is neither resident nor swapped"
                                                         : " is not resident"));
    }
  if (mode == MZC_DROP) {
    if (l0 != 0 || l1 != L)
      return fail(MZC_ERR_INVALID, "DROP must cover every layer (recompute regenerates all layers)");
    const int64_t d0 = b0 * 16, d1 = std::min(b1 * 16, n_ctx_);
    if (has_drop() && !(d1 == drop_t0_ || d0 == drop_t1_))
      return fail(MZC_ERR_INVALID, "dropped positions must stay one contiguous range");
    for (int32_t l = 0; l < L; ++l)
      for (int64_t b = b0; b < b1; ++b) {
        BlockEntry& e = at(l, b);
        if (e.st == MZC_SWAPPED)
          drop_region_slot(e.region);
        else
          pool_.release(e.phys, 1);
        e = BlockEntry{};
        e.st = MZC_DROPPED;
      }
    if (has_drop()) {
      drop_t0_ = std::min(drop_t0_, d0);
      drop_t1_ = std::max(drop_t1_, d1);
    } else {
      drop_t0_ = d0;
      drop_t1_ = d1;
    }
    return MZC_OK;
  }
  // COPY: one packed region per layer, blocks in logical order.
  const int64_t per_layer = (b1 - b0) * slot_bytes_;
  std::vector<int64_t> offs;
  for (int32_t l = l0; l < l1; ++l) {
    int64_t off = host_.alloc_contig(per_layer);
    if (off < 0) {
      for (size_t i = 0; i < offs.size(); ++i) host_.release(offs[i], per_layer);
      return fail(MZC_ERR_OOM, "pinned swap store is full");
    }
    offs.push_back(off);
  }
  for (int32_t l = l0; l < l1; ++l) {
    Region R;
    R.layer = l;
    R.host_off = offs[l - l0];
    R.n_slots = (int32_t)(b1 - b0);
    R.live = R.n_slots;
    int32_t rid = (int32_t)regions_.size();
    regions_.push_back(R);
    EvictMove mv{l, R.host_off, {}};
    for (int64_t b = b0; b < b1; ++b) {
      BlockEntry& e = at(l, b);
      mv.phys.push_back(e.phys);
      pool_.release(e.phys, 1);
      e.st = MZC_SWAPPED;
      e.phys = -1;
      e.region = rid;
      e.idx = (int32_t)(b - b0);
      maybe_swapped_ = true;
    }
    if (moves) moves->push_back(std::move(mv));
  }
  return MZC_OK;
}

mzc_status State::evict_blocks(const int32_t* layer, const int64_t* blk, int64_t n, int32_t mode,
                               std::vector<EvictMove>* moves) {
  if (mode != MZC_COPY) return fail(MZC_ERR_INVALID, "scattered eviction supports COPY only");
  if (n < 0 || (n > 0 && (!layer || !blk))) return fail(MZC_ERR_INVALID, "null block list");
  if (inflight_ || rec_pending_) return fail(MZC_ERR_STATE, "a restore or recompute is pending");
  const int32_t L = shape_.n_layers;
  const int64_t nb = ceil_div(n_ctx_, 16);
  std::vector<std::vector<int64_t>> per(L);
  for (int64_t i = 0; i < n; ++i) {
    if (layer[i] < 0 || layer[i] >= L || blk[i] < 0 || blk[i] >= nb)
      return fail(MZC_ERR_RANGE, "block index outside the context");
    if (at(layer[i], blk[i]).st != MZC_RESIDENT)
      return fail(MZC_ERR_STATE, "block is not resident");
    per[layer[i]].push_back(blk[i]);
  }
  for (int32_t l = 0; l < L; ++l) {
    auto& v = per[l];
    std::sort(v.begin(), v.end());
    if (std::adjacent_find(v.begin(), v.end()) != v.end())
      return fail(MZC_ERR_INVALID, "duplicate block in the list");
  }
  std::vector<int64_t> offs(L, -1);
  for (int32_t l = 0; l < L; ++l) {
    if (per[l].empty()) continue;
    offs[l] = host_.alloc_contig((int64_t)per[l].size() * slot_bytes_);
    if (offs[l] < 0) {
      for (int32_t j = 0; j < l; ++j)
        if (offs[j] >= 0) host_.release(offs[j], (int64_t)per[j].size() * slot_bytes_);
      return fail(MZC_ERR_OOM, "pinned swap store is full");
    }
  }
  for (int32_t l = 0; l < L; ++l) {
    if (per[l].empty()) continue;
    Region R;
    R.layer = l;
    R.host_off = offs[l];
    R.n_slots = (int32_t)per[l].size();
    R.live = R.n_slots;
    int32_t rid = (int32_t)regions_.size();
    regions_.push_back(R);
    EvictMove mv{l, R.host_off, {}};
    for (size_t i = 0; i < per[l].size(); ++i) {
      BlockEntry& e = at(l, per[l][i]);
      mv.phys.push_back(e.phys);
      pool_.release(e.phys, 1);
      e.st = MZC_SWAPPED;
      e.phys = -1;
      e.region = rid;
      e.idx = (int32_t)i;
      maybe_swapped_ = true;
    }
    if (moves) moves->push_back(std::move(mv));
  }
  return MZC_OK;
}

mzc_status State::evict_weights(int32_t l0, int32_t l1) {
  if (l0 < 0 || l1 > shape_.n_layers || l0 >= l1) return fail(MZC_ERR_RANGE, "layer range out of bounds");
  if (inflight_) return fail(MZC_ERR_STATE, "a restore is pending");
  for (int32_t l = l0; l < l1; ++l)
    if (w_state_[l] != MZC_RESIDENT) return fail(MZC_ERR_STATE, "layer weights are not resident");
  for (int32_t l = l0; l < l1; ++l) w_state_[l] = MZC_SWAPPED;
  return MZC_OK;
}

mzc_status State::recompute_tail(int64_t p, int64_t n) {
  if (!has_drop()) return fail(MZC_ERR_STATE, "nothing is dropped");
  if (p != drop_t0_ || n != drop_t1_ - drop_t0_)
    return fail(MZC_ERR_RANGE, "recompute range must equal the dropped range [" +
                                   std::to_string(drop_t0_) + ", " + std::to_string(drop_t1_) + ")");
  rec_pending_ = true;
  return MZC_OK;
}

mzc_status State::begin_restore(bool* any) {
  *any = false;
  if (inflight_) return fail(MZC_ERR_STATE, "a restore is already in flight");
  const int32_t L = shape_.n_layers;
  const int64_t nb = ceil_div(n_ctx_, 16);
  int64_t need = 0;
  if (maybe_swapped_) {
    for (int32_t l = 0; l < L; ++l)
      for (int64_t b = 0; b < nb; ++b) need += at(l, b).st == MZC_SWAPPED;
    maybe_swapped_ = need > 0;
  }
  if (need > pool_.free_total()) return fail(MZC_ERR_OOM, "KV pool cannot hold the restored blocks");
  bool w = false;
  for (int32_t l = 0; l < L; ++l) w = w || w_state_[l] == MZC_SWAPPED;
  *any = need > 0 || w;
  inflight_ = *any;
  return MZC_OK;
}

void State::plan_restore_layer(int32_t l, std::vector<mzc_copy_run>* runs, bool* weight) {
  const int64_t nb = ceil_div(n_ctx_, 16);
  *weight = false;
  if (w_state_[l] == MZC_SWAPPED) {
    w_state_[l] = MZC_INFLIGHT;
    *weight = true;
  }
  // swapped blocks of layer l grouped by region, slot order
  std::map<int32_t, std::vector<int64_t>> by_region;
  for (int64_t b = 0; b < nb; ++b)
    if (at(l, b).st == MZC_SWAPPED) by_region[at(l, b).region].push_back(b);
  for (auto& kv : by_region) {
    const Region& R = regions_[kv.first];
    auto& blocks = kv.second;  // ascending logical index == ascending slot
    auto ranges = pool_.alloc_runs((int64_t)blocks.size());
    size_t bi = 0;
    for (auto& rg : ranges) {
      for (int64_t j = 0; j < rg.second; ++j, ++bi) {
        BlockEntry& e = at(l, blocks[bi]);
        e.st = MZC_INFLIGHT;
        e.phys = (int32_t)(rg.first + j);
        int64_t off = R.host_off + (int64_t)e.idx * slot_bytes_;
        // extend the previous run when host and device are both contiguous
        if (runs && !runs->empty()) {
          mzc_copy_run& pr = runs->back();
          if (pr.layer == l && pr.phys_begin + pr.n_blocks == e.phys &&
              pr.host_off + (int64_t)pr.n_blocks * slot_bytes_ == off) {
            pr.n_blocks += 1;
            continue;
          }
        }
        if (runs) runs->push_back(mzc_copy_run{l, 1, off, (int64_t)e.phys});
      }
    }
  }
}

mzc_status State::plan_restore(std::vector<mzc_copy_run>* runs, std::vector<int32_t>* weight_layers) {
  bool any = false;
  mzc_status s = begin_restore(&any);
  if (s != MZC_OK) return s;
  if (runs) runs->clear();
  if (weight_layers) weight_layers->clear();
  for (int32_t l = 0; any && l < shape_.n_layers; ++l) {  // forward-in: earliest layer first
    bool w = false;
    plan_restore_layer(l, runs, &w);
    if (w && weight_layers) weight_layers->push_back(l);
  }
  return MZC_OK;
}

mzc_status State::prepare_prefill(int64_t n_prompt, int64_t max_rows, PrefillPlan* plan) {
  const int32_t L = shape_.n_layers;
  if (n_prompt < 0) return fail(MZC_ERR_INVALID, "negative token count");
  if (n_ctx_ + n_prompt > shape_.max_ctx) return fail(MZC_ERR_RANGE, "context would exceed max_ctx");
  if (has_drop() && !rec_pending_)
    return fail(MZC_ERR_STATE, "dropped blocks without a pending recompute");
  const int64_t nb = ceil_div(n_ctx_, 16);
  // a block the new rows write into: the context's last block when it is partial
  const int64_t write_blk = (n_ctx_ % 16 && n_prompt > 0) ? n_ctx_ / 16 : -1;
  for (int32_t l = 0; l < L; ++l) {
    if (w_state_[l] == MZC_SWAPPED) return fail(MZC_ERR_STATE, "layer weights swapped, no restore in flight");
    for (int64_t b = 0; maybe_swapped_ && b < nb; ++b) {
      if (at(l, b).st != MZC_SWAPPED) continue;
      if (!read_swapped_) return fail(MZC_ERR_STATE, "swapped blocks without a restore in flight");
      if (b == write_blk)
        return fail(MZC_ERR_STATE, "the block the new rows write into is swapped: restore it first");
    }
  }
  PrefillPlan P;
  P.rec_begin = rec_pending_ ? drop_t0_ : 0;
  P.rec_end = rec_pending_ ? drop_t1_ : 0;
  P.prompt_begin = n_ctx_;
  P.prompt_end = n_ctx_ + n_prompt;
  (void)max_rows;  // row sets larger than the activation buffers run in chunks
  // blocks to allocate per layer: dropped [db0, db1) and new [nb0, nb1)
  const int64_t db0 = P.rec_begin / 16, db1 = ceil_div(P.rec_end, 16);
  const int64_t nb0 = ceil_div(n_ctx_, 16), nb1 = ceil_div(n_ctx_ + n_prompt, 16);
  const int64_t per_layer = (db1 - db0) + (nb1 - nb0);
  if (per_layer * L > pool_.free_total()) return fail(MZC_ERR_OOM, "KV pool is full");
  for (int32_t l = 0; l < L; ++l) {
    auto ranges = pool_.alloc_runs(per_layer);
    std::vector<int32_t> ids;
    for (auto& rg : ranges)
      for (int64_t j = 0; j < rg.second; ++j) ids.push_back((int32_t)(rg.first + j));
    size_t k = 0;
    for (int64_t b = db0; b < db1; ++b) at(l, b).phys = ids[k++];  // stays DROPPED until complete()
    for (int64_t b = nb0; b < nb1; ++b) {
      BlockEntry& e = at(l, b);
      e = BlockEntry{};
      e.st = MZC_EMPTY;  // becomes RESIDENT in complete()
      e.phys = ids[k++];
    }
  }
  P.kv_wait_prompt.assign(L, 0);
  P.kv_wait_rec.assign(L, 0);
  P.kv_wait_write.assign(L, 0);
  P.w_wait.assign(L, 0);
  const int64_t last_partial = (n_ctx_ % 16) ? n_ctx_ / 16 : -1;
  for (int32_t l = 0; l < L; ++l) {
    P.w_wait[l] = w_state_[l] == MZC_INFLIGHT;
    // blocks are INFLIGHT only while a restore is
    for (int64_t b = 0; inflight_ && b < nb; ++b) {
      if (at(l, b).st != MZC_INFLIGHT) continue;
      P.kv_wait_prompt[l] = 1;
      if (b * 16 < P.rec_end) P.kv_wait_rec[l] = 1;
      if (b == last_partial && n_prompt > 0) P.kv_wait_write[l] = 1;
    }
  }
  *plan = std::move(P);
  return MZC_OK;
}

void State::abort_prefill(const PrefillPlan& P) {
  const int64_t db0 = P.rec_begin / 16, db1 = ceil_div(P.rec_end, 16);
  const int64_t nb0 = ceil_div(P.prompt_begin, 16), nb1 = ceil_div(P.prompt_end, 16);
  for (int32_t l = 0; l < shape_.n_layers; ++l) {
    for (int64_t b = db0; b < db1; ++b) {
      BlockEntry& e = at(l, b);
      if (e.phys >= 0) pool_.release(e.phys, 1);
      e.phys = -1;
    }
    for (int64_t b = nb0; b < nb1; ++b) {
      BlockEntry& e = at(l, b);
      if (e.phys >= 0) pool_.release(e.phys, 1);
      e = BlockEntry{};
    }
  }
}

void State::complete_restore() {
  if (!inflight_) return;
  const int32_t L = shape_.n_layers;
  const int64_t nb = ceil_div(n_ctx_, 16);
  for (int32_t l = 0; l < L; ++l) {
    if (w_state_[l] == MZC_INFLIGHT) w_state_[l] = MZC_RESIDENT;
    for (int64_t b = 0; b < nb; ++b) {
      BlockEntry& e = at(l, b);
      if (e.st == MZC_INFLIGHT) {
        drop_region_slot(e.region);
        e.st = MZC_RESIDENT;
        e.region = e.idx = -1;
      }
    }
  }
  inflight_ = false;
}

void State::complete(int64_t n_prompt) {
  complete_restore();
  const int32_t L = shape_.n_layers;
  const int64_t nb_new = ceil_div(n_ctx_ + n_prompt, 16);
  // what changes now: the recomputed blocks (DROPPED, given physical blocks
  // by prepare_prefill) and the new blocks past the context
  const int64_t b_first = rec_pending_ ? std::min(drop_t0_ / 16, ceil_div(n_ctx_, 16)) : ceil_div(n_ctx_, 16);
  for (int32_t l = 0; l < L; ++l) {
    for (int64_t b = b_first; b < nb_new; ++b) {
      BlockEntry& e = at(l, b);
      if (e.st == MZC_DROPPED && rec_pending_) {
        e.st = MZC_RESIDENT;
      } else if (e.st == MZC_EMPTY && e.phys >= 0) {
        e.st = MZC_RESIDENT;
      }
    }
  }
  if (rec_pending_) {
    rec_pending_ = false;
    drop_t0_ = drop_t1_ = -1;
  }
  n_ctx_ += n_prompt;
}

mzc_status State::truncate(int64_t n) {
  if (n < 0 || n > n_ctx_) return fail(MZC_ERR_RANGE, "truncate beyond the context");
  if (inflight_ || rec_pending_) return fail(MZC_ERR_STATE, "a restore or recompute is pending");
  const int64_t keep = ceil_div(n, 16), nb = ceil_div(n_ctx_, 16);
  for (int32_t l = 0; l < shape_.n_layers; ++l)
    for (int64_t b = keep; b < nb; ++b) {
      BlockEntry& e = at(l, b);
      if (e.st == MZC_RESIDENT && e.phys >= 0) pool_.release(e.phys, 1);
      if (e.st == MZC_SWAPPED) drop_region_slot(e.region);
      e = BlockEntry{};
    }
  n_ctx_ = n;
  if (has_drop()) {
    drop_t1_ = std::min(drop_t1_, n);
    if (drop_t1_ <= drop_t0_) drop_t0_ = drop_t1_ = -1;
  }
  return MZC_OK;
}

void State::counts(mzc_stats_t* o) const {
  std::memset(o, 0, sizeof(*o));
  o->context_tokens = n_ctx_;
  const int64_t nb = ceil_div(n_ctx_, 16);
  for (int32_t l = 0; l < shape_.n_layers; ++l) {
    for (int64_t b = 0; b < nb; ++b) {
      uint8_t s = at(l, b).st;
      o->blocks_resident += s == MZC_RESIDENT;
      o->blocks_swapped += s == MZC_SWAPPED || s == MZC_INFLIGHT;
      o->blocks_dropped += s == MZC_DROPPED;
    }
    o->weights_evicted_layers += w_state_[l] != MZC_RESIDENT;
  }
  o->pool_free_blocks = pool_.free_total();
}

void State::block_table(std::vector<int32_t>* out, bool host_slots) const {
  out->resize(tab_.size());
  block_table_into(out->data(), host_slots);
}

void State::block_table_into(int32_t* out, bool host_slots) const {
  const size_t n = tab_.size();
  if (!host_slots || !maybe_swapped_) {
    for (size_t i = 0; i < n; ++i) out[i] = tab_[i].phys;
    return;
  }
  for (size_t i = 0; i < n; ++i) {
    const BlockEntry& e = tab_[i];
    if (e.st == MZC_SWAPPED) {
      const int64_t slot = (regions_[e.region].host_off + static_cast<int64_t>(e.idx) * slot_bytes_) / slot_bytes_;
      out[i] = static_cast<int32_t>(-2 - slot);
    } else {
      out[i] = e.phys;
    }
  }
}

// ---- eviction policy (Algorithm 1) -----------------------------------------

int32_t plan_evict_size(mzc_evict_plan* p, int64_t bytes, int64_t* freed) {
  const int64_t q = p->t_rec_kv > 0 ? static_cast<int64_t>(std::floor(p->t_copy_w / p->t_rec_kv)) : 0;
  const int64_t T = static_cast<int64_t>(p->w_total) * q;
  int64_t f = 0;
  int32_t stage = 0;
  while (f < bytes) {
    const int64_t n_kv = p->kv_total - p->kv_copy - p->kv_rec;
    const int64_t n_w = static_cast<int64_t>(p->w_total) - p->w_evicted;
    if (n_kv > T) {  // KVonly: the unit to the path that stays faster with it (ties: link)
      stage = MZC_STAGE_KV_ONLY;
      const double rec = static_cast<double>(p->kv_rec + 1) * p->t_rec_kv;
      const double link = static_cast<double>(p->kv_copy + 1) * p->t_copy_kv +
                          static_cast<double>(p->w_evicted) * p->t_copy_w;
      if (rec < link)
        ++p->kv_rec;
      else
        ++p->kv_copy;
      f += p->kv_bytes;
    } else if (n_kv > 0 && n_w > 0) {  // KVandW: a layer, and q units to recompute
      stage = MZC_STAGE_KV_AND_W;
      const int64_t take = std::min(q, n_kv);
      ++p->w_evicted;
      p->kv_rec += take;
      f += p->w_bytes + take * p->kv_bytes;
    } else if (n_w > 0) {  // Wonly
      stage = MZC_STAGE_W_ONLY;
      ++p->w_evicted;
      f += p->w_bytes;
    } else {  // CompKV: nothing left to free on the device
      stage = MZC_STAGE_COMP_KV;
      break;
    }
  }
  if (freed) *freed = f;
  return stage;
}

mzc_status State::evicted_layout(int64_t* kv_copy, int64_t* kv_rec, int32_t* w_evicted) const {
  if (inflight_ || rec_pending_) return MZC_ERR_STATE;
  const int32_t L = shape_.n_layers;
  const int64_t nb = ceil_div(n_ctx_, 16);
  auto column = [&](int64_t b) -> int {  // the state every layer shares, or -1
    const uint8_t s0 = at(0, b).st;
    for (int32_t l = 1; l < L; ++l)
      if (at(l, b).st != s0) return -1;
    return s0;
  };
  int64_t b = nb, rec = 0, copy = 0;
  while (b > 0 && column(b - 1) == MZC_DROPPED) --b, ++rec;
  while (b > 0 && column(b - 1) == MZC_SWAPPED) --b, ++copy;
  for (int64_t c = 0; c < b; ++c)
    if (column(c) != MZC_RESIDENT) return MZC_ERR_STATE;
  int32_t w = 0;
  while (w < L && w_state_[L - 1 - w] == MZC_SWAPPED) ++w;
  for (int32_t l = 0; l < L - w; ++l)
    if (w_state_[l] != MZC_RESIDENT) return MZC_ERR_STATE;
  *kv_copy = copy;
  *kv_rec = rec;
  *w_evicted = w;
  return MZC_OK;
}

void evict_size_steps(int64_t n_ctx, int32_t n_layers, int64_t c0, int64_t r0, int32_t w0,
                      const mzc_evict_plan& p, EvictSizeSteps* out) {
  const int64_t nb = ceil_div(n_ctx, 16);
  const int64_t e0 = nb - r0 - c0;          // first evicted block before
  const int64_t e1 = nb - p.kv_rec - p.kv_copy;  // ... after
  const int64_t d0 = nb - r0;               // first dropped block before
  const int64_t d1 = nb - p.kv_rec;         // ... after
  EvictSizeSteps s;
  // newly copied blocks: the resident ones in front of the old evicted range,
  // minus any the new dropped range takes directly
  const int64_t cb1 = std::min(e0, d1);
  if (cb1 > e1) {
    s.copy_t0 = e1 * 16;
    s.copy_t1 = std::min(cb1 * 16, n_ctx);
  }
  if (d0 > d1) {
    s.drop_t0 = d1 * 16;
    s.drop_t1 = std::min(d0 * 16, n_ctx);
  }
  s.w0 = n_layers - p.w_evicted;
  s.w1 = n_layers - w0;
  *out = s;
}

}  // namespace mzc
