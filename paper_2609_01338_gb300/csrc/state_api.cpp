// C ABI of the host bookkeeping (mzc_state_*): the same State the ctx uses,
// without any device.
#include <cstring>
#include <vector>

#include "mzc.h"
#include "state.hpp"

struct mzc_state {
  mzc::State st;
};

extern "C" {

mzc_status mzc_state_create(const mzc_model_shape* shape, int64_t pool_blocks,
                            int64_t host_store_bytes, mzc_state** out) {
  if (!shape || !out) return MZC_ERR_INVALID;
  *out = nullptr;
  mzc_state* s = new mzc_state();
  mzc_status r = s->st.init(*shape, pool_blocks, host_store_bytes);
  if (r != MZC_OK) {
    delete s;
    return r;
  }
  *out = s;
  return MZC_OK;
}

mzc_status mzc_state_destroy(mzc_state* st) {
  if (!st) return MZC_ERR_INVALID;
  delete st;
  return MZC_OK;
}

mzc_status mzc_state_append(mzc_state* st, int64_t n) {
  if (!st) return MZC_ERR_INVALID;
  mzc::PrefillPlan p;
  mzc_status r = st->st.prepare_prefill(n, INT64_MAX, &p);
  if (r != MZC_OK) return r;
  st->st.complete(n);
  return MZC_OK;
}

mzc_status mzc_state_evict(mzc_state* st, int32_t l0, int32_t l1, int64_t t0, int64_t t1,
                           int32_t mode) {
  if (!st) return MZC_ERR_INVALID;
  return st->st.evict_range(l0, l1, t0, t1, mode, nullptr);
}

mzc_status mzc_state_evict_blocks(mzc_state* st, const int32_t* layer, const int64_t* blk,
                                  int64_t n, int32_t mode) {
  if (!st) return MZC_ERR_INVALID;
  return st->st.evict_blocks(layer, blk, n, mode, nullptr);
}

mzc_status mzc_plan_evict_size(mzc_evict_plan* plan, int64_t bytes, int64_t* freed_out,
                               int32_t* stage_out) {
  if (!plan) return MZC_ERR_INVALID;
  const mzc_evict_plan& p = *plan;
  if (!(p.t_copy_w >= 0) || !(p.t_copy_kv >= 0) || !(p.t_rec_kv >= 0) || p.kv_total < 0 ||
      p.w_total < 0 || p.kv_copy < 0 || p.kv_rec < 0 || p.w_evicted < 0 ||
      p.kv_copy + p.kv_rec > p.kv_total || p.w_evicted > p.w_total || p.kv_bytes < 0 || p.w_bytes < 0)
    return MZC_ERR_INVALID;
  // a step that frees no bytes would never end the loop
  if (bytes > 0 && ((p.kv_total > p.kv_copy + p.kv_rec && p.kv_bytes <= 0) ||
                    (p.w_total > p.w_evicted && p.w_bytes <= 0)))
    return MZC_ERR_INVALID;
  int64_t freed = 0;
  const int32_t stage = mzc::plan_evict_size(plan, bytes, &freed);
  if (freed_out) *freed_out = freed;
  if (stage_out) *stage_out = stage;
  return MZC_OK;
}

mzc_status mzc_state_evict_size(mzc_state* st, const mzc_evict_plan* times, int64_t bytes,
                                int64_t* freed_out, int32_t* stage_out) {
  if (!st || !times) return MZC_ERR_INVALID;
  mzc::State& S = st->st;
  mzc_evict_plan p = *times;
  const int32_t L = S.shape().n_layers;
  p.kv_total = mzc::ceil_div(S.n_ctx(), 16);
  p.w_total = L;
  int64_t c0 = 0, r0 = 0;
  int32_t w0 = 0;
  mzc_status e = S.evicted_layout(&c0, &r0, &w0);
  if (e != MZC_OK) return e;
  p.kv_copy = c0;
  p.kv_rec = r0;
  p.w_evicted = w0;
  int64_t freed = 0;
  int32_t stage = 0;
  e = mzc_plan_evict_size(&p, bytes, &freed, &stage);
  if (e != MZC_OK) return e;
  mzc::EvictSizeSteps steps;
  mzc::evict_size_steps(S.n_ctx(), L, c0, r0, w0, p, &steps);
  if (steps.copy_t1 > steps.copy_t0) {
    e = S.evict_range(0, L, steps.copy_t0, steps.copy_t1, MZC_COPY, nullptr);
    if (e != MZC_OK) return e;
  }
  if (steps.drop_t1 > steps.drop_t0) {
    e = S.evict_range(0, L, steps.drop_t0, steps.drop_t1, MZC_DROP, nullptr);
    if (e != MZC_OK) return e;
  }
  if (steps.w1 > steps.w0) {
    e = S.evict_weights(steps.w0, steps.w1);
    if (e != MZC_OK) return e;
  }
  if (freed_out) *freed_out = freed;
  if (stage_out) *stage_out = stage;
  return MZC_OK;
}

mzc_status mzc_state_recompute_tail(mzc_state* st, int64_t p, int64_t n) {
  if (!st) return MZC_ERR_INVALID;
  return st->st.recompute_tail(p, n);
}

mzc_status mzc_state_plan_restore(mzc_state* st, mzc_copy_run* runs, int64_t cap, int64_t* n_runs) {
  if (!st || !n_runs || cap < 0 || (cap > 0 && !runs)) return MZC_ERR_INVALID;
  // plan on a copy first so that a too-small buffer changes nothing
  mzc::State trial = st->st;
  std::vector<mzc_copy_run> v;
  std::vector<int32_t> wl;
  mzc_status r = trial.plan_restore(&v, &wl);
  if (r != MZC_OK) return r;
  *n_runs = static_cast<int64_t>(v.size());
  if (static_cast<int64_t>(v.size()) > cap) return MZC_ERR_OOM;
  if (!v.empty()) std::memcpy(runs, v.data(), v.size() * sizeof(mzc_copy_run));
  st->st = trial;
  return MZC_OK;
}

mzc_status mzc_state_complete(mzc_state* st) {
  if (!st) return MZC_ERR_INVALID;
  if (st->st.recompute_pending()) return mzc_state_append(st, 0);
  st->st.complete(0);
  return MZC_OK;
}

mzc_status mzc_state_truncate(mzc_state* st, int64_t n_ctx) {
  if (!st) return MZC_ERR_INVALID;
  return st->st.truncate(n_ctx);
}

mzc_status mzc_state_query(mzc_state* st, int32_t layer, int64_t b, int32_t* state, int32_t* phys) {
  if (!st) return MZC_ERR_INVALID;
  if (layer < 0 || layer >= st->st.shape().n_layers || b < 0 || b >= st->st.nblk_max())
    return MZC_ERR_RANGE;
  const mzc::BlockEntry& e = st->st.at(layer, b);
  if (state) *state = e.st;
  if (phys) *phys = e.phys;
  return MZC_OK;
}

mzc_status mzc_state_counts(mzc_state* st, mzc_stats_t* out) {
  if (!st || !out) return MZC_ERR_INVALID;
  st->st.counts(out);
  return MZC_OK;
}

}  // extern "C"
