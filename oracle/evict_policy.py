"""Plain-Python statement of the paper's eviction policy (test infrastructure).

Algorithm 1 (Sec. 4.3, "Hybrid Swap Eviction Policy") decides, for each
release request, how many units each restore path takes, in four stages:

  KVonly  while more KV units remain than the threshold T, KV units go to
          both restore paths, in inverse proportion to their per-unit times
          (the faster path takes more), so both finish together;
  KVandW  then, for every weight layer dropped, floor(t_W / t_KV') KV units go
          to the path that handles KV only;
  Wonly   once the KV units are gone, the remaining weight layers;
  CompKV  nothing left on the device: the paper moves compressed KV from
          memory to storage, which frees no device memory here.

with T = N_W_total * floor(t_W / t_KV'), the KV units that keep the KV-only
path busy while every weight layer is reloaded.  evict(size) (Sec. 5) frees
memory from the current state until `size` bytes are released.

Reading for one GB300 (the paper's paths are decompression and storage read;
here they are recompute and the host link):
  - weights can only come back over the link (t_W = one layer's bytes over
    the link); KV units can take either path: the link (COPY, t_copy) or
    recompute (DROP, t_rec), so recompute is the KV-only path;
  - a KV unit is one 16-token block of every layer (recompute regenerates a
    row's K/V in all layers at once), so T counts such units;
  - KVonly splits by balance: a unit goes to recompute only if the
    recompute path's total time with it stays strictly below the link
    path's total time with it (ties go to the link), which gives the inverse
    proportion over a run of units;
  - a stage step that frees more than asked is kept whole (the paper evicts
    slightly more than asked, Sec. 6.2).

Parity status: pinned by tests/test_oracle_evict_pins.py (hand-derived plans).
"""
from __future__ import annotations

KV_ONLY, KV_AND_W, W_ONLY, COMP_KV = 1, 2, 3, 4


def plan(t_copy_w, t_copy_kv, t_rec_kv, kv_total, w_total, kv_copy, kv_rec, w_evicted,
         kv_bytes, w_bytes, request_bytes):
    """Counts after evicting at least request_bytes from the given counts.
    Returns (kv_copy, kv_rec, w_evicted, freed_bytes, last_stage)."""
    q = int(t_copy_w // t_rec_kv) if t_rec_kv > 0 else 0   # KV units per weight layer
    T = w_total * q
    freed, stage = 0, 0
    while freed < request_bytes:
        n_kv = kv_total - kv_copy - kv_rec
        n_w = w_total - w_evicted
        if n_kv > T:
            stage = KV_ONLY
            rec_time = (kv_rec + 1) * t_rec_kv
            link_time = (kv_copy + 1) * t_copy_kv + w_evicted * t_copy_w
            if rec_time < link_time:
                kv_rec += 1
            else:
                kv_copy += 1
            freed += kv_bytes
        elif n_kv > 0 and n_w > 0:
            stage = KV_AND_W
            w_evicted += 1
            take = min(q, n_kv)
            kv_rec += take
            freed += w_bytes + take * kv_bytes
        elif n_w > 0:
            stage = W_ONLY
            w_evicted += 1
            freed += w_bytes
        else:
            stage = COMP_KV
            break
    return kv_copy, kv_rec, w_evicted, freed, stage


def layout(n_ctx, n_layers, kv_copy, kv_rec, w_evicted):
    """Where the counts sit in the context (backward-out: rearmost first): the
    recomputed units are the last kv_rec blocks of every layer, the copied
    ones the kv_copy blocks before them, the evicted weights the last
    w_evicted layers.  Returns ((copy_block_begin, copy_block_end),
    (drop_token_begin, drop_token_end), (weight_layer_begin, n_layers))."""
    nb = -(-n_ctx // 16)
    d0 = nb - kv_rec
    c0 = d0 - kv_copy
    drop = (d0 * 16, n_ctx) if kv_rec > 0 else None
    return (c0, d0), drop, (n_layers - w_evicted, n_layers)
