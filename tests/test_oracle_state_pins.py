"""Pins of the oracle's residency state machine (oracle/state_model.py).

Every expected value below is worked out by hand from the eviction rules the
C ABI states, not taken from the library or from the model itself:

  - token ranges round outward to whole 16-token blocks (the paper evicts at
    chunk granularity and takes slightly more than asked, Sec. 4.2 / 6.2);
  - COPY swaps RESIDENT blocks to the host store; a restore moves every
    SWAPPED block to INFLIGHT; a completed prefill makes INFLIGHT blocks
    RESIDENT again (Sec. 4.4 forward-in restore);
  - DROP frees blocks for recompute; it must cover every layer and the
    dropped positions must stay one contiguous range (recompute regenerates a
    row's K/V in every layer at once), else INVALID;
  - a block that is not RESIDENT cannot be evicted again (STATE);
  - a prefill over DROPPED blocks without a declared recompute is STATE; a
    recompute whose range is not the dropped range is RANGE;
  - truncation below a dropped range's end shortens that range.

Each test states the expected table literally, so that a model that rounds
inward, drops a layer subset, merges disjoint ranges, forgets to clear
INFLIGHT, or keeps a truncated range whole fails here."""
from oracle.state_model import (DROPPED, EMPTY, INFLIGHT, INVALID, OK, RANGE, RESIDENT, STATE,
                                SWAPPED, StateModel)


def _row(nblk, spans):
    """A literal table row: nblk entries, spans = [(b0, b1, state), ...] applied
    in order over an all-EMPTY row."""
    r = [EMPTY] * nblk
    for b0, b1, s in spans:
        for b in range(b0, b1):
            r[b] = s
    return r


def test_append_fills_blocks_and_bounds_the_context():
    m = StateModel(2, 100)                 # 7 blocks of 16 (the last holds 4 positions)
    assert m.nblk == 7
    assert m.append(33) == OK              # positions 0..32 -> blocks 0, 1, 2
    assert m.st == [_row(7, [(0, 3, RESIDENT)])] * 2
    assert m.append(67) == OK              # up to 100: blocks 3..6
    assert m.st == [_row(7, [(0, 7, RESIDENT)])] * 2
    assert m.append(1) == RANGE            # past max_ctx
    assert m.n_ctx == 100


def test_drop_rounds_outward_to_whole_blocks():
    # [200, 424): first block 200 // 16 = 12, last block (424 - 1) // 16 = 26
    m = StateModel(2, 1024)
    assert m.append(600) == OK             # blocks 0..37 resident (600 = 37*16 + 8)
    assert m.evict(0, 2, 200, 424, 1) == OK
    want = _row(64, [(0, 38, RESIDENT), (12, 27, DROPPED)])
    assert m.st == [want, want]
    assert m.drop == (192, 432)            # block-aligned dropped positions
    # the recompute must name exactly that range
    assert m.recompute_tail(200, 224) == RANGE
    assert m.recompute_tail(192, 240) == OK


def test_drop_of_the_ragged_last_block_stops_at_the_context_end():
    m = StateModel(1, 64)
    assert m.append(40) == OK              # blocks 0, 1, 2 (block 2 holds 32..39)
    assert m.evict(0, 1, 35, 36, 1) == OK  # rounds out to block 2 = positions [32, 40)
    assert m.drop == (32, 40)
    assert m.st == [[RESIDENT, RESIDENT, DROPPED, EMPTY]]


def test_copy_rounds_outward_and_covers_only_the_named_layers():
    m = StateModel(3, 256)
    assert m.append(256) == OK
    assert m.evict(1, 3, 17, 47, 0) == OK  # blocks 1..2 of layers 1 and 2
    assert m.st[0] == [RESIDENT] * 16
    assert m.st[1] == _row(16, [(0, 16, RESIDENT), (1, 3, SWAPPED)])
    assert m.st[2] == m.st[1]


def test_drop_of_a_layer_subset_is_invalid_and_changes_nothing():
    m = StateModel(3, 256)
    assert m.append(256) == OK
    assert m.evict(0, 2, 128, 256, 1) == INVALID
    assert m.evict(1, 3, 128, 256, 1) == INVALID
    assert m.st == [[RESIDENT] * 16] * 3
    assert m.drop is None


def test_a_second_drop_must_touch_the_first():
    m = StateModel(2, 512)
    assert m.append(512) == OK
    assert m.evict(0, 2, 256, 320, 1) == OK             # blocks 16..19
    # [400, 512) would leave two disjoint dropped ranges: refused, no change
    assert m.evict(0, 2, 400, 512, 1) == INVALID
    assert m.drop == (256, 320)
    assert m.st[0] == _row(32, [(0, 32, RESIDENT), (16, 20, DROPPED)])
    # adjacent after the range and adjacent before it: both merge
    assert m.evict(0, 2, 320, 352, 1) == OK
    assert m.evict(0, 2, 224, 256, 1) == OK
    assert m.drop == (224, 352)
    assert m.st[1] == _row(32, [(0, 32, RESIDENT), (14, 22, DROPPED)])


def test_double_eviction_is_a_state_error():
    m = StateModel(2, 256)
    assert m.append(256) == OK
    assert m.evict(0, 2, 0, 32, 0) == OK
    assert m.evict(0, 1, 16, 48, 0) == STATE   # block 1 is already SWAPPED
    assert m.evict_blocks([(1, 0)]) == STATE
    assert m.st[0] == _row(16, [(0, 16, RESIDENT), (0, 2, SWAPPED)])
    assert m.evict(0, 2, 240, 256, 1) == OK
    assert m.evict(0, 2, 240, 256, 1) == STATE  # dropped twice
    assert m.evict(0, 2, 240, 256, 0) == STATE  # a dropped block cannot be swapped


def test_drop_may_take_swapped_blocks():
    """The eviction policy can move a unit from the copy path to the recompute
    path: DROP over SWAPPED blocks discards their host copies."""
    m = StateModel(2, 256)
    assert m.append(256) == OK
    assert m.evict(0, 2, 128, 256, 0) == OK    # blocks 8..15 swapped
    assert m.evict(0, 2, 224, 256, 1) == OK    # blocks 14, 15: swapped -> dropped
    want = _row(16, [(0, 16, RESIDENT), (8, 14, SWAPPED), (14, 16, DROPPED)])
    assert m.st == [want, want]
    assert m.drop == (224, 256)
    # a range that is part resident, part swapped, adjacent to the drop
    assert m.evict(0, 2, 112, 224, 1) == OK    # blocks 7 (resident) .. 13 (swapped)
    want = _row(16, [(0, 16, RESIDENT), (7, 16, DROPPED)])
    assert m.st == [want, want]
    assert m.drop == (112, 256)
    assert m.restore() == OK and not m.inflight  # nothing left to copy back
    assert m.recompute_tail(112, 144) == OK


def test_prefill_over_dropped_blocks_needs_the_recompute():
    m = StateModel(2, 512)
    assert m.append(300) == OK
    assert m.evict(0, 2, 256, 300, 1) == OK
    assert m.append(8) == STATE                # dropped, nothing declared
    assert m.n_ctx == 300
    assert m.recompute_tail(256, 44) == OK
    assert m.append(8) == OK                   # recompute + 8 new positions
    assert m.st == [_row(32, [(0, 20, RESIDENT)])] * 2   # 308 positions -> blocks 0..19
    assert m.drop is None and not m.pending


def test_prefill_over_swapped_blocks_needs_the_restore():
    m = StateModel(1, 256)
    assert m.append(64) == OK                  # blocks 0..3
    assert m.evict(0, 1, 0, 16, 0) == OK
    assert m.append(1) == STATE                # SWAPPED and no restore issued
    assert m.restore() == OK
    assert m.st == [_row(16, [(0, 4, RESIDENT), (0, 1, INFLIGHT)])]
    assert m.restore() == STATE                # a restore is already in flight
    assert m.evict(0, 1, 16, 32, 0) == STATE   # no eviction while copies are in flight
    assert m.append(1) == OK                   # 65 positions: blocks 0..4, all resident
    assert m.st == [_row(16, [(0, 5, RESIDENT)])]


def test_recompute_range_must_equal_the_dropped_range():
    m = StateModel(2, 512)
    assert m.append(512) == OK
    assert m.recompute_tail(0, 16) == STATE    # nothing dropped
    assert m.evict(0, 2, 256, 512, 1) == OK
    assert m.recompute_tail(256, 128) == RANGE
    assert m.recompute_tail(240, 272) == RANGE
    assert m.recompute_tail(256, 256) == OK


def test_truncate_inside_a_dropped_range_shortens_it():
    m = StateModel(2, 512)
    assert m.append(512) == OK
    assert m.evict(0, 2, 256, 512, 1) == OK
    assert m.truncate(300) == OK               # blocks 19..31 leave the context
    assert m.drop == (256, 300)
    assert m.st[0] == _row(32, [(0, 16, RESIDENT), (16, 19, DROPPED)])
    assert m.recompute_tail(256, 256) == RANGE
    assert m.recompute_tail(256, 44) == OK
    # truncating below the whole dropped range clears it
    m2 = StateModel(1, 512)
    assert m2.append(512) == OK
    assert m2.evict(0, 1, 256, 512, 1) == OK
    assert m2.truncate(256) == OK
    assert m2.drop is None
    assert m2.st == [_row(32, [(0, 16, RESIDENT)])]
    assert m2.append(1) == OK                  # nothing left to recompute


def test_scattered_block_eviction_rules():
    m = StateModel(2, 64)
    assert m.append(48) == OK                  # blocks 0..2 of both layers
    assert m.evict_blocks([(0, 1), (1, 1), (0, 1)]) == INVALID   # duplicate pair
    assert m.evict_blocks([(1, 3)]) == RANGE   # block 3 is past the context
    assert m.evict_blocks([(2, 0)]) == RANGE   # no layer 2
    assert m.st == [_row(4, [(0, 3, RESIDENT)])] * 2
    assert m.evict_blocks([(0, 2), (1, 0)]) == OK
    assert m.st[0] == [RESIDENT, RESIDENT, SWAPPED, EMPTY]
    assert m.st[1] == [SWAPPED, RESIDENT, RESIDENT, EMPTY]


def test_eviction_range_checks():
    m = StateModel(2, 128)
    assert m.append(64) == OK
    assert m.evict(0, 2, 0, 65, 0) == RANGE    # past the context
    assert m.evict(0, 3, 0, 16, 0) == RANGE    # past the layers
    assert m.evict(1, 1, 0, 16, 0) == RANGE    # empty layer range
    assert m.evict(0, 2, 16, 16, 0) == RANGE   # empty token range
    assert m.evict(0, 2, 0, 16, 7) == INVALID  # unknown mode
    assert m.st == [_row(8, [(0, 4, RESIDENT)])] * 2
