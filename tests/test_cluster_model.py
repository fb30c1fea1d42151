"""Host-side model of the per-head cluster decode (restated from decode_cluster_kernel and
decode_cluster_size in dms_decode.cu).

One cluster of C CTAs per (sequence, KV head); CTA `rank` streams pages rank, rank + C, ...
through S stages, its two consumer groups taking alternate pages.  Consumer warp w forms the
CTA's partial of query-head row w and pushes it into CTA w % C, slot (w / C) C + rank, which
expects C partials for each of its rows.  Checked: the ranks' pages tile the head; each stage
is only ever consumed by one group (what the parity waits need: a stage count that is a
multiple of the group count); the merge slots are unique, inside the 16-slot receive buffer,
and the owners' expected byte counts match what lands; the new row's page id is found in the
producer lane that loaded it; and the size choice (by the layer's length in positions) for the
named shapes.
"""
import itertools

import pytest

GROUPS, CONSUMER_WARPS, RECV_SLOTS, HEAD_DIM = 2, 8, 16, 128
MAX_C, SHORT_C, LONG_C, SHORT_TOKENS = 16, 6, 10, 8192
# clusters of C CTAs resident at once, one CTA per SM (occupancy query on GB300, 152 SMs)
MAX_CLUSTERS = {1: 152, 2: 76, 3: 46, 4: 36, 5: 28, 6: 23, 7: 15, 8: 15, 9: 15, 10: 13,
                11: 8, 12: 8, 13: 7, 14: 7, 15: 7, 16: 7}
NUM_SMS = 152


def niters(rank, C, pages):
    return (pages - 1 - rank) // C + 1 if rank < pages else 0


def own_rows(rank, C, G):
    return (G - 1 - rank) // C + 1 if G > rank else 0


@pytest.mark.parametrize("C", range(1, MAX_C + 1))
def test_pages_tile_the_head(C):
    for pages in range(0, 70):
        seen = [rank + C * it for rank in range(C) for it in range(niters(rank, C, pages))]
        assert sorted(seen) == list(range(pages)), (C, pages)


@pytest.mark.parametrize("stages", [6, 12, 3])
def test_each_stage_belongs_to_one_group(stages):
    owner = {}
    clean = True
    for it in range(200):
        s, grp = it % stages, it % GROUPS
        clean &= owner.setdefault(s, grp) == grp
    # 6 (bf16) and 12 (fp8) stages: every use of a stage is consumed by the same group, in
    # order, so a parity wait can never pass on a phase one use ahead; 3 stages break it
    assert clean == (stages % GROUPS == 0)


@pytest.mark.parametrize("C,G", list(itertools.product(range(1, MAX_C + 1), range(1, 9))))
def test_merge_slots(C, G):
    landed = {}  # owner -> list of (slot, row, rank)
    for rank in range(C):
        for w in range(CONSUMER_WARPS):
            r = w
            if r >= G:
                continue
            owner, slot = r % C, (r // C) * C + rank
            landed.setdefault(owner, []).append((slot, r, rank))
    for owner in range(C):
        got = landed.get(owner, [])
        slots = [s for s, _, _ in got]
        assert len(slots) == len(set(slots)) and all(0 <= s < RECV_SLOTS for s in slots)
        own = own_rows(owner, C, G)
        # bytes the owner's receive barrier expects: own * C partials of (128 + 2) floats
        assert len(got) * (HEAD_DIM + 2) * 4 == own * C * (HEAD_DIM + 2) * 4
        # the owner merges row li C + owner (warp li) from slots li C + j, j = 0 .. C-1
        for li in range(own):
            r = li * C + owner
            for j in range(C):
                assert (li * C + j, r, j) in got


@pytest.mark.parametrize("C", range(1, MAX_C + 1))
def test_new_row_page_id_from_loaded_entries(C):
    for rank in range(C):
        loaded = {}
        for lane in range(32):  # page-table entries rank + C lane and rank + C (lane + 32)
            loaded[(lane, 0)] = rank + C * lane
            loaded[(lane, 1)] = rank + C * (lane + 32)
        for pg_new in range(rank, 80 * C, C):
            li = (pg_new - rank) // C
            if li < 64:
                assert loaded[(li & 31, 0 if li < 32 else 1)] == pg_new


def cluster_size(heads, group, length, tiled=True):
    """C for a launch over a layer of `length` positions (0: the flat split)."""
    if group > 8:
        return 0
    largest = max((c for c in range(1, MAX_C + 1) if heads <= MAX_CLUSTERS[c]), default=0)
    if largest == 0:
        return 0
    if tiled and 2 * heads * largest < NUM_SMS:
        return 0
    want = SHORT_C if length <= SHORT_TOKENS else LONG_C
    return min(largest, want)


@pytest.mark.parametrize("heads,G,length,expect", [
    (8, 4, 4353, 6),        # Llama GQA 32/8, batch 1, 4352 positions: clusters of 6
    (8, 5, 65281, 10),      # batch 1, 64K positions: clusters of 10
    (8, 5, 8193, 10),       # just past the short-layer bound
    (8, 5, 8192, 6),
    (64, 5, 32513, 2),      # Qwen-R1-32B batch 8 (the default workload): pairs
    (128, 5, 4097, 1),      # batch 16: one CTA per head
    (256, 7, 7937, 0),      # Qwen-R1-7B batch 64: more heads than SMs -> flat split
    (4, 4, 300, 0),         # 4 heads: clusters would cover too few SMs -> flat split
    (8, 16, 4353, 0),       # groups above 8 -> flat split
])
def test_cluster_size_for_named_shapes(heads, G, length, expect):
    assert cluster_size(heads, G, length) == expect
