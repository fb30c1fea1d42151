"""Host-side model of the tcgen05 prefill kernel's work decomposition, checked against the oracle.

The kernel (dms_prefill.cu) splits a prompt into (query head, 128-query tile) units and each
unit's keys into 128-row tiles: first the retained (alpha = 0) rows of the head's compacted
list that the tile's last query can see, then the dense band [j0 - w, jmax] with its start
rounded down to a multiple of 8.  Each row masks a tile to one contiguous run of keys.  This
test restates that arithmetic and checks, on random prompts, that every row's visible keys
are exactly the oracle's retained set R_j (Sec. 3.1 mask) with no key counted twice, that
every staged copy stays inside the packed arrays, and that the CTA's unit iterator (mixed
radix, no divisions) visits the same units as plain division.
"""
import numpy as np
import pytest

import oracle

ROWS = 128  # queries per tile
KEYS = 128  # keys per tile
EVICT, KEEP = 0x3F80, 0xBF80  # bf16 +1.0 (alpha = 1) and -1.0 (alpha = 0)


def _cdiv(a, b):
    return (a + b - 1) // b


def _tiles(P, w, before, j0):
    """The key tiles of the query tile starting at j0: (retained, r0, rows)."""
    jmax = min(j0 + ROWS, P) - 1
    nc = before[jmax - w] if jmax - w > 0 else 0
    bs = max(0, j0 - w) & ~7
    n_ct = _cdiv(nc, KEYS)
    out = []
    for t in range(n_ct + _cdiv(jmax + 1 - bs, KEYS)):
        if t < n_ct:
            r0 = t * KEYS
            out.append((True, r0, min(KEYS, nc - r0), nc))
        else:
            r0 = bs + (t - n_ct) * KEYS
            out.append((False, r0, min(KEYS, jmax + 1 - r0), jmax + 1))
    return out


def _visible(j, w, before, tile):
    """The run lo .. lo + nvis - 1 of the tile's rows that query j sees."""
    retained, r0, rows, _ = tile
    if retained:
        bj = before[j - w] if j - w > 0 else 0
        return 0, min(max(bj - r0, 0), rows)
    lo = max(j - w - r0, 0)
    return lo, max(min(j - r0, rows - 1) - lo + 1, 0)


@pytest.mark.parametrize("P,w,p,seed", [
    (300, 32, 0.75, 1), (1000, 64, 0.9, 2), (77, 8, 0.5, 3), (200, 0, 1.0, 4),
    (130, 500, 0.6, 5), (257, 128, 0.0, 6), (1, 0, 1.0, 7), (129, 3, 0.7, 8),
    (700, 256, 0.75, 9), (1100, 16, 0.5, 10),
])
def test_tiles_cover_the_retained_set(P, w, p, seed):
    rng = np.random.default_rng(seed)
    alpha = rng.random(P) < p  # 1 = evict
    logits = np.where(alpha, EVICT, KEEP).astype(np.uint16)
    kept = np.flatnonzero(~alpha)  # the compacted list: positions of alpha = 0 tokens
    before = np.concatenate([[0], np.cumsum(~alpha)])  # alpha = 0 tokens below each position
    for j0 in range(0, P, ROWS):
        tiles = _tiles(P, w, before, j0)
        for retained, r0, rows, limit in tiles:
            assert 1 <= rows <= KEYS and r0 >= 0 and r0 + rows <= limit
            assert r0 % 8 == 0  # the pack's row-chunk permutation lines up with the tile's
        for j in range(j0, min(j0 + ROWS, P)):
            seen = []
            for tile in tiles:
                lo, nvis = _visible(j, w, before, tile)
                assert 0 <= lo and lo + nvis <= tile[2]
                keys = np.arange(tile[1] + lo, tile[1] + lo + nvis)
                seen.extend(kept[keys] if tile[0] else keys)
            seen = np.array(seen, dtype=np.int64)
            assert len(np.unique(seen)) == len(seen), (j, "a key counted twice")
            np.testing.assert_array_equal(np.sort(seen), oracle.retained(logits, j, w))


def _digits(u, G, H, B):
    g, u = u % G, u // G
    hk, u = u % H, u // H
    return [g, hk, u % B, u // B]


def _advance(it, st, G, H, B):
    g, hk, b, rank = it
    g += st[0]
    c = g >= G
    g -= G * c
    hk += st[1] + c
    c = hk >= H
    hk -= H * c
    b += st[2] + c
    c = b >= B
    b -= B * c
    return [g, hk, b, rank + st[3] + c]


def test_unit_iterator_matches_division():
    """A CTA visits units c, c + grid, ...; u = ((rank B + b) H + hk) G + g."""
    rng = np.random.default_rng(0)
    for _ in range(500):
        G, H, B, nq = (int(rng.integers(1, 9)), int(rng.integers(1, 9)),
                       int(rng.integers(1, 70)), int(rng.integers(1, 70)))
        n_units = nq * B * H * G
        grid = min(int(rng.choice([152, 148, 7, 1, n_units])), n_units)
        st = _digits(grid, G, H, B)
        for c in rng.choice(grid, size=min(grid, 4), replace=False):
            it, u = _digits(int(c), G, H, B), int(c)
            while u < n_units:
                rank, r = divmod(u, B * H * G)
                b, hq = divmod(r, H * G)
                assert it == [hq % G, hq // G, b, rank]
                it, u = _advance(it, st, G, H, B), u + grid
            assert it[3] >= nq  # past the last query tile exactly when past the last unit
