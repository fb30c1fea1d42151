"""Host-side model of the tiled decode kernel's work list (a-5), restated from dms_decode.cu.

All heads' pages form one flat list (a per-head page prefix over the counts).  It is split
over the CTAs in contiguous ranges, balanced, except that, in large launches, the last 16
CTAs take 0.9 of the others' weight.  Each CTA walks its range as part A (the pages of its
first head), part C (the pages of its last head), then part B (the heads in between), a
segment per head.  Checked on random ragged heads (including empty ones): the ranges tile
the list, each page's owner is the CTA whose range holds it, every page is visited once, each
(head, page) of the walk is the flat page it stands for, and segments never cross a head.
"""
import numpy as np
import pytest

TAPER_CTAS, TAPER_PERMILLE = 16, 900


class Split:
    def __init__(self, q, r):
        self.q, self.r = q, r

    def begin(self, k):
        return k * self.q + min(k, self.r)

    def cta_of(self, x):
        big = self.r * (self.q + 1)
        return x // (self.q + 1) if x < big else self.r + (x - big) // self.q


class Partition:
    def __init__(self, N, P):
        self.P1, self.N1 = P, N
        if TAPER_CTAS > 0 and P > 4 * TAPER_CTAS and N >= 8 * P:
            self.P1 = P - TAPER_CTAS
            self.N1 = N * self.P1 * 1000 // (self.P1 * 1000 + TAPER_CTAS * TAPER_PERMILLE)
        self.a = Split(self.N1 // self.P1, self.N1 % self.P1)
        T, N2 = P - self.P1, N - self.N1
        self.b = Split(N2 // T if T > 0 else 0, N2 % T if T > 0 else 0)

    def begin(self, k):
        return self.a.begin(k) if k <= self.P1 else self.N1 + self.b.begin(k - self.P1)

    def cta_of(self, x):
        return self.a.cta_of(x) if x < self.N1 else self.P1 + self.b.cta_of(x - self.N1)


def head_of_page(pstart, heads, x):
    lo, hi = 0, heads
    while lo < hi:
        mid = (lo + hi) >> 1
        if pstart[mid] > x:
            hi = mid
        else:
            lo = mid + 1
    return lo - 1


def walk(pstart, heads, pbeg, pend):
    """(flat, h, pg, seg_start, seg_end) per iteration, as the kernel's PageWalk yields them."""
    h_first, h_last = head_of_page(pstart, heads, pbeg), head_of_page(pstart, heads, pend - 1)
    a_end = pend if h_first == h_last else pstart[h_first + 1]
    c_beg = pend if h_first == h_last else pstart[h_last]
    nA, nC, n = a_end - pbeg, pend - c_beg, pend - pbeg

    def flat(it):
        return pbeg + it if it < nA else (c_beg + it - nA if it < nA + nC else a_end + it - nA - nC)

    h, pg, out = h_first, 0, []
    for it in range(n):
        if it in (0, nA, nA + nC):
            x = flat(it)
            h = head_of_page(pstart, heads, x)
            pg = x - pstart[h]
        npg = pstart[h + 1] - pstart[h]
        seg_start = it == 0 or pg == 0
        seg_end = it in (nA - 1, nA + nC - 1, n - 1) or pg == npg - 1
        out.append((flat(it), h, pg, seg_start, seg_end))
        pg += 1
        if pg == npg:
            pg = 0
            h += 1
            while h < heads and pstart[h + 1] == pstart[h]:
                h += 1
            h = min(h, heads - 1)
    return out, nA, nC


@pytest.mark.parametrize("heads,P,seed", [(8, 1, 0), (256, 152, 1), (64, 152, 2), (872, 152, 3),
                                          (5, 7, 4), (300, 148, 5)])
def test_partition_and_walk(heads, P, seed):
    rng = np.random.default_rng(seed)
    for trial in range(20):
        pages = rng.integers(0, 40, heads)
        pages[rng.random(heads) < 0.15] = 0  # empty heads
        if trial % 5 == 0:
            pages = rng.integers(0, 3, heads)  # few pages: small launches split evenly
        pstart = np.concatenate([[0], np.cumsum(pages)]).astype(np.int64)
        N = int(pstart[-1])
        if N == 0:
            continue
        Pk = min(P, N)
        part = Partition(N, Pk)
        begins = [part.begin(k) for k in range(Pk + 1)]
        assert begins[0] == 0 and begins[-1] == N and all(np.diff(begins) >= 0)
        for x in range(N):
            k = part.cta_of(x)
            assert begins[k] <= x < begins[k + 1]
        counts = np.diff(begins)
        if part.P1 < Pk:  # tapered: the last CTAs take 0.9 of the others' pages
            head_mean, tail_mean = counts[:part.P1].mean(), counts[part.P1:].mean()
            assert abs(tail_mean / head_mean - TAPER_PERMILLE / 1000) < 0.05
        else:
            assert counts.max() - counts.min() <= 1
        seen = np.zeros(N, dtype=int)
        for k in range(Pk):
            pbeg, pend = begins[k], begins[k + 1]
            if pend == pbeg:
                continue
            it_list, nA, nC = walk(pstart, heads, pbeg, pend)
            flats = [f for f, *_ in it_list]
            # parts in order: first head's pages, last head's pages, then the middle heads
            assert flats == (list(range(pbeg, pbeg + nA)) + list(range(pend - nC, pend)) +
                             list(range(pbeg + nA, pend - nC)))
            for f, h, pg, ss, se in it_list:
                seen[f] += 1
                assert pstart[h] + pg == f and 0 <= pg < pages[h]
            # segments: from a start to the next end, one head, consecutive pages
            seg = None
            for f, h, pg, ss, se in it_list:
                if ss:
                    assert seg is None
                    seg = (h, pg)
                assert seg is not None and seg[0] == h
                if se:
                    seg = None
            assert seg is None
        assert np.all(seen == 1)
