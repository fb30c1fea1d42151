"""Host-side model of the page layouts (restated from dms_internal.cuh and the decode kernels'
shared-memory reads).

bf16 pages: 64 K rows then 64 V rows of 256 bytes, each row's sixteen 16-byte chunks permuted
by chunk ^ (row & 7).  fp8 pages: 64 K rows of 128 E4M3 codes (k8_offset), V transposed (128
rows of 64 codes, vt8_offset), then 64 key and 64 value fp32 row scales: 16896 bytes, one bulk
copy.  Checked: each map is a bijection onto its region; the regions tile the page; the four
codes an m16n8k16 A-fragment register needs are 4 consecutive, 4-aligned bytes; and the warp's
shared-memory reads of a staged page fall on distinct banks (ldmatrix row groups for bf16, the
16-byte K loads of a quarter warp and the 32-bit V^T loads of a warp for fp8).
"""
import itertools

import pytest

PAGE_TOKENS, HEAD_DIM = 64, 128
ROW_BYTES = 2 * HEAD_DIM                        # bf16 row
HALF_BYTES = PAGE_TOKENS * ROW_BYTES            # 16384
HALF_BYTES_FP8 = PAGE_TOKENS * HEAD_DIM         # 8192
SCALE_BYTES = 2 * PAGE_TOKENS * 4               # 512
CODES_BYTES_FP8 = 2 * HALF_BYTES_FP8            # 16384
PAGE_BYTES_FP8 = CODES_BYTES_FP8 + SCALE_BYTES  # 16896


def swizzled_offset(row, chunk):
    return row * ROW_BYTES + ((chunk ^ (row & 7)) << 4)


def pair_index(j):
    return (j & 1) | ((j >> 3) << 1)


def k8_swizzle(row):
    return (row & 7) ^ ((row & 1) << 2)


def k8_offset(row, d):
    kk, j = d >> 4, d & 15
    chunk = (4 * (kk >> 2) + ((j & 7) >> 1)) ^ k8_swizzle(row)
    return row * 128 + (chunk << 4) + 4 * (kk & 3) + pair_index(j)


def vt8_offset(slot, d):
    j = slot & 15
    chunk = (slot >> 4) ^ ((d >> 1) & 3)
    return HALF_BYTES_FP8 + d * 64 + (chunk << 4) + 4 * ((j & 7) >> 1) + pair_index(j)


def scale_offset(kv, row):  # page_scales_fp8(pool, page)[kv * 64 + row]
    return CODES_BYTES_FP8 + 4 * (kv * PAGE_TOKENS + row)


def bank(byte_offset):
    return (byte_offset // 4) % 32


def test_bf16_rows_bijective_and_ldmatrix_conflict_free():
    offs = {swizzled_offset(r, c) for r in range(PAGE_TOKENS) for c in range(16)}
    assert offs == set(range(0, HALF_BYTES, 16))
    # an ldmatrix 8x8 matrix reads one logical chunk of 8 consecutive rows (16 bytes each):
    # the 8 physical chunks must fall on 8 different 16-byte bank groups
    for r0 in range(0, PAGE_TOKENS, 8):
        for c in range(16):
            groups = {(swizzled_offset(r0 + i, c) // 16) % 8 for i in range(8)}
            assert len(groups) == 8, (r0, c)


def test_fp8_page_regions_tile_the_page():
    k = [k8_offset(r, d) for r in range(PAGE_TOKENS) for d in range(HEAD_DIM)]
    v = [vt8_offset(s, d) for s in range(PAGE_TOKENS) for d in range(HEAD_DIM)]
    sc = [scale_offset(kv, r) + b for kv in range(2) for r in range(PAGE_TOKENS) for b in range(4)]
    assert sorted(k) == list(range(0, HALF_BYTES_FP8))
    assert sorted(v) == list(range(HALF_BYTES_FP8, CODES_BYTES_FP8))
    assert sorted(sc) == list(range(CODES_BYTES_FP8, PAGE_BYTES_FP8))
    # one bulk copy per page: size and every page start (page * 16896) on 16 bytes
    assert PAGE_BYTES_FP8 % 16 == 0 and PAGE_BYTES_FP8 == 16896


@pytest.mark.parametrize("c", range(4))
def test_fp8_fragment_words_are_consecutive(c):
    # K: thread (g, c) of k-step kk needs d = 16 kk + {2c, 2c+1, 2c+8, 2c+9} of its row, in
    # that order as the low / high halves of two f16x2 registers
    for row, kk in itertools.product(range(PAGE_TOKENS), range(8)):
        ds = [16 * kk + 2 * c, 16 * kk + 2 * c + 1, 16 * kk + 2 * c + 8, 16 * kk + 2 * c + 9]
        offs = [k8_offset(row, d) for d in ds]
        assert offs[0] % 4 == 0 and offs == list(range(offs[0], offs[0] + 4)), (row, kk)
        # and word kk % 4 of the 16-byte chunk (4 (kk / 4) + c) ^ k8_swizzle(row)
        assert offs[0] == row * 128 + (((4 * (kk >> 2) + c) ^ k8_swizzle(row)) << 4) + 4 * (kk & 3)
    # V^T: thread (g, c) of row d needs tokens {2c, 2c+1, 2c+8, 2c+9} of a 16-slot block
    for d, blk in itertools.product(range(HEAD_DIM), range(4)):
        slots = [16 * blk + 2 * c, 16 * blk + 2 * c + 1, 16 * blk + 2 * c + 8, 16 * blk + 2 * c + 9]
        offs = [vt8_offset(s, d) for s in slots]
        assert offs[0] % 4 == 0 and offs == list(range(offs[0], offs[0] + 4)), (d, blk)


def test_fp8_k_loads_of_a_quarter_warp_hit_distinct_bank_groups():
    # lane (g, c4) of a quarter warp (g = 2q, 2q + 1) loads 16 bytes of row tb + g at chunk
    # (4 kg + c4) ^ k8_swizzle(g); eight 16-byte loads, eight distinct 16-byte bank groups
    for tb, kg, q in itertools.product(range(0, PAGE_TOKENS, 16), range(2), range(4)):
        groups = set()
        for g in (2 * q, 2 * q + 1):
            for c4 in range(4):
                off = (tb + g) * 128 + (((4 * kg + c4) ^ k8_swizzle(g)) << 4)
                groups.add((off // 16) % 8)
        assert len(groups) == 8, (tb, kg, q)


def test_fp8_vt_loads_of_a_warp_hit_distinct_banks():
    # lane (g, c4) loads the 32-bit word of row d0 = 16 mt + g (and d0 + 8), block tb / 16
    for tb, mt, half in itertools.product(range(0, PAGE_TOKENS, 16), range(8), range(2)):
        banks = set()
        for g, c4 in itertools.product(range(8), range(4)):
            d = 16 * mt + g + 8 * half
            banks.add(bank(vt8_offset(tb + 2 * c4, d)))
        assert len(banks) == 32, (tb, mt, half)


def test_a_planted_swizzle_mistake_is_caught():
    # without the (row & 1) << 2 term the two rows of a quarter warp share four chunks
    groups = set()
    for g in (0, 1):
        for c4 in range(4):
            groups.add(((g * 128 + (((c4) ^ (g & 7)) << 4)) // 16) % 8)
    assert len(groups) < 8
