"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test ties the oracle to something other than itself:
  * Fig. 1b's printed mask pattern (golden fixture),
  * the training-mask formulation of Sec. 3.1 evaluated as a dense masked softmax
    by a library routine (torch SDPA, float64) -- a different computation from
    the oracle's gather over the retained set,
  * dense causal attention when nothing is evicted (library routine),
  * the degenerate w = 0 / all-evict case (out = v_j exactly),
  * the closed-form retained count and its monotonicity,
  * the sign rule that round(sigmoid(x)) reduces to (Sec. 3.2),
  * App. H's KV-read coefficient for the byte model.
A few tests also show that a plausible mistake (an off-by-one window, a wrong
scale, a transposed operand) is caught by these pins.
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle
import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _bf16(x) -> np.ndarray:
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


def _f64(bits: np.ndarray) -> np.ndarray:
    return torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).double().numpy()


def _rand_case(rng, T, G, D, p):
    q = _bf16(rng.standard_normal((T, G, D)))
    k = _bf16(rng.standard_normal((T, D)))
    v = _bf16(rng.standard_normal((T, D)))
    lg = _bf16(rng.standard_normal(T) + (math.inf if p >= 1 else (-math.inf if p <= 0 else
                                                                    _probit(p))))
    return q, k, v, lg


def _probit(p):
    import statistics
    return statistics.NormalDist().inv_cdf(p)


def _read_fig1b():
    rows = []
    with open(os.path.join(GOLDEN, "fig1b_mask.txt")) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            rows.append(line.split()[1:])
    return rows


# --------------------------------------------------------------------------- Fig. 1b


def test_fig1b_pattern_all_evict():
    """With every alpha = 1, the retained sets reproduce the printed mask (w = 3)."""
    rows = _read_fig1b()
    T = len(rows)
    lg = _bf16(np.ones(T))  # logit 1 > 0 -> alpha = 1 for every key
    for j, row in enumerate(rows):
        R = set(oracle.retained(lg, j, 3).tolist())
        for i, e in enumerate(row):
            if e == "-":
                assert i not in R, (j, i)
            elif e == "0":
                assert i in R, (j, i)
            else:  # "L": log(1 - alpha) with alpha = 1 -> -inf -> masked
                assert i not in R, (j, i)
        assert j in R  # diagonal is always 0


def test_fig1b_pattern_no_evict():
    """With every alpha = 0, log(1 - alpha) = 0: nothing outside the causal mask is hidden."""
    rows = _read_fig1b()
    lg = _bf16(-np.ones(len(rows)))
    for j, row in enumerate(rows):
        R = set(oracle.retained(lg, j, 3).tolist())
        for i, e in enumerate(row):
            assert (i in R) == (e != "-"), (j, i)


def test_fig1b_rejects_off_by_one_window():
    """A window one shorter or longer than the figure's does not reproduce it."""
    rows = _read_fig1b()
    lg = _bf16(np.ones(len(rows)))
    for w_bad in (2, 4):
        mismatch = False
        for j, row in enumerate(rows):
            R = set(oracle.retained(lg, j, w_bad).tolist())
            for i, e in enumerate(row):
                if (i in R) != (e == "0"):
                    mismatch = True
        assert mismatch, w_bad


# --------------------------------------------------------------------------- decision rule


@pytest.mark.parametrize("bits,expect", [
    (0x0000, 0),   # +0: sigmoid = 1/2 exactly, the tie keeps
    (0x8000, 0),   # -0
    (0x0001, 1),   # smallest positive subnormal
    (0x8001, 0),   # smallest negative subnormal
    (0x3F80, 1),   # 1.0
    (0xBF80, 0),   # -1.0
    (0x7F80, 1),   # +inf: sigmoid = 1
    (0xFF80, 0),   # -inf: sigmoid = 0
    (0x7FC0, 0),   # NaN: compares false, keeps
    (0xFFC1, 0),   # negative NaN
    (0x7F7F, 1),   # largest finite
])
def test_alpha_sign_rule_edges(bits, expect):
    assert oracle.alpha(bits) == expect


def test_alpha_matches_rounded_sigmoid():
    """round(sigmoid(x)) computed in float64 agrees wherever float64 resolves sigmoid - 1/2."""
    rng = np.random.default_rng(0)
    xs = np.concatenate([rng.standard_normal(4000) * 3, rng.standard_normal(1000) * 1e-6,
                         np.array([2.0 ** -30, -2.0 ** -30, 40.0, -40.0])])
    bits = _bf16(xs)
    for b, x in zip(bits, _f64(bits)):
        if abs(x) < 2.0 ** -40:
            continue
        s = 1.0 / (1.0 + math.exp(-x))
        assert s != 0.5
        assert oracle.alpha(int(b)) == (1 if s > 0.5 else 0), x


# --------------------------------------------------------------------------- retained counts


@pytest.mark.parametrize("w", [0, 1, 3, 16, 255, 256])
def test_closed_form_count_and_monotone(w):
    rng = np.random.default_rng(w + 7)
    T = 700
    lg = _bf16(rng.standard_normal(T) + 0.7)
    a = _f64(lg) > 0
    prev = 0
    for j in range(T):
        n = len(oracle.retained(lg, j, w))
        evicted_left = int(np.sum(a[: max(0, j - w)]))  # positions i <= j - w - 1
        assert n == (j + 1) - evicted_left
        assert n >= prev
        prev = n


def test_retained_sorted_and_contains_window():
    rng = np.random.default_rng(3)
    T, w = 300, 17
    lg = _bf16(rng.standard_normal(T) + 1.0)
    for j in (0, 5, 17, 18, 150, T - 1):
        R = oracle.retained(lg, j, w)
        assert np.all(np.diff(R) > 0)
        assert set(range(max(0, j - w), j + 1)) <= set(R.tolist())


def test_expected_count_statistics():
    """Mean retained count over many heads is within a few sigma of T - p (T - w - 1)."""
    rng = np.random.default_rng(11)
    T, w, p, H = 2000, 256, 0.875, 64
    mu = _probit(p)
    counts = []
    for _ in range(H):
        lg = _bf16(rng.standard_normal(T) + mu)
        counts.append(len(oracle.retained(lg, T - 1, w)))
    expect = T - p * (T - w - 1)
    sigma = math.sqrt((T - w - 1) * p * (1 - p) / H)
    assert abs(np.mean(counts) - expect) < 5 * sigma


# --------------------------------------------------------------------------- attention values


def _sdpa_masked(q, k, v, mask_add, scale):
    """Dense masked softmax via the library routine, float64.

    q: [Tq, D] queries, k, v: [T, D], mask_add: [Tq, T] additive mask -> [Tq, D].
    """
    return torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(np.ascontiguousarray(q))[None], torch.from_numpy(k)[None],
        torch.from_numpy(v)[None], attn_mask=torch.from_numpy(np.ascontiguousarray(mask_add))[None],
        scale=scale).numpy()[0]


def _training_mask(alpha, w):
    """M_alpha of Sec. 3.1 / Fig. 1b for binary alpha: -inf above the diagonal,
    0 inside the window, log(1 - alpha_i) outside it."""
    T = len(alpha)
    M = np.full((T, T), -np.inf)
    with np.errstate(divide="ignore"):
        la = np.log(1.0 - alpha.astype(np.float64))
    for j in range(T):
        for i in range(j + 1):
            M[j, i] = 0.0 if j - i <= w else la[i]
    return M


@pytest.mark.parametrize("T,G,D,w,p,seed", [
    (40, 4, 16, 3, 0.6, 0), (64, 1, 32, 0, 0.5, 1), (50, 7, 8, 9, 0.875, 2),
    (33, 5, 128, 4, 0.9, 3), (20, 2, 16, 30, 0.7, 4)])
def test_brute_force_training_mask(T, G, D, w, p, seed):
    """Every step's decode equals the dense softmax with the training mask M_alpha."""
    rng = np.random.default_rng(seed)
    q, k, v, lg = _rand_case(rng, T, G, D, p)
    alpha = (_f64(lg) > 0).astype(np.float64)
    M = _training_mask(alpha, w)
    scale = 1.0 / math.sqrt(D)
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    # the query at step j is row j of M for each of the G heads
    ref = np.stack([_sdpa_masked(qd[:, g], kd, vd, M, scale) for g in range(G)],
                   axis=1)  # [T, G, D]
    for j in range(T):
        got = oracle.decode(q[j], k, v, lg, j, w)
        np.testing.assert_allclose(got, ref[j], rtol=0, atol=1e-12)


def test_no_eviction_equals_dense_causal():
    rng = np.random.default_rng(5)
    T, G, D, w = 96, 4, 64, 8
    q, k, v, _ = _rand_case(rng, T, G, D, 0.5)
    lg = _bf16(-np.abs(rng.standard_normal(T)) - 0.01)  # all logits < 0: nothing evicted
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    for g in range(G):
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(qd[:, g])[None], torch.from_numpy(kd)[None],
            torch.from_numpy(vd)[None], is_causal=True).numpy()[0]
        for j in range(T):
            got = oracle.decode(q[j], k, v, lg, j, w)[g]
            np.testing.assert_allclose(got, ref[j], rtol=0, atol=1e-12)


def test_window_covering_everything_is_dense():
    rng = np.random.default_rng(6)
    T, G, D = 70, 2, 32
    q, k, v, _ = _rand_case(rng, T, G, D, 0.5)
    lg = _bf16(np.ones(T))  # all evict, but the window covers the whole history
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    ref = torch.nn.functional.scaled_dot_product_attention(
        torch.from_numpy(qd.transpose(1, 0, 2)), torch.from_numpy(kd)[None].expand(G, T, D),
        torch.from_numpy(vd)[None].expand(G, T, D), is_causal=True).numpy()
    for j in range(T):
        np.testing.assert_allclose(oracle.decode(q[j], k, v, lg, j, T), ref[:, j], rtol=0,
                                   atol=1e-12)


def test_w0_all_evict_keeps_only_current_token():
    rng = np.random.default_rng(7)
    T, G, D = 50, 3, 128
    q, k, v, _ = _rand_case(rng, T, G, D, 0.5)
    lg = _bf16(np.ones(T))
    vd = _f64(v)
    for j in range(T):
        assert oracle.retained(lg, j, 0).tolist() == [j]
        out = oracle.decode(q[j], k, v, lg, j, 0)
        assert np.array_equal(out, np.broadcast_to(vd[j], out.shape))


def test_scale_and_gqa_rows():
    """Explicit scale equals the default 1/sqrt(D); G heads equal G single-head calls."""
    rng = np.random.default_rng(8)
    T, G, D, w = 60, 5, 128, 10
    q, k, v, lg = _rand_case(rng, T, G, D, 0.8)
    j = T - 1
    full = oracle.decode(q[j], k, v, lg, j, w)
    np.testing.assert_array_equal(full, oracle.decode(q[j], k, v, lg, j, w, 1 / math.sqrt(D)))
    for g in range(G):
        np.testing.assert_array_equal(full[g], oracle.decode(q[j][g:g + 1], k, v, lg, j, w)[0])


def test_empty_history_gives_zeros():
    q = _bf16(np.ones((2, 8)))
    k = _bf16(np.ones((1, 8)))
    out = oracle.decode(q, k, k, _bf16(np.ones(1)), -1, 4)
    assert np.all(out == 0)


def test_pins_catch_planted_mistakes():
    """A wrong scale or swapped K/V in the oracle's call would fail the brute-force pin."""
    rng = np.random.default_rng(9)
    T, G, D, w = 30, 2, 16, 4
    q, k, v, lg = _rand_case(rng, T, G, D, 0.7)
    j = T - 1
    lg[j - w] = _bf16([1.0])[0]  # the token at distance w is flagged: an off-by-one drops it
    alpha = (_f64(lg) > 0).astype(np.float64)
    M = _training_mask(alpha, w)
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    ref = np.stack([_sdpa_masked(qd[j:j + 1, g], kd, vd, M[j:j + 1], 1 / math.sqrt(D))[0]
                    for g in range(G)])
    good = oracle.decode(q[j], k, v, lg, j, w)
    np.testing.assert_allclose(good, ref, atol=1e-12, rtol=0)
    assert not np.allclose(oracle.decode(q[j], k, v, lg, j, w, 2 / math.sqrt(D)), ref, atol=1e-6)
    assert not np.allclose(oracle.decode(q[j], v, k, lg, j, w), ref, atol=1e-6)
    assert not np.allclose(oracle.decode(q[j], k, v, lg, j, w - 1), ref, atol=1e-6)


# --------------------------------------------------------------------------- App. H byte model


def test_appH_kv_read_coefficient():
    vals = {}
    with open(os.path.join(GOLDEN, "appH_llama31_8b_reads.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                key, val = line.split()
                vals[key] = float(val)
    n, d_kv = int(vals["layers"]), int(vals["d_kv"])
    kv_heads = d_kv // workloads.HEAD_DIM
    coef = workloads.kv_bytes_per_token_head() * kv_heads * n  # bytes per (B*L) per step
    digits = int(vals["printed_digits"])
    assert float(f"{coef:.{digits - 1}e}") == vals["kv_read_coefficient"]


# --------------------------------------------------------------------------- App. B neuron


def test_borrowed_neuron_decisions_and_attention():
    """App. B: the decision of each token comes from the sign of element 0 of the group's
    first query head, and the attention no longer depends on that element's value: the
    first head equals the masked dense softmax with the element set to 0, and the group's
    other heads equal the plain path's bit for bit."""
    rng = np.random.default_rng(11)
    T, G, D, w = 48, 4, 32, 5
    q, k, v, _ = _rand_case(rng, T, G, D, 0.5)
    q[:, 0, 0] = _bf16(rng.standard_normal(T) + _probit(0.7))  # the neuron carries the logit
    lg, q_att = oracle.borrowed(q, G)  # one KV head: logits [T, 1]
    lg = lg[:, 0]
    alpha = (_f64(q[:, 0, 0]) > 0).astype(np.float64)
    M = _training_mask(alpha, w)
    scale = 1.0 / math.sqrt(D)
    q0 = _f64(q)[:, 0].copy()
    q0[:, 0] = 0.0
    ref0 = _sdpa_masked(q0, _f64(k), _f64(v), M, scale)
    # same signs, other magnitudes: nothing may change
    q2 = q.copy()
    q2[:, 0, 0] = _bf16(np.where(alpha > 0, 1.0, -1.0) * (0.5 + rng.random(T)))
    lg2, q_att2 = oracle.borrowed(q2, G)
    lg2 = lg2[:, 0]
    for j in range(T):
        want = set(i for i in range(j + 1) if alpha[i] == 0 or j - i <= w)
        assert set(oracle.retained(lg, j, w).tolist()) == want
        assert np.array_equal(oracle.retained(lg2, j, w), oracle.retained(lg, j, w))
        got = oracle.decode(q_att[j], k, v, lg, j, w)
        np.testing.assert_allclose(got[0], ref0[j], rtol=0, atol=1e-12)
        plain = oracle.decode(q[j], k, v, lg, j, w)
        assert np.array_equal(got[1:], plain[1:])
        assert np.array_equal(oracle.decode(q_att2[j], k, v, lg2, j, w), got)


def test_borrowed_neuron_multi_head_layout():
    """[B, kv_heads * G, D] queries: the logit of KV head h is element 0 of query head h * G."""
    rng = np.random.default_rng(12)
    B, H, G, D = 3, 5, 3, 16
    q = _bf16(rng.standard_normal((B, H * G, D)))
    lg, q_att = oracle.borrowed(q, G)
    assert lg.shape == (B, H)
    for b in range(B):
        for h in range(H):
            assert lg[b, h] == q[b, h * G, 0]
            assert q_att[b, h * G, 0] == 0
            for g in range(G):
                d0 = 1 if g == 0 else 0
                assert np.array_equal(q_att[b, h * G + g, d0:], q[b, h * G + g, d0:])
    with pytest.raises(ValueError):
        oracle.borrowed(q[:, :-1], G)


# --------------------------------------------------------------------------- Sec. 5 ablation


@pytest.mark.parametrize("w", [0, 1, 3, 16])
def test_immediate_eviction_is_delayed_on_shifted_decisions(w):
    """Immediate eviction (token i decided by alpha_{i+w}) equals delayed eviction on the
    decisions shifted by w; w = 0 makes the two policies identical; the count is
    (j + 1) - #{k in [w, j - 1] : alpha_k = 1}."""
    rng = np.random.default_rng(13 + w)
    T = 120
    lg = _bf16(rng.standard_normal(T) + 0.4)
    alpha = (_f64(lg) > 0).astype(int)
    shifted = np.concatenate([lg[w:], np.zeros(w, dtype=np.uint16)])  # +0 keeps
    for j in range(T):
        imm = oracle.retained(lg, j, w, immediate=True)
        assert np.array_equal(imm, oracle.retained(shifted, j, w))
        if w == 0:
            assert np.array_equal(imm, oracle.retained(lg, j, w))
        assert len(imm) == (j + 1) - int(alpha[w:j].sum()) if j > w else len(imm) == j + 1


def test_immediate_eviction_decode_brute_force():
    """Decode under immediate eviction equals the dense softmax with its mask."""
    rng = np.random.default_rng(17)
    T, G, D, w = 50, 3, 32, 4
    q, k, v, lg = _rand_case(rng, T, G, D, 0.6)
    alpha = (_f64(lg) > 0).astype(np.float64)
    M = np.full((T, T), -np.inf)
    for j in range(T):
        for i in range(j + 1):
            if j - i <= w or alpha[i + w] == 0:
                M[j, i] = 0.0
    scale = 1.0 / math.sqrt(D)
    qd, kd, vd = _f64(q), _f64(k), _f64(v)
    ref = np.stack([_sdpa_masked(qd[:, g], kd, vd, M, scale) for g in range(G)], axis=1)
    differs = False
    for j in range(T):
        got = oracle.decode(q[j], k, v, lg, j, w, immediate=True)
        np.testing.assert_allclose(got, ref[j], rtol=0, atol=1e-12)
        differs |= not np.array_equal(got, oracle.decode(q[j], k, v, lg, j, w))
    assert differs  # the ablation is a different policy


# --------------------------------------------------------------------------- fp8 KV page format


def _torch_e4m3_codes(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.asarray(x, dtype=np.float32)).to(torch.float8_e4m3fn) \
        .view(torch.uint8).numpy()


def test_e4m3_values_match_torch():
    """Every code's value equals PyTorch's float8_e4m3fn (an independent implementation of
    the OCP E4M3FN definition), NaN codes included."""
    ref = torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).double().numpy()
    mine = np.array([oracle.e4m3_to_double(c) for c in range(256)])
    assert np.array_equal(np.isnan(ref), np.isnan(mine))
    ok = ~np.isnan(ref)
    assert np.array_equal(ref[ok], mine[ok])
    assert mine[0x7E] == 448.0 and mine[0x08] == 2.0 ** -6 and mine[0x01] == 2.0 ** -9
    assert mine[0x38] == 1.0 and np.isnan(mine[0x7F]) and np.isnan(mine[0xFF])


def test_e4m3_encoding_matches_torch_and_ties_to_even():
    """Round to nearest, ties to even, on every value, every midpoint between neighbours
    and random floats in [-448, 448]; saturation above 448."""
    vals = np.array([oracle.e4m3_to_double(c) for c in range(0x7F)])  # 0 .. 448, increasing
    assert np.all(np.diff(vals) > 0)
    mids = (vals[:-1] + vals[1:]) / 2  # exact in float32 (at most 5 significant bits)
    rng = np.random.default_rng(5)
    xs = np.concatenate([vals, mids, -vals, -mids, rng.uniform(-448, 448, 4000),
                         rng.standard_normal(4000) * 0.01]).astype(np.float32)
    mine = np.array([oracle.e4m3_from_float(x) for x in xs], dtype=np.uint8)
    assert np.array_equal(mine, _torch_e4m3_codes(xs))
    for m_lo, m_hi in zip(range(0, 0x7E), range(1, 0x7F)):
        got = oracle.e4m3_from_float((vals[m_lo] + vals[m_hi]) / 2)
        assert got == (m_lo if m_lo % 2 == 0 else m_hi)
    for x, code in [(449.0, 0x7E), (464.0, 0x7E), (1e30, 0x7E), (-1e30, 0xFE), (-0.0, 0x80)]:
        assert oracle.e4m3_from_float(x) == code
    assert oracle.e4m3_from_float(float("nan")) == 0x7F


def test_quantize_rows_bounds_and_scale():
    """scale = fl32(amax / 448); the largest element maps to +-448 (code 0x7E / 0xFE); every
    dequantised element is within half a step of its value; zero rows stay zero."""
    rng = np.random.default_rng(6)
    rows = _bf16(rng.standard_normal((64, 128)) * rng.uniform(1e-3, 50, (64, 1)))
    rows[3] = 0
    rows[5, 7] = _bf16([-300.0])[0]  # a negative outlier sets amax
    codes, scales = oracle.quantize_rows_e4m3(rows)
    x = _f64(rows)
    amax = np.abs(x).max(axis=1).astype(np.float32)
    assert np.array_equal(scales, (amax / np.float32(448)).astype(np.float32))
    assert scales[3] == 0 and np.all(codes[3] == 0)
    deq = oracle.dequantize_e4m3(codes, scales)
    for i in range(64):
        if scales[i] == 0:
            continue
        top = np.argmax(np.abs(x[i]))
        assert codes[i, top] & 0x7F == 0x7E
        y = x[i] / scales[i]
        step = np.where(np.abs(y) >= 2.0 ** -6, 2.0 ** (np.floor(np.log2(np.maximum(np.abs(y), 2.0 ** -6))) - 3),
                        2.0 ** -9)
        assert np.all(np.abs(deq[i] - x[i]) <= 0.5 * step * scales[i] * (1 + 1e-6))
    assert codes[5, 7] == 0xFE


def test_fp8_decode_exact_rows_equal_bf16_decode():
    """Rows already on the E4M3 grid times 2^k with amax = 448 * 2^k quantise exactly, so the
    quantised-cache attention equals the bf16 attention on the same rows."""
    rng = np.random.default_rng(7)
    T, G, D, w = 40, 3, 128, 6
    grid = np.array([oracle.e4m3_to_double(c) for c in range(0x7F)])
    def exact_rows(n):
        r = rng.choice(np.concatenate([grid, -grid]), (n, D))
        r[:, 0] = 448.0
        return r * 2.0 ** rng.integers(-12, -4, (n, 1))
    kf, vf = exact_rows(T), exact_rows(T)
    k, v = _bf16(kf), _bf16(vf)
    assert np.array_equal(_f64(k), kf) and np.array_equal(_f64(v), vf)
    q = _bf16(rng.standard_normal((G, D)))
    lg = _bf16(rng.standard_normal(T) + 0.5)
    kc, ks = oracle.quantize_rows_e4m3(k)
    vc, vs = oracle.quantize_rows_e4m3(v)
    assert np.array_equal(oracle.dequantize_e4m3(kc, ks), kf)
    for j in (0, 17, T - 1):
        np.testing.assert_allclose(oracle.decode_fp8(q, kc, ks, vc, vs, lg, j, w),
                                   oracle.decode(q, k, v, lg, j, w), rtol=0, atol=1e-12)
    # a plausible mistake (the value scales applied to the keys) is caught
    bad = oracle.decode_fp8(q, kc, vs, vc, ks, lg, T - 1, w)
    assert not np.allclose(bad, oracle.decode(q, k, v, lg, T - 1, w), atol=1e-6)
