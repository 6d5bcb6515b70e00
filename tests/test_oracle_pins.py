"""Pins of the CPU oracle against what the paper and plain mathematics fix.

Nothing here compares the oracle with itself: each test checks it against a value
the paper prints, a hand-worked fixture, a closed form, a special case the paper
names, or a brute force written differently (dense softmax with -inf masking).
Runs on the CPU only.
"""
import numpy as np
import pytest

import oracle as O
from golden_io import map_cases

rng_global = np.random.default_rng(1234)


def bf16(x):
    """float array -> bf16 bit patterns (round to nearest even), as uint16."""
    f = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    rounded = (f + 0x7FFF + ((f >> 16) & 1)) >> 16
    return rounded.astype(np.uint16)


def bf16_to_f64(b):
    return (np.asarray(b, np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# ---------------------------------------------------------------- map: paper values

@pytest.mark.parametrize("Tc,D", [(130816, 1013), (32512, 245)])
def test_bin_count_matches_appendix_a(Tc, D):
    """App. A: with 128 sink, 1,024 recent and 128-token bins, a 130,816-token
    context has D = 1,013 bins and a 32,512-token one has D = 245."""
    geo = O.Geometry(L=1, H=1, Hkv=1, D=D)
    far = O.distance_bin(geo.sink, Tc, geo)           # farthest compressible position
    near = O.distance_bin(Tc - geo.recent - 1, Tc, geo)  # nearest compressible position
    assert near == 0
    assert far == D - 1
    M = np.ones((1, 1, D), np.uint8)
    assert O.validate(M, [Tc], geo) == O.OK
    short = O.Geometry(L=1, H=1, Hkv=1, D=D - 1)
    assert O.validate(np.ones((1, 1, D - 1), np.uint8), [Tc], short) == O.ERR_RANGE


@pytest.mark.parametrize("case", map_cases(), ids=lambda c: c["name"])
def test_map_hand_worked_cases(case):
    geo = O.Geometry(**case["geometry"])
    m = O.map_pattern(case["M"], case["ctx"], geo)
    got = [list(m.idx[m.ioff[h]:m.ioff[h + 1]]) for h in range(len(m.len))]
    assert got == case["kept"]


def test_memory_arithmetic_sec43_and_app_c():
    """Sec. 4.3 / App. C: the full Llama-3.1-8B context cache at 128K is
    15.625 GiB and Distance-KV's 65.4% cut leaves 5.41 GiB; Qwen2.5-7B's full
    cache is 6.836 GiB and a 52.0% cut leaves 3.28 GiB. Context '128K' is
    128,000 tokens and a row is head_dim * 2 bytes of K plus the same of V."""
    geo = O.Geometry(L=1, H=1, Hkv=1, D=(128000 - 1152 + 127) // 128)
    m = O.map_pattern(np.ones((1, 1, geo.D), np.uint8), [128000], geo, with_idx=False)
    rows_per_head = int(m.len[0])
    row_bytes = 2 * 128 * 2  # K + V, bf16
    gib = 2.0 ** 30
    llama = rows_per_head * 32 * 8 * row_bytes / gib
    qwen = rows_per_head * 28 * 4 * row_bytes / gib
    assert llama == pytest.approx(15.625, abs=1e-12)
    assert round(llama * (1 - 0.654), 2) == 5.41
    assert round(qwen, 3) == 6.836
    assert round(qwen * (1 - 0.520), 2) == 3.28


# ---------------------------------------------------------------- map: closed forms

def closed_form_len(M, geo, layer, g, Tc):
    """Kept count of one KV head, counted bin by bin instead of position by
    position: min(Tc, S+R) + sum over union bins d of |bin d inside the span|."""
    G = geo.H // geo.Hkv
    union = M[layer, g * G:(g + 1) * G].max(axis=0)
    C = Tc - geo.sink - geo.recent
    n = min(Tc, geo.sink + geo.recent)
    for d in range(geo.D):
        if union[d]:
            n += max(0, min(geo.bin_width, C - d * geo.bin_width))
    return n


@pytest.mark.parametrize("seed", range(6))
def test_length_closed_form(seed):
    rng = np.random.default_rng(seed)
    L, Hkv, G = 2, 3, [1, 2, 4][seed % 3]
    geo = O.Geometry(L=L, H=Hkv * G, Hkv=Hkv, D=7, sink=5, recent=9, bin_width=6)
    M = (rng.random((L, geo.H, geo.D)) < 0.4).astype(np.uint8)
    Tc = rng.integers(0, 5 + 9 + 7 * 6 + 1, size=4).astype(np.int32)
    Tc[0] = 5 + 9 + 7 * 6          # exactly D full bins
    Tc[1] = 5 + 9 + 3 * 6 + 2      # partial far bin
    m = O.map_pattern(M, Tc, geo, reserve=seed)
    h = 0
    for l in range(L):
        for b in range(len(Tc)):
            for g in range(Hkv):
                assert m.len[h] == closed_form_len(M, geo, l, g, int(Tc[b]))
                h += 1
    steps = (m.len.astype(np.int64) + seed)
    assert np.array_equal(m.off, np.concatenate([[0], np.cumsum(steps)]))
    assert np.array_equal(m.ioff, np.concatenate([[0], np.cumsum(m.len.astype(np.int64))]))


def test_streaming_llm_special_case():
    """M == 0 is StreamingLLM with 128 sink + 1,024 recent tokens (baseline setup)."""
    geo = O.Geometry(L=1, H=4, Hkv=2, D=40)
    for Tc in (0, 1, 500, 1152, 1153, 5000):
        m = O.map_pattern(np.zeros((1, 4, 40), np.uint8), [Tc], geo)
        expect = sorted(set(range(min(128, Tc))) | set(range(max(0, Tc - 1024), Tc)))
        for h in range(2):
            assert list(m.idx[m.ioff[h]:m.ioff[h + 1]]) == expect


def test_all_keep_is_dense():
    geo = O.Geometry(L=1, H=2, Hkv=1, D=40)
    for Tc in (3, 1152, 6000):
        m = O.map_pattern(np.ones((1, 2, 40), np.uint8), [Tc], geo)
        assert list(m.idx) == list(range(Tc))


def test_head_level_special_case():
    """Sec. 3.2: M[l,h,d] = z[l,h] is a distance-agnostic head-level policy: a KV
    head keeps everything if any of its q-heads has z=1, else only sink+recent."""
    rng = np.random.default_rng(7)
    geo = O.Geometry(L=3, H=8, Hkv=2, D=20, sink=4, recent=10, bin_width=5)
    z = (rng.random((3, 8)) < 0.3).astype(np.uint8)
    M = np.repeat(z[:, :, None], 20, axis=2)
    Tc = 4 + 10 + 20 * 5
    m = O.map_pattern(M, [Tc], geo)
    for l in range(3):
        for g in range(2):
            h = l * 2 + g
            any_on = z[l, g * 4:(g + 1) * 4].any()
            assert m.len[h] == (Tc if any_on else 14)


def test_gqa_union_of_query_head_sets():
    """Sec. 3.4: a KV head keeps a position iff some q-head of its group does.
    Per-q-head kept sets come from the MHA reading (one KV head per q-head)."""
    rng = np.random.default_rng(11)
    G, Hkv, L = 4, 2, 2
    gqa = O.Geometry(L=L, H=G * Hkv, Hkv=Hkv, D=9, sink=3, recent=4, bin_width=3)
    mha = O.Geometry(L=L, H=G * Hkv, Hkv=G * Hkv, D=9, sink=3, recent=4, bin_width=3)
    M = (rng.random((L, G * Hkv, 9)) < 0.25).astype(np.uint8)
    Tc = [3 + 4 + 27, 20]
    mg = O.map_pattern(M, Tc, gqa)
    mm = O.map_pattern(M, Tc, mha)
    for l in range(L):
        for b in range(2):
            for g in range(Hkv):
                hg = (l * 2 + b) * Hkv + g
                union = set()
                for j in range(G):
                    hm = (l * 2 + b) * (G * Hkv) + g * G + j
                    union |= set(mm.idx[mm.ioff[hm]:mm.ioff[hm + 1]].tolist())
                assert mg.idx[mg.ioff[hg]:mg.ioff[hg + 1]].tolist() == sorted(union)


def test_indices_ascending_unique_in_range():
    rng = np.random.default_rng(5)
    geo = O.Geometry(L=2, H=6, Hkv=2, D=16, sink=8, recent=16, bin_width=7)
    M = (rng.random((2, 6, 16)) < 0.5).astype(np.uint8)
    Tc = [8 + 16 + 16 * 7, 30, 0, 24]
    m = O.map_pattern(M, Tc, geo)
    h = 0
    for l in range(2):
        for b in range(4):
            for g in range(2):
                seg = m.idx[m.ioff[h]:m.ioff[h + 1]]
                assert np.all(np.diff(seg) > 0)
                assert seg.size == 0 or (seg[0] >= 0 and seg[-1] < Tc[b])
                h += 1


def test_bad_arguments():
    geo = O.Geometry(L=1, H=3, Hkv=2, D=4)
    assert O.validate(np.zeros((1, 3, 4), np.uint8), [10], geo) == O.ERR_INVALID_ARG
    geo = O.Geometry(L=1, H=2, Hkv=1, D=4, sink=1, recent=1, bin_width=2)
    M = np.zeros((1, 2, 4), np.uint8)
    M[0, 0, 0] = 2
    assert O.validate(M, [10], geo) == O.ERR_INVALID_ARG
    assert O.validate(np.zeros((1, 2, 4), np.uint8), [-1], geo) == O.ERR_INVALID_ARG
    assert O.validate(np.zeros((1, 2, 4), np.uint8), [1 + 1 + 8], geo) == O.OK
    assert O.validate(np.zeros((1, 2, 4), np.uint8), [1 + 1 + 9], geo) == O.ERR_RANGE


# ---------------------------------------------------------------- compaction

def test_compact_is_ordered_gather():
    rng = np.random.default_rng(3)
    L, B, Hkv, T, hd = 2, 2, 2, 40, 128
    geo = O.Geometry(L=L, H=4, Hkv=Hkv, D=6, sink=2, recent=5, bin_width=6)
    M = (rng.random((L, 4, 6)) < 0.5).astype(np.uint8)
    Tc = [40, 17]
    K = rng.integers(0, 2 ** 16, size=(L, B, Hkv, T, hd), dtype=np.uint16)
    V = rng.integers(0, 2 ** 16, size=(L, B, Hkv, T, hd), dtype=np.uint16)
    m = O.map_pattern(M, Tc, geo, reserve=3)
    Kc, Vc = O.compact(m, L, B, Hkv, K, V, T)
    h = 0
    for l in range(L):
        for b in range(B):
            for g in range(Hkv):
                keep = m.idx[m.ioff[h]:m.ioff[h + 1]]
                rows = slice(m.off[h], m.off[h] + m.len[h])
                assert np.array_equal(Kc[rows], K[l, b, g][keep])
                assert np.array_equal(Vc[rows], V[l, b, g][keep])
                gap = slice(m.off[h] + m.len[h], m.off[h + 1])
                assert not Kc[gap].any() and not Vc[gap].any()
                h += 1


# ---------------------------------------------------------------- attention

def masked_dense_attention(q, K, V, keep, scale):
    """Brute force: scores over ALL positions, dropped ones set to -inf."""
    qf, Kf, Vf = bf16_to_f64(q), bf16_to_f64(K), bf16_to_f64(V)
    s = scale * (qf @ Kf.T)
    s[:, ~keep] = -np.inf
    s = s - s.max(axis=1, keepdims=True)
    e = np.exp(s)
    return (e / e.sum(axis=1, keepdims=True)) @ Vf


@pytest.mark.parametrize("G,hd", [(1, 4), (2, 8), (4, 128), (7, 128)])
def test_compacted_attention_equals_masked_dense(G, hd):
    rng = np.random.default_rng(G * 100 + hd)
    T = 40
    geo = O.Geometry(L=1, H=G, Hkv=1, D=9, head_dim=hd, sink=2, recent=3, bin_width=4)
    M = (rng.random((1, G, 9)) < 0.4).astype(np.uint8)
    K = bf16(rng.standard_normal((1, 1, 1, T, hd)))
    V = bf16(rng.standard_normal((1, 1, 1, T, hd)))
    q = bf16(rng.standard_normal((1, G, hd)))
    m = O.map_pattern(M, [T], geo)
    Kc, Vc = O.compact(m, 1, 1, 1, K, V, T, head_dim=hd)
    got = O.decode(m, 0, 1, G, 1, q, Kc, Vc, head_dim=hd)[0]
    keep = np.zeros(T, bool)
    keep[m.idx] = True
    want = masked_dense_attention(q[0], K[0, 0, 0], V[0, 0, 0], keep, 1 / np.sqrt(hd))
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_all_keep_attention_is_dense_attention():
    rng = np.random.default_rng(9)
    T, hd, G = 33, 128, 4
    geo = O.Geometry(L=1, H=G, Hkv=1, D=10, sink=1, recent=2, bin_width=3)
    K = bf16(rng.standard_normal((1, 1, 1, T, hd)))
    V = bf16(rng.standard_normal((1, 1, 1, T, hd)))
    q = bf16(rng.standard_normal((1, G, hd)))
    m = O.map_pattern(np.ones((1, G, 10), np.uint8), [T], geo)
    Kc, Vc = O.compact(m, 1, 1, 1, K, V, T)
    got = O.decode(m, 0, 1, G, 1, q, Kc, Vc)[0]
    want = masked_dense_attention(q[0], K[0, 0, 0], V[0, 0, 0], np.ones(T, bool), 1 / np.sqrt(hd))
    np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)


def test_single_row_returns_that_value_row():
    rng = np.random.default_rng(1)
    q = bf16(rng.standard_normal((3, 128)))
    K = bf16(rng.standard_normal((1, 128)) * 50)
    V = bf16(rng.standard_normal((1, 128)))
    out = O.attend(q, K, V)
    assert np.array_equal(out, np.repeat(bf16_to_f64(V), 3, axis=0))


def test_identical_keys_give_mean_of_values():
    rng = np.random.default_rng(2)
    q = bf16(rng.standard_normal((2, 128)))
    K = np.repeat(bf16(rng.standard_normal((1, 128))), 5, axis=0)
    V = bf16(rng.standard_normal((5, 128)))
    out = O.attend(q, K, V)
    np.testing.assert_allclose(out, np.repeat(bf16_to_f64(V).mean(0, keepdims=True), 2, 0),
                               rtol=0, atol=1e-15)


def test_softmax_weights_sum_to_one_and_two_row_closed_form():
    rng = np.random.default_rng(4)
    q = bf16(rng.standard_normal((4, 128)))
    K = bf16(rng.standard_normal((50, 128)) * 3)
    V = bf16(rng.standard_normal((50, 128)))
    _, w = O.attend(q, K, V, with_weights=True)
    np.testing.assert_allclose(w.sum(1), 1.0, rtol=0, atol=1e-14)
    assert (w >= 0).all()
    # Two rows, q = e0, k1 = 2 e0, k2 = 0, scale 1: w1 = e^2 / (e^2 + 1).
    q2 = np.zeros((1, 128), np.float32)
    q2[0, 0] = 1
    K2 = np.zeros((2, 128), np.float32)
    K2[0, 0] = 2
    V2 = np.zeros((2, 128), np.float32)
    V2[0, :] = 1
    V2[1, :] = -3
    out, w2 = O.attend(bf16(q2), bf16(K2), bf16(V2), scale=1.0, with_weights=True)
    w1 = np.e ** 2 / (np.e ** 2 + 1)
    np.testing.assert_allclose(w2[0], [w1, 1 - w1], rtol=1e-15)
    np.testing.assert_allclose(out[0], w1 * 1 + (1 - w1) * -3, rtol=1e-14)


def test_default_scale_is_inverse_sqrt_head_dim():
    rng = np.random.default_rng(6)
    q = bf16(rng.standard_normal((2, 128)))
    K = bf16(rng.standard_normal((9, 128)))
    V = bf16(rng.standard_normal((9, 128)))
    a = O.attend(q, K, V)
    b = O.attend(q, K, V, scale=1 / np.sqrt(128))
    assert np.array_equal(a, b)
    c = O.attend(q, K, V, scale=0.5)
    assert not np.allclose(a, c)


def test_zero_rows_give_zero_output():
    q = bf16(np.ones((2, 128)))
    out = O.attend(q, np.zeros((0, 128), np.uint16), np.zeros((0, 128), np.uint16))
    assert not out.any() and np.isfinite(out).all()


def test_append_then_decode_equals_attention_with_new_token():
    """Sec. 3.4: generated tokens are appended after the packed context and kept
    in full; attention then covers context-kept rows plus every appended row."""
    rng = np.random.default_rng(8)
    L, B, Hkv, G, T, hd = 2, 2, 2, 2, 30, 128
    geo = O.Geometry(L=L, H=Hkv * G, Hkv=Hkv, D=6, sink=2, recent=4, bin_width=4)
    M = (rng.random((L, Hkv * G, 6)) < 0.3).astype(np.uint8)
    Tc = [30, 11]
    K = bf16(rng.standard_normal((L, B, Hkv, T, hd)))
    V = bf16(rng.standard_normal((L, B, Hkv, T, hd)))
    m = O.map_pattern(M, Tc, geo, reserve=3)
    Kc, Vc = O.compact(m, L, B, Hkv, K, V, T)
    layer = 1
    new_k = [bf16(rng.standard_normal((B, Hkv, hd))) for _ in range(2)]
    new_v = [bf16(rng.standard_normal((B, Hkv, hd))) for _ in range(2)]
    for step in range(2):
        O.append(m, layer, B, Hkv, 3, [step] * B, new_k[step], new_v[step], Kc, Vc)
    q = bf16(rng.standard_normal((B, Hkv * G, hd)))
    got = O.decode(m, layer, B, Hkv * G, Hkv, q, Kc, Vc, n_rows_app=[2] * B)
    for b in range(B):
        for g in range(Hkv):
            h = (layer * B + b) * Hkv + g
            keep = m.idx[m.ioff[h]:m.ioff[h + 1]]
            Kall = np.concatenate([K[layer, b, g][keep], new_k[0][b, g][None], new_k[1][b, g][None]])
            Vall = np.concatenate([V[layer, b, g][keep], new_v[0][b, g][None], new_v[1][b, g][None]])
            want = masked_dense_attention(q[b, g * G:(g + 1) * G], Kall, Vall,
                                          np.ones(len(Kall), bool), 1 / np.sqrt(hd))
            np.testing.assert_allclose(got[b, g * G:(g + 1) * G], want, rtol=1e-12, atol=1e-12)
    with pytest.raises(O.OracleError):
        O.append(m, layer, B, Hkv, 3, [3] * B, new_k[0], new_v[0], Kc, Vc)


# ---------------------------------------------------------------- exact-budget Top-K (Eq. 3, App. A.3)

def test_budget_rounding_app_a3():
    # K_rho = round(rho L H D), round read as floor(x + 1/2).
    assert O.budget(0.35, 32, 32, 1013) == 363059  # 363059.2
    assert O.budget(0.5, 1, 1, 5) == 3             # 2.5 rounds up
    assert O.budget(0.5, 1, 1, 3) == 2             # 1.5 rounds up
    assert O.budget(0.25, 28, 28, 64) == 12544     # exact
    assert O.budget(0.0, 32, 32, 128) == 0
    assert O.budget(1.0, 32, 32, 128) == 32 * 32 * 128
    assert O.budget(-0.1, 1, 1, 1) == -1 and O.budget(1.1, 1, 1, 1) == -1 and O.budget(float("nan"), 1, 1, 1) == -1


def _rank_by_definition(P):
    """Rank of every entry under the selection order, counted pairwise: larger
    value first, equal values (+0 == -0) by lower index, NaN after all numbers."""
    n = len(P)
    rank = np.zeros(n, np.int64)
    for i in range(n):
        for j in range(n):
            if i == j:
                continue
            a, b = P[j], P[i]  # does j come before i?
            if np.isnan(a) != np.isnan(b):
                before = np.isnan(b)
            elif not np.isnan(a) and a != b:
                before = a > b
            else:
                before = j < i
            rank[i] += int(before)
    return rank


@pytest.mark.parametrize("seed", range(4))
def test_topk_matches_pairwise_rank_definition(seed):
    rng = np.random.default_rng(seed)
    n = 23
    P = rng.choice(np.array([0.0, -0.0, 0.25, 0.5, 0.5, 0.75, 1.0, np.nan, -np.inf, np.inf], np.float32), n)
    P[:5] = rng.random(5).astype(np.float32)
    rank = _rank_by_definition(P)
    assert sorted(rank.tolist()) == list(range(n))  # a total order
    for K in range(n + 1):
        M = O.topk_mask(P, K)
        assert np.array_equal(M, (rank < K).astype(np.uint8)), f"K={K}"
        assert int(M.sum()) == K


def test_topk_equals_stable_library_sort():
    rng = np.random.default_rng(7)
    P = rng.random((6, 8, 37)).astype(np.float32)
    P[1, 2, :10] = 0.5  # ties
    flat = P.reshape(-1)
    order = np.lexsort((np.arange(flat.size), -flat.astype(np.float64)))
    for K in (0, 1, 100, 1776 // 2, flat.size - 1, flat.size):
        want = np.zeros(flat.size, np.uint8)
        want[order[:K]] = 1
        assert np.array_equal(O.topk_mask(P, K).reshape(-1), want)


def test_topk_bad_arguments():
    P = np.zeros(5, np.float32)
    for K in (-1, 6):
        with pytest.raises(O.OracleError):
            O.topk_mask(P, K)
