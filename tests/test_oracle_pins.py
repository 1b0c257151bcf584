"""Pins for the CPU oracle: each function checked against something other than
itself -- closed forms, an independent library route, scalar brute force, or
invariants the mathematics fixes -- and mutation checks that show each pin
catches a plausible mistake planted in a copy of the oracle (on the CPU)."""
import math
import os

import numpy as np
import pytest
import scipy.linalg
import scipy.special

import oracle as O
from oracle import pic_oracle as PO

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
RNG = np.random.default_rng(1234)


# ---------------------------------------------------------------- helpers ---
def _pairs(d, style):
    h = d // 2
    if style == O.HALF:
        return np.arange(h), np.arange(h) + h
    return 2 * np.arange(h), 2 * np.arange(h) + 1


def rotary_by_complex(x, pos, theta, style):
    """Independent route: pair (u, w) as the complex number u + i w, times e^{i pos theta}."""
    a, b = _pairs(x.shape[-1], style)
    z = x[..., a] + 1j * x[..., b]
    z = z * np.exp(1j * np.asarray(pos, np.float64)[..., None] * theta)
    out = np.empty_like(x, dtype=np.float64)
    out[..., a], out[..., b] = z.real, z.imag
    return out


def rotary_by_matrix(x, pos, theta, style):
    """Independent route: build the d x d block rotation and multiply."""
    d = x.shape[-1]
    a, b = _pairs(d, style)
    blocks = [np.array([[math.cos(pos * t), -math.sin(pos * t)],
                        [math.sin(pos * t), math.cos(pos * t)]]) for t in theta]
    bd = scipy.linalg.block_diag(*blocks)          # acts on (x_a0, x_b0, x_a1, x_b1, ...)
    order = np.stack([a, b], 1).reshape(-1)
    Rm = np.zeros((d, d))
    Rm[np.ix_(order, order)] = bd
    return x @ Rm.T


def attention_brute_force(q, q_pos, K, V, scale):
    """Scalar loops with math.exp; kv heads expanded by np.repeat (repeat_kv)."""
    T, Hq, d = q.shape
    G = Hq // K.shape[1]
    Kr, Vr = np.repeat(K, G, axis=1), np.repeat(V, G, axis=1)
    out = np.zeros((T, Hq, d))
    for t in range(T):
        for h in range(Hq):
            vis = [s for s in range(K.shape[0]) if s <= q_pos[t]]
            sc = [scale * sum(q[t, h, i] * Kr[s, h, i] for i in range(d)) for s in vis]
            m = max(sc)
            w = [math.exp(x - m) for x in sc]
            z = sum(w)
            for i in range(d):
                out[t, h, i] = sum(w[j] * Vr[vis[j], h, i] for j in range(len(vis))) / z
    return out


def check_rotary(fn):
    """Pin for R(p): hand values at d=2 and agreement with two independent routes."""
    ok = True
    th = np.array([1.0])
    ok &= np.allclose(fn(np.array([1.0, 0.0]), 1, th, O.HALF), [math.cos(1), math.sin(1)], atol=1e-15)
    ok &= np.allclose(fn(np.array([0.0, 1.0]), 1, th, O.HALF), [-math.sin(1), math.cos(1)], atol=1e-15)
    for style in (O.HALF, O.INTERLEAVED):
        theta = O.rope_frequencies(16, 1e4)
        x = RNG.standard_normal((5, 3, 16))
        pos = RNG.integers(0, 200000, size=(5, 3))
        ok &= np.allclose(fn(x, pos, theta, style), rotary_by_complex(x, pos, theta, style),
                          rtol=0, atol=1e-9)
        ok &= np.allclose(fn(x[0, 0], 7, theta, style), rotary_by_matrix(x[0, 0], 7, theta, style),
                          rtol=0, atol=1e-12)
    return bool(ok)


def check_attention(fn):
    scale = 1 / math.sqrt(8)
    ok = True
    for (T, S, Hq, Hkv) in [(3, 5, 4, 2), (4, 9, 6, 3), (2, 4, 2, 2)]:
        q = RNG.standard_normal((T, Hq, 8))
        K = RNG.standard_normal((S, Hkv, 8))
        V = RNG.standard_normal((S, Hkv, 8))
        qp = np.sort(RNG.choice(S, T, replace=False))
        ok &= np.allclose(fn(q, qp, K, V), attention_brute_force(q, qp, K, V, scale), atol=1e-12)
    return bool(ok)


# ------------------------------------------------------------ rotary pins ---
def test_rope_frequencies_closed_form():
    th = O.rope_frequencies(128, 5e5)
    assert th[0] == 1.0
    assert th.shape == (64,)
    np.testing.assert_allclose(th[1:] / th[:-1], 5e5 ** (-2 / 128), rtol=1e-13)
    np.testing.assert_allclose(th[-1], 5e5 ** (-126 / 128), rtol=1e-14)


def test_rotary_pinned():
    assert check_rotary(O.rotary)


def test_rotary_position_zero_is_exact_identity():
    x = RNG.standard_normal((7, 64))
    theta = O.rope_frequencies(64, 1e4)
    assert np.array_equal(O.rotary(x, 0, theta), x)


def test_rotation_preserves_pair_norms():
    theta = O.rope_frequencies(64, 1e4)
    x = RNG.standard_normal((10, 64))
    y = O.rotary(x, RNG.integers(0, 10**5, size=10), theta)
    a, b = _pairs(64, O.HALF)
    np.testing.assert_allclose(x[:, a] ** 2 + x[:, b] ** 2, y[:, a] ** 2 + y[:, b] ** 2, rtol=1e-12)


def test_rope_relative_position_property():
    """<R(m)q, R(n)k> depends only on m - n (the property re-rotation relies on)."""
    theta = O.rope_frequencies(128, 5e5)
    q, k = RNG.standard_normal(128), RNG.standard_normal(128)
    for m, n, s in [(5, 3, 100), (1000, 40, 77777), (0, 0, 131071)]:
        a = O.rotary(q, m, theta) @ O.rotary(k, n, theta)
        b = O.rotary(q, m + s, theta) @ O.rotary(k, n + s, theta)
        assert abs(a - b) < 1e-9 * (1 + abs(a))


# ------------------------------------------------------- re-rotation pins ---
def test_rerotate_delta_zero_identity():
    theta = O.rope_frequencies(128, 5e5)
    k = RNG.standard_normal((9, 128))
    np.testing.assert_allclose(O.rerotate_key(k, 1234, 1234, theta), k, rtol=0, atol=1e-12)
    assert np.array_equal(O.rerotate_key(k, 0, 0, theta), k)


def test_rerotate_additivity_and_inverse():
    theta = O.rope_frequencies(128, 1e6)
    k = RNG.standard_normal((4, 128))
    two = O.rerotate_key(O.rerotate_key(k, 10, 5000, theta), 5000, 140000, theta)
    one = O.rerotate_key(k, 10, 140000, theta)
    np.testing.assert_allclose(two, one, rtol=0, atol=1e-9)
    back = O.rerotate_key(O.rerotate_key(k, 3, 90000, theta), 90000, 3, theta)
    np.testing.assert_allclose(back, k, rtol=0, atol=1e-9)


@pytest.mark.parametrize("style", [O.HALF, O.INTERLEAVED])
def test_relocated_key_equals_key_computed_at_target(style):
    """Eq. 3: a key made at a and moved to b equals the key made at b."""
    theta = O.rope_frequencies(64, 1e4)
    raw = RNG.standard_normal((6, 2, 64))
    a = RNG.integers(0, 5000, size=(6, 1))
    b = RNG.integers(0, 150000, size=(6, 1))
    moved = O.rerotate_key(O.rotary(raw, a, theta, style), a, b, theta, style)
    np.testing.assert_allclose(moved, rotary_by_complex(raw, np.broadcast_to(b, (6, 2)), theta, style),
                               rtol=0, atol=1e-9)


def test_rerotate_d2_hand_case():
    # d = 2, theta = 1: moving (1, 0) from position 0 to 1 gives (cos 1, sin 1)
    r = O.rerotate_key(np.array([1.0, 0.0]), 0, 1, np.array([1.0]))
    np.testing.assert_allclose(r, [math.cos(1), math.sin(1)], atol=1e-15)


# ------------------------------------------------------------ layout pins ---
def _read_golden(name):
    out = {"slot": []}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.split("#")[0].strip()
            if not line:
                continue
            key, *vals = line.split()
            vals = [int(v) for v in vals]
            if key == "slot":
                out["slot"].append(tuple(vals))
            else:
                out[key] = vals
    return out


def test_compose_layout_matches_hand_enumeration():
    g = _read_golden("tiny_layout.txt")
    lay = O.compose_layout(g["doc_len"], g["doc_base"], g["doc_order"], g["prefix_len"][0],
                           g["query_len"][0], g["block_table"], 16)
    assert lay.doc_offset == g["doc_offset"]
    assert lay.doc_delta == g["doc_delta"]
    assert lay.query_start == g["query_start"][0]
    assert lay.ctx_len == g["ctx"][0]
    assert list(lay.inline_pos) == g["inline_pos"]
    for t, s in g["slot"]:
        assert lay.slot_mapping[t] == s


def test_compose_layout_brute_force_properties():
    rng = np.random.default_rng(7)
    for _ in range(20):
        n_pool = int(rng.integers(1, 9))
        lens = rng.integers(1, 70, size=n_pool)
        base = rng.integers(0, 50, size=n_pool)
        order = list(rng.permutation(n_pool)[: int(rng.integers(0, n_pool + 1))])
        P, Tq = int(rng.integers(0, 40)), int(rng.integers(1, 40))
        ctx = P + int(lens[order].sum()) + Tq
        bt = rng.permutation(200)[: -(-ctx // 16) + 3]
        lay = O.compose_layout(lens, base, order, P, Tq, bt, 16)
        # every logical position owned by exactly one of prefix / a doc / query
        owner = np.full(ctx, -2)
        owner[:P] = -1
        for i, d in enumerate(order):
            seg = slice(lay.doc_offset[i], lay.doc_offset[i] + lens[d])
            assert (owner[seg] == -2).all()
            owner[seg] = i
            assert lay.doc_delta[i] == lay.doc_offset[i] - base[d]
        assert (owner[lay.query_start:] == -2).all() and ctx - lay.query_start == Tq
        # slots: injective, on the right pages, in order inside each page
        assert len(set(lay.slot_mapping.tolist())) == ctx
        for t in range(ctx):
            assert lay.slot_mapping[t] // 16 == bt[t // 16] and lay.slot_mapping[t] % 16 == t % 16
        # docs appear in the requested order
        assert lay.doc_offset == sorted(lay.doc_offset)


def _layout_from_golden(g, fn=None):
    fn = fn or O.compose_layout
    return fn(g["doc_len"], g["doc_base"], g["doc_order"], g["prefix_len"][0], g["query_len"][0],
              g["block_table"], g["page_size"][0], span_len=g["span_len"])


def test_compose_layout_with_spans_matches_hand_enumeration():
    g = _read_golden("spans_layout.txt")
    lay = _layout_from_golden(g)
    assert lay.doc_offset == g["doc_offset"]
    assert lay.doc_delta == g["doc_delta"]
    assert lay.span_start == g["span_start"]
    assert lay.query_start == g["query_start"][0]
    assert lay.ctx_len == g["ctx"][0]
    assert list(lay.inline_pos) == g["inline_pos"]
    for t, s in g["slot"]:
        assert lay.slot_mapping[t] == s


def test_pins_catch_planted_span_layout_mistakes():
    """Two plausible misreadings of the canonical order, planted in copies of
    the layout: documents packed back to back with every span after the last
    one, and spans placed before their documents."""
    def spans_at_end(doc_len, doc_base_pos, doc_ids, P, Tq, bt, page_size=16, span_len=None):
        # the spans' tokens treated as part of the query, after the last document
        return PO.compose_layout(doc_len, doc_base_pos, doc_ids, P, Tq + sum(span_len), bt,
                                 page_size)

    def spans_before(doc_len, doc_base_pos, doc_ids, P, Tq, bt, page_size=16, span_len=None):
        return PO.compose_layout(doc_len, doc_base_pos, doc_ids, P + span_len[0], Tq, bt,
                                 page_size, span_len=list(span_len[1:]) + [0])

    g = _read_golden("spans_layout.txt")
    for mutant in (spans_at_end, spans_before):
        lay = _layout_from_golden(g, mutant)
        assert (lay.doc_offset != g["doc_offset"] or list(lay.inline_pos) != g["inline_pos"]), \
            mutant.__name__


def test_zero_spans_reduce_to_the_plain_layout():
    rng = np.random.default_rng(11)
    for _ in range(10):
        n_pool = int(rng.integers(1, 7))
        lens, base = rng.integers(1, 50, size=n_pool), rng.integers(0, 30, size=n_pool)
        order = list(rng.permutation(n_pool))
        P, Tq = int(rng.integers(0, 20)), int(rng.integers(1, 20))
        bt = rng.permutation(100)
        a = O.compose_layout(lens, base, order, P, Tq, bt, 16)
        b = O.compose_layout(lens, base, order, P, Tq, bt, 16, span_len=[0] * len(order))
        assert a.doc_offset == b.doc_offset and a.doc_delta == b.doc_delta
        assert np.array_equal(a.inline_pos, b.inline_pos)
        assert np.array_equal(a.slot_mapping, b.slot_mapping)


def test_compose_layout_with_spans_brute_force_properties():
    """Positions are a partition: each document holds a contiguous run right
    after the previous document's span, and the inline positions are exactly
    the positions no document holds, in increasing order (prefix, spans, query)."""
    rng = np.random.default_rng(8)
    for _ in range(20):
        n_pool = int(rng.integers(1, 9))
        lens, base = rng.integers(1, 70, size=n_pool), rng.integers(0, 50, size=n_pool)
        order = list(rng.permutation(n_pool)[: int(rng.integers(1, n_pool + 1))])
        spans = [int(x) for x in rng.integers(0, 12, size=len(order))]
        P, Tq = int(rng.integers(0, 40)), int(rng.integers(1, 40))
        ctx = P + int(lens[order].sum()) + sum(spans) + Tq
        bt = rng.permutation(300)[: -(-ctx // 16) + 2]
        lay = O.compose_layout(lens, base, order, P, Tq, bt, 16, span_len=spans)
        assert lay.ctx_len == ctx
        doc_at = np.zeros(ctx, bool)
        expect = P
        for i, d in enumerate(order):
            assert lay.doc_offset[i] == expect
            assert lay.doc_delta[i] == expect - base[d]
            assert not doc_at[expect:expect + lens[d]].any()
            doc_at[expect:expect + lens[d]] = True
            expect += lens[d] + spans[i]
        assert np.array_equal(lay.inline_pos, np.flatnonzero(~doc_at))
        assert len(lay.inline_pos) == P + sum(spans) + Tq


def test_compose_layout_rejects_bad_requests():
    with pytest.raises(ValueError):
        O.compose_layout([0], [0], [0], 4, 4, [0], 16)
    with pytest.raises(ValueError):
        O.compose_layout([64], [0], [0], 16, 16, [0, 1], 16)   # needs 6 pages


def test_paged_round_trip_is_bijective():
    g = _read_golden("tiny_layout.txt")
    lay = O.compose_layout(g["doc_len"], g["doc_base"], g["doc_order"], 16, 16, g["block_table"], 16)
    K = RNG.standard_normal((lay.ctx_len, 2, 8))
    V = RNG.standard_normal((lay.ctx_len, 2, 8))
    kc = np.full((10, 2, 16, 8), np.nan)
    vc = np.full((10, 2, 16, 8), np.nan)
    O.scatter_to_pages(lay, K, V, kc, vc, 16)
    assert not np.isnan(kc).any()                  # every slot written exactly once
    K2, V2 = O.gather_from_pages(lay.slot_mapping, kc, vc, 16)
    assert np.array_equal(K, K2) and np.array_equal(V, V2)


# --------------------------------------------------------- attention pins ---
def test_attention_pinned_to_brute_force():
    assert check_attention(O.attention)


def test_attention_single_visible_key_returns_its_value():
    K = RNG.standard_normal((6, 1, 16))
    V = RNG.standard_normal((6, 1, 16))
    q = RNG.standard_normal((1, 3, 16)) * 50
    o = O.attention(q, np.array([0]), K, V)
    for h in range(3):
        assert np.array_equal(o[0, h], V[0, 0])


def test_attention_equal_keys_give_mean_of_visible_values():
    K = np.tile(RNG.standard_normal((1, 2, 16)), (9, 1, 1))
    V = RNG.standard_normal((9, 2, 16))
    q = RNG.standard_normal((2, 4, 16))
    o = O.attention(q, np.array([4, 8]), K, V)
    np.testing.assert_allclose(o[0, 0], V[:5, 0].mean(0), atol=1e-14)
    np.testing.assert_allclose(o[1, 3], V[:9, 1].mean(0), atol=1e-14)


def test_attention_matches_scipy_softmax_and_lse():
    q = RNG.standard_normal((5, 4, 32))
    K = RNG.standard_normal((20, 2, 32))
    V = RNG.standard_normal((20, 2, 32))
    qp = np.array([3, 7, 11, 15, 19])
    o, lse = O.attention(q, qp, K, V, return_lse=True)
    for t in range(5):
        for h in range(4):
            s = q[t, h] @ K[: qp[t] + 1, h // 2].T / math.sqrt(32)
            np.testing.assert_allclose(o[t, h], scipy.special.softmax(s) @ V[: qp[t] + 1, h // 2],
                                       atol=1e-13)
            np.testing.assert_allclose(lse[t, h], scipy.special.logsumexp(s), atol=1e-12)


def test_attention_key_permutation_invariance():
    q = RNG.standard_normal((3, 2, 16))
    K = RNG.standard_normal((12, 1, 16))
    V = RNG.standard_normal((12, 1, 16))
    pos = np.arange(12)
    perm = RNG.permutation(12)
    a = O.attention(q, np.array([5, 9, 11]), K, V, k_pos=pos)
    b = O.attention(q, np.array([5, 9, 11]), K[perm], V[perm], k_pos=pos[perm])
    np.testing.assert_allclose(a, b, atol=1e-13)


# ----------------------------------------------------------- whole path ---
def _tiny_request(base=(0, 0), P=16, lens=(64, 64), Tq=16, d=64, Hq=4, Hkv=1, seed=0,
                  spans=None):
    rng = np.random.default_rng(seed)
    theta = O.rope_frequencies(d, 1e4)
    raw = [rng.standard_normal((n, Hkv, d)) for n in lens]
    k_docs = [O.rotary(raw[i], (base[i] + np.arange(lens[i]))[:, None], theta) for i in range(len(lens))]
    v_docs = [rng.standard_normal((n, Hkv, d)) for n in lens]
    tin = P + (sum(spans) if spans else 0) + Tq
    ctx = sum(lens) + tin
    bt = rng.permutation(-(-ctx // 16) + 2)
    lay = O.compose_layout(list(lens), list(base), list(range(len(lens))), P, Tq, bt, 16,
                           span_len=spans)
    q = rng.standard_normal((tin, Hq, d))
    k = rng.standard_normal((tin, Hkv, d))
    v = rng.standard_normal((tin, Hkv, d))
    return theta, raw, k_docs, v_docs, lay, q, k, v


def test_composed_cache_equals_cache_built_at_target_positions():
    """The PIC identity: relocated doc keys == keys computed directly at their
    final logical positions; values are the cached values unchanged (Eq. 3)."""
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request(base=(5, 11), lens=(37, 50))
    K, V = O.dense_context(lay, k_docs, v_docs, [5, 11], k, v, theta)
    for i in range(2):
        seg = slice(lay.doc_offset[i], lay.doc_offset[i] + raw[i].shape[0])
        direct = rotary_by_complex(raw[i], np.broadcast_to(np.arange(seg.start, seg.stop)[:, None],
                                                           raw[i].shape[:2]), theta, O.HALF)
        np.testing.assert_allclose(K[seg], direct, atol=1e-9)
        assert np.array_equal(V[seg], v_docs[i])
    np.testing.assert_allclose(K[:16], rotary_by_complex(k[:16], np.arange(16)[:, None] + 0 * k[:16, :, 0],
                                                         theta, O.HALF), atol=1e-12)


def test_composed_cache_with_spans_equals_direct_computation():
    """With spans S_k between the documents, the stitched context is the
    request computed in place: document keys rotated directly at their final
    positions, span and query keys at theirs, values unchanged."""
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request(base=(5, 11), lens=(37, 50),
                                                             spans=[9, 4], seed=4)
    K, V = O.dense_context(lay, k_docs, v_docs, [5, 11], k, v, theta)
    expect_k = np.empty_like(K)
    expect_v = np.empty_like(V)
    for i in range(2):
        pos = np.arange(lay.doc_offset[i], lay.doc_offset[i] + raw[i].shape[0])
        expect_k[pos] = rotary_by_complex(raw[i], np.broadcast_to(pos[:, None], raw[i].shape[:2]),
                                          theta, O.HALF)
        expect_v[pos] = v_docs[i]
    ip = lay.inline_pos
    expect_k[ip] = rotary_by_complex(k, np.broadcast_to(ip[:, None], k.shape[:2]), theta, O.HALF)
    expect_v[ip] = v
    np.testing.assert_allclose(K, expect_k, atol=1e-9)
    assert np.array_equal(V, expect_v)
    assert list(ip[16:16 + 9]) == list(range(16 + 37, 16 + 37 + 9))    # S_1 right after D_1


def test_span_tokens_do_not_see_later_documents():
    """Frontier mask with spans: a span token's output does not change when a
    later document's values change, and does change for an earlier one."""
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request(lens=(30, 30), spans=[6, 3], seed=5)
    (o1, _), _, _ = O.cache_hit_prefill(lay, k_docs, v_docs, [0, 0], q, k, v, theta, return_lse=True)
    row = 16 + 2                                      # third token of S_1, before D_2
    v_later = [v_docs[0], v_docs[1] + 5.0]
    (o2, _), _, _ = O.cache_hit_prefill(lay, k_docs, v_later, [0, 0], q, k, v, theta,
                                        return_lse=True)
    np.testing.assert_array_equal(o1[row], o2[row])
    v_earlier = [v_docs[0] + 5.0, v_docs[1]]
    (o3, _), _, _ = O.cache_hit_prefill(lay, k_docs, v_earlier, [0, 0], q, k, v, theta,
                                        return_lse=True)
    assert np.abs(o1[row] - o3[row]).max() > 1.0
    assert np.abs(o1[-1] - o2[-1]).max() > 1.0          # the query sees both


def test_prefill_output_invariant_to_global_position_shift():
    """Shifting every position by s leaves the outputs unchanged (RoPE is relative)."""
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request()
    K, V = O.dense_context(lay, k_docs, v_docs, [0, 0], k, v, theta)
    o1 = O.attention(O.rotary(q, lay.inline_pos[:, None], theta), lay.inline_pos, K, V)
    s = 100000
    Ks = O.rerotate_key(K, np.arange(lay.ctx_len)[:, None], s + np.arange(lay.ctx_len)[:, None], theta)
    o2 = O.attention(O.rotary(q, (lay.inline_pos + s)[:, None], theta), lay.inline_pos + s, Ks, V,
                     k_pos=np.arange(lay.ctx_len) + s)
    np.testing.assert_allclose(o1, o2, atol=1e-9)


def test_needle_is_found_only_at_the_right_relocated_position():
    """A planted doc key aligned with the query after relocation dominates the
    softmax; the same key left at its base position (no re-rotation) does not."""
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request(P=3000, lens=(64, 64), seed=3)
    qpos = lay.inline_pos[-1]
    tgt = lay.doc_offset[1] + 20                    # needle: doc 1, token 20
    qrot = O.rotary(q[-1, 0], qpos, theta)
    needle_at_target = 2.0 * qrot / np.linalg.norm(qrot) * math.sqrt(64)
    raw_needle = O.rotary(needle_at_target, -tgt, theta)       # key as compiled at position 0 ...
    k_docs[1][20, 0] = O.rotary(raw_needle, 20, theta)         # ... of doc 1 at base 0, token 20
    (o, _), K, V = (O.cache_hit_prefill(lay, k_docs, v_docs, [0, 0], q, k, v, theta,
                                        return_lse=True))
    np.testing.assert_allclose(K[tgt, 0], needle_at_target, atol=1e-9)
    assert np.linalg.norm(o[-1, 0] - v_docs[1][20, 0]) < 0.1
    # without re-rotation the needle is not where the query looks
    K_norot = K.copy()
    K_norot[lay.doc_offset[1]:lay.doc_offset[1] + 64] = k_docs[1]
    o_norot = O.attention(O.rotary(q, lay.inline_pos[:, None], theta), lay.inline_pos, K_norot, V)
    assert np.linalg.norm(o_norot[-1, 0] - v_docs[1][20, 0]) > 0.5 * np.linalg.norm(v_docs[1][20, 0])


def test_decode_step_equals_prefill_of_that_token():
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request()
    K, V = O.dense_context(lay, k_docs, v_docs, [0, 0], k, v, theta)
    rng = np.random.default_rng(9)
    qn, kn, vn = rng.standard_normal((4, 64)), rng.standard_normal((1, 64)), rng.standard_normal((1, 64))
    o_dec, K2, V2 = O.decode_step(K, V, qn, kn, vn, lay.ctx_len, theta)
    # the same token as the last row of a prefill over the extended context
    o_pre = O.attention(rotary_by_complex(qn[None], np.full((1, 4), lay.ctx_len), theta, O.HALF),
                        np.array([lay.ctx_len]), K2, V2)
    np.testing.assert_allclose(o_dec, o_pre[0], atol=1e-12)
    np.testing.assert_allclose(K2[-1], rotary_by_complex(kn, np.full((1,), lay.ctx_len), theta, O.HALF),
                               atol=1e-12)


# --------------------------------------------------------- mutation checks ---
def test_pins_catch_planted_rotary_mistakes():
    def wrong_sign(x, pos, theta, style=O.HALF):       # sin with the wrong sign
        return PO.rotary(x, -np.asarray(pos), theta, style)

    def wrong_pairing(x, pos, theta, style=O.HALF):    # half-split treated as interleaved
        return PO.rotary(x, pos, theta, O.INTERLEAVED if style == O.HALF else O.HALF)

    def off_by_one_freq(x, pos, theta, style=O.HALF):  # theta_i shifted by one index
        return PO.rotary(x, pos, np.concatenate([theta[1:], theta[-1:] ** 2]), style)

    for mutant in (wrong_sign, wrong_pairing, off_by_one_freq):
        assert not check_rotary(mutant), mutant.__name__


def test_pins_catch_planted_attention_mistakes():
    def no_scale(q, qp, K, V, **kw):
        return PO.attention(q, qp, K, V, scale=1.0)

    def strict_mask(q, qp, K, V, **kw):                # sees only keys strictly before
        with np.errstate(invalid="ignore"):
            return PO.attention(q, np.asarray(qp) - 1, K, V)

    def wrong_gqa(q, qp, K, V, **kw):                  # head h -> kv head h % Hkv
        G = q.shape[1] // K.shape[1]
        perm = np.array([(h % K.shape[1]) * G + h // K.shape[1] for h in range(q.shape[1])])
        return PO.attention(q[:, np.argsort(perm)], qp, K, V)[:, perm]

    def transposed_pv(q, qp, K, V, **kw):              # values taken from the keys
        return PO.attention(q, qp, K, K)

    for mutant in (no_scale, strict_mask, wrong_gqa, transposed_pv):
        assert not check_attention(mutant), mutant.__name__


def test_pins_catch_planted_rerotation_mistakes():
    theta = O.rope_frequencies(64, 1e4)
    raw = RNG.standard_normal((3, 64))
    a, b = 17, 90210
    good = rotary_by_complex(raw, np.full(3, b), theta, O.HALF)
    made_at_a = O.rotary(raw, a, theta)
    # R(a) R(b)^-1 instead of R(b) R(a)^-1
    swapped = PO.rotary(PO.rotary(made_at_a, -b, theta), a, theta)
    # rotate by the target position instead of the delta
    absolute = PO.rotary(made_at_a, b, theta)
    assert np.allclose(O.rerotate_key(made_at_a, a, b, theta), good, atol=1e-9)
    assert not np.allclose(swapped, good, atol=1e-3)
    assert not np.allclose(absolute, good, atol=1e-3)


# ---------------------------------------------------------- bf16 storage ---
def test_round_bf16_matches_torch_on_float32_values():
    """Library route: torch's float32 -> bfloat16 conversion rounds to nearest even."""
    import torch
    rng = np.random.default_rng(5)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        [0.0, -0.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -(1.0 + 2 ** -8),
                         2.0 ** -130, 3 * 2.0 ** -134, 3.3e38, -3.4e38, np.inf, -np.inf]])
    x32 = x.astype(np.float32)
    ref = torch.from_numpy(x32).to(torch.bfloat16).float().numpy().astype(np.float64)
    got = O.round_bf16(x32.astype(np.float64))
    assert np.array_equal(got, ref)


def test_round_bf16_hand_values_and_brute_force():
    from fractions import Fraction
    assert O.round_bf16(1.0 + 2 ** -8) == 1.0                    # tie -> even (1.0)
    assert O.round_bf16(1.0 + 3 * 2 ** -8) == 1.0 + 2 ** -6      # tie -> even (...10)
    assert O.round_bf16(1.0 + 2 ** -8 + 2 ** -40) == 1.0 + 2 ** -7
    assert np.isnan(O.round_bf16(np.nan))
    rng = np.random.default_rng(11)
    for v in rng.standard_normal(300) * 3:
        # brute force: nearest of all bf16 values with the same exponent, ties even
        e = int(np.floor(np.log2(abs(v))))
        step = Fraction(2) ** (e - 7)
        lo = (Fraction(v) // step) * step
        cands = [lo, lo + step]
        dist = [abs(Fraction(v) - c) for c in cands]
        if dist[0] != dist[1]:
            best = cands[int(dist[1] < dist[0])]
        else:
            best = cands[0] if (lo / step) % 2 == 0 else cands[1]
        assert O.round_bf16(v) == float(best), v


def test_bf16_storage_only_rounds_rotated_keys_and_queries():
    theta, raw, k_docs, v_docs, lay, q, k, v = _tiny_request()
    K, V = O.dense_context(lay, k_docs, v_docs, [0, 0], k, v, theta)
    Kb, Vb = O.dense_context(lay, k_docs, v_docs, [0, 0], k, v, theta, storage="bf16")
    assert np.array_equal(Kb, O.round_bf16(K)) and np.array_equal(Vb, V)
    # unit roundoff of an 8-bit significand: |round(x) - x| <= 2^-8 |x|
    assert (np.abs(Kb - K) <= 2.0 ** -8 * np.abs(K)).all()


# ------------------------------------------- attention-deviation diagnostic ---
def _deviation_brute_force(q, q_pos, Ka, Kb, offsets, lens, edges):
    """Scalar loops: probabilities with math.exp per row, regions by the
    exact rational test e_i <= j / n < e_(i+1)."""
    from fractions import Fraction
    T, Hq, d = q.shape
    G = Hq // Ka.shape[1]
    scale = 1 / math.sqrt(d)

    def probs(K, t, h):
        vis = [s for s in range(K.shape[0]) if s <= q_pos[t]]
        sc = {s: scale * sum(q[t, h, i] * K[s, h // G, i] for i in range(d)) for s in vis}
        m = max(sc.values())
        w = {s: math.exp(x - m) for s, x in sc.items()}
        z = sum(w.values())
        return {s: w[s] / z for s in vis}

    R = len(edges) - 1
    sums, counts = [0.0] * R, [0] * R
    E = [Fraction(e) for e in edges]
    for t in range(T):
        for h in range(Hq):
            pa, pb = probs(Ka, t, h), probs(Kb, t, h)
            for off, n in zip(offsets, lens):
                for j in range(n):
                    u = Fraction(j, n)
                    for i in range(R):
                        if E[i] <= u < E[i + 1]:
                            sums[i] += abs(pa.get(off + j, 0.0) - pb.get(off + j, 0.0))
                            counts[i] += 1
    return np.array(sums), np.array(counts)


def _deviation_case(seed=0, lens=(7, 13, 23), P=3, Tq=4, d=8, Hq=4, Hkv=2):
    rng = np.random.default_rng(seed)
    ctx = P + sum(lens) + Tq
    lay = O.compose_layout(list(lens), [0] * len(lens), list(range(len(lens))), P, Tq,
                           np.arange(-(-ctx // 16)), 16)
    q = rng.standard_normal((Tq, Hq, d))
    q_pos = lay.inline_pos[P:]
    Ka = rng.standard_normal((ctx, Hkv, d))
    Kb = Ka.copy()
    Kb[lay.doc_offset[1]:lay.doc_offset[1] + lens[1]] *= -0.5     # B differs in doc 1
    Kb[lay.doc_offset[2] + 2] += 1.0                              # and one key of doc 2
    return q, q_pos, Ka, Kb, lay, lens


def test_attention_deviation_pinned_to_brute_force():
    for edges in ((0.0, 0.1, 0.9), (0.0, 0.25, 0.5, 1.0)):
        q, q_pos, Ka, Kb, lay, lens = _deviation_case()
        s, c = O.attention_deviation(q, q_pos, Ka, Kb, lay, lens, edges)
        sb, cb = _deviation_brute_force(q, q_pos, Ka, Kb, lay.doc_offset, lens, edges)
        np.testing.assert_allclose(s, sb, rtol=1e-12, atol=1e-15)
        assert np.array_equal(c, cb)


def test_attention_deviation_identity_symmetry_and_bound():
    q, q_pos, Ka, Kb, lay, lens = _deviation_case(seed=3)
    s0, c0 = O.attention_deviation(q, q_pos, Ka, Ka, lay, lens)
    assert (s0 == 0).all() and c0.sum() > 0                  # D(A, A) = 0
    s1, _ = O.attention_deviation(q, q_pos, Ka, Kb, lay, lens)
    s2, _ = O.attention_deviation(q, q_pos, Kb, Ka, lay, lens)
    np.testing.assert_allclose(s1, s2, rtol=1e-14)           # symmetric
    assert s1.sum() <= 2 * q.shape[0] * q.shape[1] + 1e-12   # total variation <= 2 per row
    assert (s1 > 0).all()


def test_pins_catch_planted_deviation_mistakes():
    q, q_pos, Ka, Kb, lay, lens = _deviation_case(seed=5)
    edges = (0.0, 0.1, 0.9)
    ref = _deviation_brute_force(q, q_pos, Ka, Kb, lay.doc_offset, lens, edges)[0]

    class Shifted:  # regions taken one document off
        doc_offset = lay.doc_offset[1:] + [lay.doc_offset[0]]
    s_shift, _ = O.attention_deviation(q, q_pos, Ka, Kb, Shifted, lens, edges)
    # unnormalised region edges (fractions of the longest block)
    s_abs, _ = O.attention_deviation(q, q_pos, Ka, Kb, lay, [max(lens)] * len(lens), edges)
    for s in (s_shift, s_abs):
        assert not np.allclose(s, ref, rtol=1e-6)
