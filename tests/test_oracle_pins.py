"""Pins for the fp64 oracle against facts fixed by mathematics, not by itself.

Each test would fail under a plausible slip in the oracle (a dropped term, a
wrong sign, a wrong head or page index, a transposed operand):
  * closed forms: one key, all-equal scores, the hand-derived two-key case,
    the empty key set;
  * invariants: a constant added to every score, key order, page placement;
  * library cross-checks: scipy.special.logsumexp / softmax on the scores;
  * brute force: pure-Python loops straight from the pool on tiny workloads;
  * the merge algebra: split + merge equals the unsplit attention.
"""

import math
import os

import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import oracle
from oracle import attention_rows, bf16_bits_to_f64, lse_merge
from paper_2606_17518_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rng(seed=0):
    return np.random.default_rng(seed)


# ---------------------------------------------------------------- bf16 widening
def test_bf16_widening_known_patterns():
    bits = np.array([0x3F80, 0xC000, 0x0000, 0x8000, 0x3E00, 0x7F80, 0x0001, 0x4049],
                    dtype=np.uint16)
    got = bf16_bits_to_f64(bits)
    want = [1.0, -2.0, 0.0, -0.0, 0.125, math.inf, 2.0 ** -133, 3.140625]
    assert got.tolist() == want
    assert np.signbit(got[3])
    assert np.isnan(bf16_bits_to_f64(np.array([0x7FC0], dtype=np.uint16)))[0]


def test_workload_bf16_rounding_is_rne():
    import torch
    x = _rng(3).standard_normal(20000).astype(np.float32)
    # halfway cases: low 16 bits exactly 0x8000
    half = (np.arange(1, 200, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, half, -half])
    mine = wl.round_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(mine, ref)


# ---------------------------------------------------------------- paging
def test_gather_logical_brute_force():
    rng = _rng(1)
    pool = rng.integers(0, 2 ** 16, size=(7, 3, 4, 5), dtype=np.uint16)
    table = np.array([5, 0, 6, 2], dtype=np.int32)
    for length in (0, 1, 3, 4, 5, 13, 16):
        for head in range(3):
            got = oracle.gather_logical(pool, table, length, 4, head)
            assert got.shape == (length, 5)
            for j in range(length):
                page, slot = table[j // 4], j % 4
                want = bf16_bits_to_f64(pool[page, head, slot])
                assert np.array_equal(got[j], want, equal_nan=True)


# ---------------------------------------------------------------- closed forms
def test_single_key_returns_its_value_row():
    rng = _rng(2)
    q = rng.standard_normal((3, 16))
    k = rng.standard_normal((1, 16))
    v = rng.standard_normal((1, 9))
    o, lse = attention_rows(q, k, v, 0.37)
    assert np.array_equal(o, np.repeat(v, 3, axis=0))
    np.testing.assert_allclose(lse, 0.37 * (q @ k[0]), rtol=0, atol=1e-14)


def test_zero_query_gives_mean_and_log_n():
    rng = _rng(4)
    for n in (1, 2, 7, 100):
        k = rng.standard_normal((n, 8))
        v = rng.standard_normal((n, 5))
        o, lse = attention_rows(np.zeros((2, 8)), k, v, 0.5)
        np.testing.assert_allclose(o, np.repeat(v.mean(axis=0, keepdims=True), 2, 0),
                                   rtol=0, atol=1e-14)
        np.testing.assert_allclose(lse, [math.log(n)] * 2, rtol=0, atol=1e-14)


def test_two_key_golden_fixture():
    vals = {}
    with open(os.path.join(GOLDEN, "two_key_closed_form.txt")) as fh:
        for line in fh:
            if line.strip() and not line.startswith("#"):
                name, *nums = line.split()
                vals[name] = np.array([float(x) for x in nums])
    o, lse = attention_rows(vals["q"][None], np.stack([vals["k0"], vals["k1"]]),
                            np.stack([vals["v0"], vals["v1"]]), float(vals["scale"][0]))
    np.testing.assert_allclose(o[0], vals["o"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse[0], vals["lse"][0], rtol=0, atol=1e-15)


def test_fork_decode_golden_fixture():
    """A shared paged prefix and two private suffixes, worked by hand
    (tests/golden/fork_decode_small.txt): pins the prefix/suffix concatenation,
    the page and slot lookup and the per-fork independence of the suffixes."""
    vals, kv = {}, []
    with open(os.path.join(GOLDEN, "fork_decode_small.txt")) as fh:
        for line in fh:
            if not line.strip() or line.startswith("#"):
                continue
            name, *nums = line.split()
            if name in ("k", "v"):
                kv.append((name, [float(x) for x in nums]))
            else:
                vals[name] = [float(x) for x in nums]
    B, P = int(vals["page_size"][0]), int(vals["num_pages"][0])
    pools = {n: np.full((P, 1, B, 2), wl.BF16_QNAN, dtype=np.uint16) for n in ("k", "v")}
    for name, (page, slot, x, y) in kv:
        pools[name][int(page), 0, int(slot)] = wl.round_to_bf16_bits(np.array([x, y]))
    q = wl.round_to_bf16_bits(np.array([vals["q"], vals["q"]])).reshape(2, 1, 2)
    w = dict(q=q, k_pages=pools["k"], v_pages=pools["v"],
             prefix_table=np.array(vals["prefix_table"], np.int32),
             prefix_bt_offsets=np.array([0, 1], np.int32),
             prefix_lens=np.array(vals["prefix_len"], np.int32),
             fork_offsets=np.array([0, 2], np.int32),
             suffix_table=np.array(vals["suffix_table"], np.int32),
             suffix_bt_offsets=np.array([0, 1, 2], np.int32),
             suffix_lens=np.array(vals["suffix_lens"], np.int32),
             num_traces=1, total_forks=2, num_pages=P, hq=1, hkv=1, dqk=2, dv=2,
             page_size=B, scale=math.log(vals["scale_log_of"][0]))
    o, lse = oracle.fork_attn_decode(w)
    np.testing.assert_allclose(o[0, 0], vals["o0"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(o[1, 0], vals["o1"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(lse[:, 0], [vals["lse0"][0], vals["lse1"][0]], rtol=0, atol=1e-14)
    assert abs(vals["lse0"][0] - math.log(7)) < 1e-15 and abs(vals["lse1"][0] - math.log(4)) < 1e-15


def test_empty_key_set():
    o, lse = attention_rows(np.ones((2, 4)), np.zeros((0, 4)), np.zeros((0, 3)), 1.0)
    assert np.array_equal(o, np.zeros((2, 3)))
    assert np.all(lse == -np.inf)


# ---------------------------------------------------------------- invariants
def test_score_shift_changes_only_lse():
    rng = _rng(5)
    q = rng.standard_normal((1, 12))
    k = rng.standard_normal((30, 12))
    v = rng.standard_normal((30, 6))
    scale, c = 0.3, 2.75
    # moving every key by c/(scale |q|^2) * q adds exactly c to every score
    k2 = k + (c / (scale * float(q[0] @ q[0]))) * q
    o1, l1 = attention_rows(q, k, v, scale)
    o2, l2 = attention_rows(q, k2, v, scale)
    np.testing.assert_allclose(o2, o1, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l2, l1 + c, rtol=0, atol=1e-12)


def test_key_order_does_not_matter():
    rng = _rng(6)
    q = rng.standard_normal((4, 10))
    k = rng.standard_normal((50, 10))
    v = rng.standard_normal((50, 7))
    perm = rng.permutation(50)
    o1, l1 = attention_rows(q, k, v, 0.4)
    o2, l2 = attention_rows(q, k[perm], v[perm], 0.4)
    np.testing.assert_allclose(o2, o1, rtol=0, atol=1e-13)
    np.testing.assert_allclose(l2, l1, rtol=0, atol=1e-13)


def test_large_scores_stay_finite():
    q = np.array([[1.0, 0.0]])
    k = np.array([[1000.0, 0.0], [999.0, 0.0]])
    v = np.array([[1.0], [0.0]])
    o, lse = attention_rows(q, k, v, 1.0)
    e = math.exp(-1.0)
    np.testing.assert_allclose(o[0, 0], 1.0 / (1.0 + e), rtol=1e-15)
    np.testing.assert_allclose(lse[0], 1000.0 + math.log1p(e), rtol=1e-15)
    # a spread of 800 nats: exp of an unshifted or min-shifted score overflows fp64
    k = np.array([[800.0, 0.0], [0.0, 0.0], [-5.0, 0.0]])
    v = np.array([[2.0], [7.0], [9.0]])
    o, lse = attention_rows(q, k, v, 1.0)
    np.testing.assert_allclose(o[0, 0], 2.0, rtol=1e-15)
    np.testing.assert_allclose(lse[0], 800.0, rtol=1e-15)


def test_against_scipy_softmax_and_logsumexp():
    rng = _rng(7)
    q = rng.standard_normal((5, 24))
    k = rng.standard_normal((77, 24))
    v = rng.standard_normal((77, 11))
    o, lse = attention_rows(q, k, v, 0.2)
    s = 0.2 * np.einsum("rd,nd->rn", q, k)
    np.testing.assert_allclose(lse, logsumexp(s, axis=1), rtol=0, atol=1e-12)
    np.testing.assert_allclose(o, softmax(s, axis=1) @ v, rtol=0, atol=1e-12)


# ---------------------------------------------------------------- merge algebra
def test_split_merge_equals_unsplit():
    rng = _rng(8)
    q = rng.standard_normal((6, 16))
    k = rng.standard_normal((40, 16)) * 2
    v = rng.standard_normal((40, 9))
    o, lse = attention_rows(q, k, v, 0.25)
    for cut in (0, 1, 17, 39, 40):
        oa, la = attention_rows(q, k[:cut], v[:cut], 0.25)
        ob, lb = attention_rows(q, k[cut:], v[cut:], 0.25)
        om, lm = lse_merge(oa, la, ob, lb)
        np.testing.assert_allclose(om, o, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lm, lse, rtol=0, atol=1e-12)
    # merging is order independent
    oa, la = attention_rows(q, k[:13], v[:13], 0.25)
    ob, lb = attention_rows(q, k[13:], v[13:], 0.25)
    o1, l1 = lse_merge(oa, la, ob, lb)
    o2, l2 = lse_merge(ob, lb, oa, la)
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-14)
    np.testing.assert_allclose(l1, l2, rtol=0, atol=1e-14)


def test_merge_with_empty_part_is_identity():
    rng = _rng(9)
    o = rng.standard_normal((3, 4))
    lse = rng.standard_normal(3)
    empty_o = np.full((3, 4), 123.0)     # must be ignored, whatever it holds
    empty_l = np.full(3, -np.inf)
    for args in ((o, lse, empty_o, empty_l), (empty_o, empty_l, o, lse)):
        om, lm = lse_merge(*args)
        np.testing.assert_allclose(om, o, rtol=0, atol=1e-15)
        np.testing.assert_allclose(lm, lse, rtol=0, atol=1e-15)
    om, lm = lse_merge(empty_o, empty_l, empty_o, empty_l)
    assert np.array_equal(om, np.zeros((3, 4))) and np.all(lm == -np.inf)


def test_merge_weights_by_normaliser():
    # parts with equal LSE average their outputs; a part 1 nat larger weighs e times more
    oa, ob = np.array([[1.0, 0.0]]), np.array([[0.0, 1.0]])
    om, lm = lse_merge(oa, np.array([0.5]), ob, np.array([1.5]))
    e = math.e
    np.testing.assert_allclose(om[0], [1 / (1 + e), e / (1 + e)], rtol=1e-15)
    np.testing.assert_allclose(lm[0], 1.5 + math.log1p(1 / e), rtol=1e-15)


# ---------------------------------------------------------------- whole workloads
def _tiny(**kw):
    base = dict(name="t", num_traces=2, prefix_len=(5, 37), forks=(1, 3), suffix_len=(0, 9),
                hq=6, hkv=2, dqk=8, dv=4, page_size=4)
    base.update(kw)
    return wl.WorkloadSpec(**base)


def _brute(w):
    """Pure-Python loops from the pool, straight from the definition."""
    nf, hq, g_size = w["total_forks"], w["hq"], w["hq"] // w["hkv"]
    B, dv = w["page_size"], w["dv"]
    o = np.zeros((nf, hq, dv))
    lse = np.zeros((nf, hq))

    def val(pool, page, g, slot, d):
        bits = int(pool[page, g, slot, d])
        return float(np.array([bits << 16], dtype=np.uint32).view(np.float32)[0])

    for t in range(w["num_traces"]):
        for f in range(w["fork_offsets"][t], w["fork_offsets"][t + 1]):
            toks = []
            pt = w["prefix_table"][w["prefix_bt_offsets"][t]:]
            for j in range(w["prefix_lens"][t]):
                toks.append((pt[j // B], j % B))
            st = w["suffix_table"][w["suffix_bt_offsets"][f]:]
            for j in range(w["suffix_lens"][f]):
                toks.append((st[j // B], j % B))
            for h in range(hq):
                g = h // g_size
                qrow = [float(np.array([int(x) << 16], dtype=np.uint32).view(np.float32)[0])
                        for x in w["q"][f, h]]
                if not toks:
                    lse[f, h] = -math.inf
                    continue
                s = [w["scale"] * math.fsum(qrow[d] * val(w["k_pages"], p, g, sl, d)
                                            for d in range(w["dqk"])) for p, sl in toks]
                z = math.fsum(math.exp(x) for x in s)
                lse[f, h] = math.log(z)
                vp = w["v_pages"]
                for d in range(dv):
                    o[f, h, d] = math.fsum(
                        math.exp(x - lse[f, h]) * (val(vp, p, g, sl, d) if vp is not None
                                                   else val(w["k_pages"], p, g, sl, d))
                        for x, (p, sl) in zip(s, toks))
    return o, lse


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_fork_decode_brute_force(seed):
    w = wl.make_workload(_tiny(), seed=seed)
    o, lse = oracle.fork_attn_decode(w)
    ob, lb = _brute(w)
    np.testing.assert_allclose(lse, lb, rtol=0, atol=1e-12)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
    assert np.all(np.isfinite(o))


def test_fork_decode_brute_force_latent_kv():
    w = wl.make_workload(_tiny(hq=4, hkv=1, dqk=10, dv=6, separate_v=False), seed=5)
    assert w["v_pages"] is None
    o, lse = oracle.fork_attn_decode(w)
    ob, lb = _brute(w)
    np.testing.assert_allclose(lse, lb, rtol=0, atol=1e-12)
    np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)


def test_latent_kv_equals_explicit_value_pool():
    w = wl.make_workload(_tiny(hq=4, hkv=1, dqk=10, dv=6, separate_v=False), seed=6)
    w2 = dict(w)
    w2["v_pages"] = np.ascontiguousarray(w["k_pages"][..., :6])
    o1, l1 = oracle.fork_attn_decode(w)
    o2, l2 = oracle.fork_attn_decode(w2)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


@pytest.mark.parametrize("name", ["tiny_p512_f4"])
def test_split_merge_equals_monolithic_workload(name):
    w = wl.make_workload(name)
    o, lse = oracle.fork_attn_decode(w)
    o2, l2 = oracle.fork_attn_split_merge(w)
    np.testing.assert_allclose(o2, o, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l2, lse, rtol=0, atol=1e-12)


def test_split_merge_with_empty_suffixes_and_prefixes():
    w = wl.make_workload(_tiny(prefix_len=(0, 9), suffix_len=(0, 3)), seed=11)
    assert (w["suffix_lens"] == 0).any() or (w["prefix_lens"] == 0).any()
    o, lse = oracle.fork_attn_decode(w)
    o2, l2 = oracle.fork_attn_split_merge(w)
    np.testing.assert_allclose(o2, o, rtol=0, atol=1e-12)
    np.testing.assert_allclose(l2, lse, rtol=0, atol=1e-12)


def test_page_placement_is_bit_invariant():
    w = wl.make_workload(_tiny(), seed=3)
    o1, l1 = oracle.fork_attn_decode(w)
    perm = _rng(12).permutation(w["num_pages"]).astype(np.int32)
    w2 = dict(w)
    for key in ("k_pages", "v_pages"):
        pool2 = np.empty_like(w[key])
        pool2[perm] = w[key]                 # physical page p moves to perm[p]
        w2[key] = pool2
    w2["prefix_table"] = perm[w["prefix_table"]]
    w2["suffix_table"] = perm[w["suffix_table"]]
    o2, l2 = oracle.fork_attn_decode(w2)
    assert np.array_equal(o1, o2) and np.array_equal(l1, l2)


def test_gqa_head_map_contiguous_groups():
    """Query head h reads kv head h // G: changing kv head 1 changes exactly heads G..2G-1."""
    w = wl.make_workload(_tiny(hq=6, hkv=3), seed=4)
    o1, _ = oracle.fork_attn_decode(w)
    w2 = dict(w)
    w2["k_pages"] = w["k_pages"].copy()
    w2["k_pages"][:, 1] = wl.bf16_normal(_rng(99), w["k_pages"][:, 1].shape)
    o2, _ = oracle.fork_attn_decode(w2)
    changed = np.any(o1 != o2, axis=(0, 2))
    assert changed.tolist() == [False, False, True, True, False, False]


def test_mha_special_case_matches_per_head_attention():
    """G = 1 is ordinary multi-head decode: head h over kv head h alone."""
    w = wl.make_workload(_tiny(hq=3, hkv=3), seed=8)
    o, lse = oracle.fork_attn_decode(w)
    f = w["total_forks"] - 1
    t = int(np.searchsorted(w["fork_offsets"], f, side="right") - 1)
    pt = w["prefix_table"][w["prefix_bt_offsets"][t]:w["prefix_bt_offsets"][t + 1]]
    st = w["suffix_table"][w["suffix_bt_offsets"][f]:w["suffix_bt_offsets"][f + 1]]
    for h in range(3):
        k = np.concatenate([oracle.gather_logical(w["k_pages"], pt, w["prefix_lens"][t], 4, h),
                            oracle.gather_logical(w["k_pages"], st, w["suffix_lens"][f], 4, h)])
        v = np.concatenate([oracle.gather_logical(w["v_pages"], pt, w["prefix_lens"][t], 4, h),
                            oracle.gather_logical(w["v_pages"], st, w["suffix_lens"][f], 4, h)])
        s = w["scale"] * (k @ bf16_bits_to_f64(w["q"][f, h]))
        np.testing.assert_allclose(lse[f, h], logsumexp(s), rtol=0, atol=1e-12)
        np.testing.assert_allclose(o[f, h], softmax(s) @ v, rtol=0, atol=1e-12)


def test_unused_slots_and_sentinels_are_never_read():
    w = wl.make_workload(_tiny(), seed=7)
    assert np.isnan(bf16_bits_to_f64(w["k_pages"][w["sentinel_ids"]])).all()
    o, lse = oracle.fork_attn_decode(w)
    assert np.all(np.isfinite(o)) and np.all(np.isfinite(lse))


def test_rows_entry_matches_full():
    w = wl.make_workload(_tiny(), seed=2)
    o, lse = oracle.fork_attn_decode(w)
    rows = [(w["total_forks"] - 1, 5), (0, 0), (0, 3)]
    ro, rl = oracle.fork_attn_decode_rows(w, rows)
    for i, (f, h) in enumerate(rows):
        np.testing.assert_allclose(ro[i], o[f, h], rtol=0, atol=1e-14)
        np.testing.assert_allclose(rl[i], lse[f, h], rtol=0, atol=1e-14)


# ----------------------------------------------------------------- decode-step append

def _read_fixture(name):
    vals = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if line and not line.startswith("#"):
            key, *rest = line.split()
            vals[key] = rest
    return vals


def test_append_golden_fixture():
    g = _read_fixture("append_small.txt")
    B = int(g["page_size"][0])
    lens = np.array([int(x) for x in g["lens"]], dtype=np.int32)
    offs = np.array([int(x) for x in g["offsets"]], dtype=np.int32)
    table = np.array([int(x) for x in g["table_before"]], dtype=np.int32)
    free = np.array([int(x) for x in g["free"]], dtype=np.int32)
    rows = [float(x) for x in g["new_row_values"]]
    pool = np.full((8, 1, B, 2), 0x7FC0, dtype=np.uint16)   # NaN everywhere
    k_new = wl.round_to_bf16_bits(np.array([[[r, r]] for r in rows], dtype=np.float32))
    k, v, t, taken = oracle.append_kv(pool, None, table, offs, lens, k_new, None, free, B)
    assert v is None
    assert t.tolist() == [int(x) for x in g["table_after"]]
    assert taken == int(g["taken"][0])
    written = [tuple(int(y) for y in w.split(":")) for w in g["written"]]
    for (page, head, slot), r in zip(written, rows):
        assert oracle.bf16_bits_to_f64(k[page, head, slot]).tolist() == [r, r]
    mask = np.ones(k.shape[:3], dtype=bool)
    for page, head, slot in written:
        mask[page, head, slot] = False
    assert np.array_equal(k[mask], pool[mask])          # nothing else touched
    assert table.tolist() == [int(x) for x in g["table_before"]]   # inputs not modified


def _python_sequence(pool, table, offs, f, n, B, head):
    """Pure-Python gather of the first n rows of fork f's paged sequence."""
    out = []
    for j in range(n):
        page = int(table[int(offs[f]) + j // B])
        out.append([int(x) for x in pool[page, head, j % B]])
    return out


@pytest.mark.parametrize("B", [1, 2, 16])
def test_append_grows_every_sequence_by_its_row(B):
    """Appending n steps one at a time gives, for every fork and head, the old
    sequence followed by the n new rows in order (pure-Python gather), with the
    free list consumed exactly when a fork crosses a page boundary."""
    rng = np.random.default_rng(B)
    F, H, W, steps = 5, 2, 3, 2 * B + 3
    lens0 = rng.integers(0, 3 * B, F).astype(np.int32)
    cap = -(-(lens0 + steps) // B)
    offs = np.concatenate([[0], np.cumsum(cap)]).astype(np.int32)
    used = -(-lens0 // B)
    n_pages = int(cap.sum()) + 4
    perm = rng.permutation(n_pages).astype(np.int32)
    table = np.full(int(cap.sum()), -1, dtype=np.int32)
    nxt = 0
    for f in range(F):
        table[offs[f]: offs[f] + used[f]] = perm[nxt: nxt + used[f]]
        nxt += int(used[f])
    free = perm[nxt:].copy()
    pool_k = rng.integers(0, 1 << 15, (n_pages, H, B, W)).astype(np.uint16)
    pool_v = rng.integers(0, 1 << 15, (n_pages, H, B, W)).astype(np.uint16)
    before = {f: [_python_sequence(pool_k, table, offs, f, int(lens0[f]), B, h) for h in range(H)]
              for f in range(F)}
    news = rng.integers(0, 1 << 15, (steps, F, H, 2, W)).astype(np.uint16)
    k, v, t, lens, fi = pool_k, pool_v, table, lens0.copy(), 0
    for s in range(steps):
        k, v, t, taken = oracle.append_kv(k, v, t, offs, lens, news[s, :, :, 0], news[s, :, :, 1],
                                          free[fi:], B)
        assert taken == int(np.sum(lens % B == 0))
        fi += taken
        lens = lens + 1
    for f in range(F):
        for h in range(H):
            seq_k = _python_sequence(k, t, offs, f, int(lens[f]), B, h)
            seq_v = _python_sequence(v, t, offs, f, int(lens[f]), B, h)
            assert seq_k[: lens0[f]] == before[f][h]
            assert seq_k[lens0[f]:] == [[int(x) for x in news[s, f, h, 0]] for s in range(steps)]
            assert seq_v[lens0[f]:] == [[int(x) for x in news[s, f, h, 1]] for s in range(steps)]
    assert fi == int(np.sum(cap - used))  # every fork filled its capacity exactly


def test_append_rejects_full_table_and_empty_free_list():
    pool = np.zeros((4, 1, 2, 2), dtype=np.uint16)
    row = np.zeros((1, 1, 2), dtype=np.uint16)
    with pytest.raises(ValueError):   # length 2 needs a second page; capacity is 1
        oracle.append_kv(pool, None, np.array([0], np.int32), np.array([0, 1], np.int32),
                         np.array([2], np.int32), row, None, np.array([3], np.int32), 2)
    with pytest.raises(ValueError):   # new page needed, free list empty
        oracle.append_kv(pool, None, np.array([-1], np.int32), np.array([0, 1], np.int32),
                         np.array([0], np.int32), row, None, np.array([], np.int32), 2)


# ----------------------------------------------------------------- prefix page pack / unpack

def test_pack_pages_hand_example():
    """Two pages (ids 2 then 0) of a 3-page pool, B = 2, one head, width 1:
    the buffer is K of page 2, K of page 0, V of page 2, V of page 0."""
    k = np.arange(6, dtype=np.uint16).reshape(3, 1, 2, 1)          # page p holds 2p, 2p+1
    v = (100 + np.arange(6, dtype=np.uint16)).reshape(3, 1, 2, 1)
    buf = oracle.pack_pages(k, v, [2, 0])
    assert buf.tolist() == [4, 5, 0, 1, 104, 105, 100, 101]
    assert oracle.pack_pages(k, None, [1]).tolist() == [2, 3]


@pytest.mark.parametrize("latent", [False, True])
def test_pack_then_unpack_moves_a_sequence(latent):
    """Packing a sequence and unpacking it under a new table gives, by a
    pure-Python gather, the same logical rows at the new pages; pages outside
    the new table keep their contents."""
    rng = np.random.default_rng(5)
    P, H, B, W = 12, 2, 4, 3
    k = rng.integers(0, 1 << 15, (P, H, B, W)).astype(np.uint16)
    v = None if latent else rng.integers(0, 1 << 15, (P, H, B, W + 1)).astype(np.uint16)
    perm = rng.permutation(P)
    old, new = perm[:5], perm[5:10]
    buf = oracle.pack_pages(k, v, old)
    k2, v2 = oracle.unpack_pages(k, v, new, buf)
    n = len(old) * B
    for h in range(H):
        assert _python_sequence(k2, new, [0], 0, n, B, h) == _python_sequence(k, old, [0], 0, n, B, h)
        if v is not None:
            assert (_python_sequence(v2, new, [0], 0, n, B, h)
                    == _python_sequence(v, old, [0], 0, n, B, h))
    rest = np.setdiff1d(np.arange(P), new)
    assert np.array_equal(k2[rest], k[rest])
    if v is not None:
        assert np.array_equal(v2[rest], v[rest])


# ----------------------------------------------------------------- fork prefill

def test_prefill_with_one_token_chunks_is_decode():
    """A chunk of one token per fork is the decode of that fork's last token."""
    w = wl.make_workload(_tiny(seed=3))
    pf = wl.make_prefill(w, 1)
    o, lse = oracle.fork_prefill(w, pf["chunk_lens"], pf["q_rows"])
    has = pf["chunk_lens"] > 0
    w_dec = dict(w, q=np.zeros_like(w["q"]))
    w_dec["q"][has] = pf["q_rows"]
    o_d, lse_d = oracle.fork_attn_decode(w_dec)
    assert np.allclose(o, o_d[has], rtol=0, atol=1e-14)
    assert np.allclose(lse, lse_d[has], rtol=0, atol=1e-14)


@pytest.mark.parametrize("seed", [0, 1])
def test_prefill_is_causal_brute_force(seed):
    """Row (f, j) equals the pure-Python brute force over the prefix and the
    fork's first S_f - c_f + j + 1 suffix tokens, with the row's own query."""
    w = wl.make_workload(_tiny(seed=seed))
    pf = wl.make_prefill(w, 5)
    o, lse = oracle.fork_prefill(w, pf["chunk_lens"], pf["q_rows"])
    r = 0
    for f in range(w["total_forks"]):
        c = int(pf["chunk_lens"][f])
        for j in range(c):
            lens = w["suffix_lens"].copy()
            lens[f] = w["suffix_lens"][f] - c + j + 1
            q = w["q"].copy()
            q[f] = pf["q_rows"][r]
            ob, lb = _brute(dict(w, suffix_lens=lens, q=q))
            assert np.allclose(o[r], ob[f], rtol=0, atol=1e-12)
            assert np.allclose(lse[r], lb[f], rtol=0, atol=1e-12)
            r += 1
    assert r == pf["rows"]


# ----------------------------------------------------------------- nested-prefix cascade

@pytest.mark.parametrize("points,forks", [((8,), (3,)), ((8, 20, 28), (2, 1, 3)),
                                          ((4, 12), (1, 2))])
def test_cascade_equals_flat_decode(points, forks):
    """Forks that attend to a chain of shared segments get the decode result of
    one flat prefix per fork event (the segments' pages concatenated)."""
    w = wl.make_cascade(points, forks, suffix_len=(0, 9), hq=6, hkv=2, dqk=8, dv=4,
                        page_size=4, seed=len(points))
    o, lse = oracle.fork_cascade_decode(w)
    o_f, lse_f = oracle.fork_attn_decode(w["flat"])
    assert np.allclose(o, o_f, rtol=0, atol=1e-13)
    assert np.allclose(lse[np.isfinite(lse)], lse_f[np.isfinite(lse_f)], rtol=0, atol=1e-13)
    assert np.array_equal(np.isfinite(lse), np.isfinite(lse_f))


def test_cascade_brute_force():
    w = wl.make_cascade((8, 16), (2, 2), suffix_len=(1, 6), hq=4, hkv=2, dqk=8, dv=8,
                        page_size=4, seed=1)
    o, lse = oracle.fork_cascade_decode(w)
    ob, lb = _brute(w["flat"])
    assert np.allclose(o, ob, rtol=0, atol=1e-12)
    assert np.allclose(lse, lb, rtol=0, atol=1e-12)
