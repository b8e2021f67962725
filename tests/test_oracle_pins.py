"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a value
worked by hand from the paper's equations (tests/golden/), a closed form, an
invariant, a special case that reduces to a library routine, or brute force.
"""
import itertools
import math
import os

import numpy as np
import pytest
import torch

from oracle import mpcache_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            out.setdefault(key, []).append([float(v) for v in vals])
    return out


# --------------------------------------------------------- worked examples --

def test_similarity_worked_example():
    g = _golden("eq1_eq2_eq3_cluster_similarity.txt")
    q = np.array(g["q"][0])
    keys = np.array(g["k"])
    lev = O.cluster_pyramid(keys, 3, (), 0.6)[0]
    assert np.array_equal(lev.r_max[0], g["r_max"][0])
    assert np.array_equal(lev.r_min[0], g["r_min"][0])
    assert np.allclose(lev.rep[0], g["rep_alpha_0.6"][0], atol=1e-15)
    assert O.sim_max_dot(q, keys) == g["max_dot"][0][0]
    assert O.sim_bound(q, lev.r_max[0], lev.r_min[0]) == g["bound"][0][0]
    for a in ("0.6", "1.0", "0.0"):
        want = g["linear_alpha_" + a][0][0]
        assert abs(O.sim_linear(q, lev.r_max[0], lev.r_min[0], float(a)) - want) < 1e-14
    assert abs(O.sim_average(q, keys) - g["average"][0][0]) < 1e-15


def test_static_window_worked_example():
    g = _golden("static_window_scores.txt")
    k = np.array(g["keys"][0])[:, None]
    qw = np.array(g["queries"][0])[None, :, None]          # [G=1][w=2][d=1]
    score = O.accumulated_attention(qw, k, scale=1.0)
    assert np.allclose(score, g["score"][0], atol=1e-12)
    assert list(O.static_evict(score, 2)) == [int(x) for x in g["keep2"][0]]
    assert list(O.static_evict(score, 1)) == [int(x) for x in g["keep1"][0]]
    assert O.window_length(3, window_ppm=600_000) == 2   # ceil(1.8)


def test_hierarchical_worked_example():
    g = _golden("hierarchical_selection.txt")
    keys = np.array(g["keys"][0])[:, None]
    levels = O.cluster_pyramid(keys, 1, (2,), 0.6)
    assert np.allclose(levels[1].rep[:, 0], g["parent_rep"][0], atol=1e-15)
    q = np.ones((1, 1))
    hier = O.hierarchical_select(q, levels, (2,), (250_000, 500_000))
    assert list(hier) == [int(x) for x in g["hierarchical"][0]]
    flat = O.hierarchical_select(q, levels[:1], (), (250_000,))
    assert list(flat) == [int(x) for x in g["flat"][0]]


def test_table5_ratio_semantics():
    """Table 5: coarse x fine ratio = 0.2.  With the fine ratio read as a share
    of the coarse level's survivors, the oracle keeps ~20% of the finest
    clusters overall and ~fine_ratio of the candidates."""
    rng = np.random.default_rng(5)
    with open(os.path.join(GOLDEN, "table5_hierarchy_ratios.txt")) as f:
        rows = [list(map(float, l.split())) for l in f if l.strip() and not l.startswith("#")]
    assert len(rows) == 8
    for cs, rc, fs, rf in rows:
        assert abs(rc * rf - 0.2) < 0.01
        f = int(cs // fs)
        n_fine = 256
        keys = rng.standard_normal((n_fine * int(fs), 8))
        levels = O.cluster_pyramid(keys, int(fs), (f,), 0.6)
        q = rng.standard_normal((1, 8))
        keep = (round(rc * rf * 1e6), round(rc * 1e6))
        sel = O.hierarchical_select(q, levels, (f,), keep)
        n_cand = f * O.selected_count(len(levels[1].rep), keep[1], len(levels[1].rep))
        # the printed fine ratio is 0.2 / coarse ratio to two digits
        assert abs(rf - 0.2 / rc) < 0.006
        assert abs(len(sel) / n_fine - 0.2) < 0.01
        # both counts are ceilings: up to one parent (f candidates) and one
        # cluster of rounding
        assert abs(len(sel) / n_cand - 0.2 / rc) < (f + 1.0) / n_cand


# ------------------------------------------------------------ counts -------

def test_counts_and_rules():
    assert O.window_length(512) == 103            # ceil(0.2 * 512)
    assert O.window_length(2048) == 410
    assert O.window_length(8192) == 1639
    assert O.window_length(24_576) == 4916        # 24k is not "longer than 24k"
    assert O.window_length(32_768) == 3277        # 10% above 24k tokens
    assert O.window_length(1000) == 200           # exact integer arithmetic
    assert O.kept_count(2048, 500_000) == 1024
    assert O.kept_count(32_768, 250_000) == 8192
    assert O.kept_count(5, 1) == 1
    assert O.kept_count(7, 1_000_000) == 7
    assert O.selected_count(512, 50_000, 128) == 26
    assert O.selected_count(64, 250_000, 32) == 16
    assert O.selected_count(8, 500_000, 8) == 4
    assert O.selected_count(0, 500_000, 0) == 0
    assert O.selected_count(10, 900_000, 3) == 3  # clamped to candidates
    assert O.level_keep_fractions(50_000, 3) == [50_000, 250_000, 500_000]
    assert O.level_keep_fractions(125_000, 2) == [125_000, 500_000]
    assert O.level_keep_fractions(1_000_000, 2) == [1_000_000, 1_000_000]
    assert O.level_keep_fractions(250_000, 1) == [250_000]
    # sharing: first two layers lead themselves; groups of m after them
    assert [O.leader_of(l, 2) for l in range(8)] == [0, 1, 2, 2, 4, 4, 6, 6]
    assert [O.leader_of(l, 4) for l in range(11)] == [0, 1, 2, 2, 2, 2, 6, 6, 6, 6, 10]
    assert len({O.leader_of(l, 2) for l in range(32)}) == 17
    assert len({O.leader_of(l, 4) for l in range(32)}) == 10
    assert [O.leader_of(l, 1) for l in range(4)] == [0, 1, 2, 3]


# ---------------------------------------------------------------- P1 -------

def _dense_decode(q, K, V, scale):
    """Dense decode attention through torch's SDPA in float64."""
    qt = torch.from_numpy(q)[None, None, None]            # [1,1,1,d]
    kt = torch.from_numpy(K)[None, None]
    vt = torch.from_numpy(V)[None, None]
    return torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, scale=scale)[0, 0, 0].numpy()


@pytest.mark.parametrize("G", [1, 2])
def test_p1_keep_all_equals_dense(G):
    rng = np.random.default_rng(11 + G)
    Hkv, d, T, E, s = 2, 16, 37, 5, 4
    Hq = Hkv * G
    K = rng.standard_normal((Hkv, T, d)); V = rng.standard_normal((Hkv, T, d))
    R = T
    Qw = rng.standard_normal((Hq, R, d))
    q = rng.standard_normal((E, Hq, d)); kn = rng.standard_normal((E, Hkv, d))
    vn = rng.standard_normal((E, Hkv, d))
    p = O.Params(keep_ppm=O.PPM, cluster_size=s, fanouts=(2,), level_keep_ppm=(O.PPM, O.PPM),
                 share_every=1)
    res = O.run(lambda l, b: K, lambda l, b: V, lambda l, b: Qw, lambda e, l, b: q[e],
                lambda e, l, b: kn[e], lambda e, l, b: vn[e], [T], p, steps=E, layers=[0])
    scale = 1 / math.sqrt(d)
    for e in range(E):
        for h in range(Hkv):
            Kf = np.vstack([K[h], kn[:e + 1, h]])
            Vf = np.vstack([V[h], vn[:e + 1, h]])
            for g in range(G):
                want = _dense_decode(q[e, h * G + g], Kf, Vf, scale)
                assert np.abs(res.out[(e, 0, 0)][h * G + g] - want).max() < 1e-12


# ---------------------------------------------------------------- P2 -------

@pytest.mark.parametrize("T,w,G", [(50, 10, 1), (130, 26, 4), (9, 9, 2)])
def test_p2_window_mass(T, w, G):
    rng = np.random.default_rng(T)
    d = 8
    qw = rng.standard_normal((G, w, d)) * 2
    k = rng.standard_normal((T, d)) * 2
    score = O.accumulated_attention(qw, k, 1 / math.sqrt(d))
    assert abs(score.sum() - w * G) < 1e-9 * w * G
    assert (score >= 0).all()
    # a key after every window row's position is never attended: only the
    # last row sees key T-1, only rows >= i see key T-w+i
    assert score[T - 1] <= G + 1e-12


def test_p2_causal_mask_brute_force():
    """Each window row's softmax, taken over exactly the causal prefix by a
    per-row python loop, summed per column."""
    rng = np.random.default_rng(3)
    T, w, d = 12, 5, 4
    qw = rng.standard_normal((1, w, d)); k = rng.standard_normal((T, d))
    want = np.zeros(T)
    for i in range(w):
        pos = T - w + i
        logits = [float(np.dot(qw[0, i], k[j])) / 2.0 for j in range(pos + 1)]
        mx = max(logits)
        ex = [math.exp(x - mx) for x in logits]
        z = sum(ex)
        for j in range(pos + 1):
            want[j] += ex[j] / z
    assert np.allclose(O.accumulated_attention(qw, k, 0.5), want, atol=1e-13)


# ---------------------------------------------------------------- P3 -------

@pytest.mark.parametrize("N,s,fan", [(64, 16, (4,)), (70, 16, (4,)), (200, 4, (3, 2)), (15, 16, (4,)),
                                     (512, 16, (8, 8))])
def test_p3_partition(N, s, fan):
    rng = np.random.default_rng(N)
    keys = rng.standard_normal((N, 6))
    levels = O.cluster_pyramid(keys, s, fan, 0.6)
    n_full = N // s
    covered = np.arange(n_full * s)
    for lvl, lev in enumerate(levels):
        allm = np.concatenate(lev.members) if lev.members else np.zeros(0, int)
        assert np.array_equal(np.sort(allm), covered)          # disjoint + covering
        if lvl == 0:
            assert all(len(m) == s for m in lev.members)
        if lvl > 0:
            f = fan[lvl - 1]
            assert len(lev.members) == -(-len(levels[lvl - 1].members) // f)
        for c, m in enumerate(lev.members):
            assert np.array_equal(lev.r_max[c], keys[m].max(0))
            assert np.array_equal(lev.r_min[c], keys[m].min(0))
        # coarse summaries equal the element-wise max/min of their children
        if lvl > 0:
            f = fan[lvl - 1]
            ch = levels[lvl - 1]
            for p in range(len(lev.members)):
                kids = range(p * f, min((p + 1) * f, len(ch.members)))
                assert np.array_equal(lev.r_max[p], np.max([ch.r_max[c] for c in kids], 0))
                assert np.array_equal(lev.r_min[p], np.min([ch.r_min[c] for c in kids], 0))
    # attended set = selected clusters + tail, disjoint
    sel = np.array([0, 2]) if n_full >= 3 else np.arange(n_full)
    toks = O.attended_tokens(N, s, sel)
    assert len(set(toks.tolist())) == len(toks)
    assert toks.max() == N   # the token appended at this step


# ---------------------------------------------------------------- P4 -------

@pytest.mark.parametrize("G,k_ppm", [(1, 250_000), (4, 100_000), (2, 1_000_000)])
def test_p4_token_wise_equals_topk(G, k_ppm):
    """s = 1 (one token per cluster, no hierarchy): rep = k, so selection is
    the exact token top-k of (sum_g q_g) . k, computed here by torch.topk."""
    rng = np.random.default_rng(G)
    N, d = 97, 16
    keys = rng.standard_normal((N, d))
    qg = rng.standard_normal((G, d))
    levels = O.cluster_pyramid(keys, 1, (), 0.6)
    assert np.allclose(levels[0].rep, keys, rtol=1e-15, atol=0)   # 0.6 k + 0.4 k
    sel = O.hierarchical_select(qg, levels, (), (k_ppm,))
    k = O.selected_count(N, k_ppm, N)
    scores = torch.from_numpy(keys) @ torch.from_numpy(qg).sum(0)
    want = np.sort(torch.topk(scores, k).indices.numpy())
    assert np.array_equal(sel, want)
    # a one-token cluster's mean is its key: the average baseline agrees
    assert np.array_equal(levels[0].mean, keys)
    assert np.array_equal(O.hierarchical_select(qg, levels, (), (k_ppm,), metric="mean"), want)


# ---------------------------------------------------------------- P5 / P6 --

def test_p5_identical_tokens():
    rng = np.random.default_rng(5)
    key = rng.standard_normal(32)
    keys = np.tile(key, (16, 1))
    q = rng.standard_normal(32)
    lev = O.cluster_pyramid(keys, 16, (), 0.6)[0]
    assert np.array_equal(lev.r_max[0], lev.r_min[0])
    assert abs(float(lev.rep[0] @ q) - float(key @ q)) < 1e-12
    assert abs(O.sim_bound(q, lev.r_max[0], lev.r_min[0]) - O.sim_max_dot(q, keys)) < 1e-12


def test_p6_bound_and_linearisation():
    rng = np.random.default_rng(6)
    for _ in range(200):
        s, d = rng.integers(1, 20), rng.integers(1, 40)
        keys = rng.standard_normal((s, d)) * rng.uniform(0.1, 5)
        q = rng.standard_normal(d)
        lev = O.cluster_pyramid(keys, s, (), 0.6)[0]
        rmax, rmin = lev.r_max[0], lev.r_min[0]
        bound = O.sim_bound(q, rmax, rmin)
        assert bound >= O.sim_max_dot(q, keys) - 1e-9          # Eq. 1 <= Eq. 2
        # Eq. 3 reordering: linearised sum == q . rep
        for a in (0.0, 0.3, 0.6, 1.0):
            rep = a * rmax + (1 - a) * rmin
            assert abs(O.sim_linear(q, rmax, rmin, a) - float(q @ rep)) < 1e-9
        # alpha = 1 with q >= 0 reaches the bound exactly
        qp = np.abs(q)
        assert abs(O.sim_linear(qp, rmax, rmin, 1.0) - O.sim_bound(qp, rmax, rmin)) < 1e-9
        # the linearised value never exceeds the bound
        assert O.sim_linear(q, rmax, rmin, 0.6) <= bound + 1e-9


# ---------------------------------------------------------------- P7 -------

def _brute_select(qsum, keys, s, fanouts, level_keep, metric="eq3", qg=None, frac_bits=18):
    """Coarse-to-fine selection by exhaustive search: at every level, try every
    subset of the candidates of the required size and keep the one with the
    largest total similarity (ties: the lexicographically smallest id list).
    Summaries are recomputed from the member tokens with explicit loops; the
    similarity is Eq. 3 (alpha 0.6), the Eq. 2 bound, the mean key, or Eq. 3
    in fixed point with Python integers (round() is half to even, // floors),
    channel by channel."""
    N, d = keys.shape
    one = 1 << frac_bits
    n_full = N // s
    sizes = [s]
    for f in fanouts:
        sizes.append(sizes[-1] * f)

    def members(lvl, c):
        lo = c * sizes[lvl]
        return list(range(lo, min(lo + sizes[lvl], n_full * s)))

    def sim(lvl, c):
        toks = members(lvl, c)
        total = 0.0
        for i in range(d):
            mx = max(keys[t][i] for t in toks)
            mn = min(keys[t][i] for t in toks)
            if metric == "eq3":
                total += qsum[i] * (0.6 * mx + 0.4 * mn)
            elif metric == "bound":
                total += max(qsum[i] * mx, qsum[i] * mn)
            elif metric == "fxp":
                qi = sum(round(float(qg[g][i]) * one) for g in range(len(qg)))
                rep = round(0.6 * one) * round(float(mx) * one) // one + \
                    round(0.4 * one) * round(float(mn) * one) // one
                total += qi * rep
            else:
                acc = 0.0
                for t in toks:
                    acc += keys[t][i]
                total += qsum[i] * acc / len(toks)
        if metric == "fxp":
            return float(min(max(total // one, -(1 << 31)), (1 << 31) - 1))
        return total

    n_level = [n_full]
    for f in fanouts:
        n_level.append(-(-n_level[-1] // f))
    cand = list(range(n_level[-1]))
    chosen = []
    for lvl in range(len(sizes) - 1, -1, -1):
        k = O.selected_count(n_level[lvl], level_keep[lvl], len(cand))
        best, best_val = None, None
        for sub in itertools.combinations(cand, k):
            val = sum(sim(lvl, c) for c in sub)
            if best is None or val > best_val + 1e-12:
                best, best_val = list(sub), val
        chosen = best
        if lvl > 0:
            f = fanouts[lvl - 1]
            cand = [c for p in chosen for c in range(p * f, min((p + 1) * f, n_level[lvl - 1]))]
    return chosen


@pytest.mark.parametrize("metric", ["eq3", "bound", "mean", "fxp"])
@pytest.mark.parametrize("seed", range(6))
def test_p7_brute_force_tiny(seed, metric):
    rng = np.random.default_rng(100 + seed)
    s = int(rng.choice([2, 4]))
    fan = [(), (2,), (3,), (2, 2)][seed % 4]
    N = int(rng.integers(s * 3, 64))
    d, G = 5, int(rng.choice([1, 3]))
    keys = rng.standard_normal((N, d))
    qg = rng.standard_normal((G, d))
    keep = O.level_keep_fractions(int(rng.choice([250_000, 400_000])), 1 + len(fan))
    levels = O.cluster_pyramid(keys, s, fan, 0.6)
    # few fractional bits make equal fixed-point scores (the tie rule) likely
    fb = (3, 6, 18)[seed % 3]
    got = O.hierarchical_select(qg, levels, fan, keep, metric=metric, frac_bits=fb)
    want = _brute_select(qg.sum(0), keys, s, fan, keep, metric, qg=qg, frac_bits=fb)
    assert list(got) == sorted(want)


# ------------------------------------------------ fixed-point emulation ----

def test_fxp_worked_example():
    g = _golden("fxp_eq3_ring_worked_example.txt")
    got = O.sim_fxp(np.array(g["a_q"]), np.array(g["a_r_max"]), np.array(g["a_r_min"]),
                    g["a_alpha"][0][0], int(g["a_f"][0][0]))
    assert got.tolist() == [int(g["a_sim"][0][0])]
    got = O.sim_fxp(np.array(g["b_q"]), np.array(g["b_r_max"]), np.array(g["b_r_min"]),
                    g["b_alpha"][0][0], int(g["b_f"][0][0]))
    assert got.tolist() == [int(g["b_sim"][0][0])]
    assert O.fxp_encode(g["enc_f3_in"][0], 3).tolist() == [int(v) for v in g["enc_f3_out"][0]]


@pytest.mark.parametrize("seed", range(4))
def test_fxp_exact_on_dyadic_inputs(seed):
    # values on a 2^-4 grid, alpha = 3/4: every encoding and every truncation
    # is exact at f = 16, so the ring result is Eq. 3 itself, computed here
    # with exact rationals from the definition
    from fractions import Fraction as F
    rng = np.random.default_rng(700 + seed)
    G, d, C = 3, 8, 5
    qg = rng.integers(-40, 41, (G, d)) / 16.0
    rmin = rng.integers(-60, 20, (C, d)) / 16.0
    rmax = rmin + rng.integers(0, 50, (C, d)) / 16.0
    got = O.sim_fxp(qg, rmax, rmin, 0.75, 16)
    for c in range(C):
        exact = sum(F(float(qg[gg, i])) * (F(3, 4) * F(float(rmax[c, i])) + F(1, 4) * F(float(rmin[c, i])))
                    for gg in range(G) for i in range(d))
        assert F(int(got[c]), 1 << 16) == exact


def _fxp_bound(qg, r_max, r_min, fb):
    """Rounding bound of the fixed-point Eq. 3 per cluster (derivation below)."""
    G = len(qg)
    q = np.asarray(qg).sum(0)
    u = 2.0 ** -fb
    e = G * u / 2
    E = u / 2 * (np.abs(r_max) + np.abs(r_min)) + u / 2 * (1 + u) + 2 * u
    rep_abs = np.maximum(np.abs(r_max), np.abs(r_min))
    return (e * rep_abs + np.abs(q) * E + e * E).sum(axis=1) + u


@pytest.mark.parametrize("fb", [6, 10, 18])
def test_fxp_error_within_rounding_bound(fb):
    # Encodings are off by at most u/2 (u = 2^-f), each truncation by less
    # than u.  With q' = q + e (|e_i| <= G u/2) and rep' = rep + E
    # (|E_i| <= u/2 (|r_max_i| + |r_min_i|) + u/2 (1 + u) + 2u):
    #   |sim' - sim| <= sum_i (|e_i||rep_i| + |q_i||E_i| + |e_i||E_i|) + u
    rng = np.random.default_rng(800 + fb)
    G, d, C, a = 4, 128, 64, 0.6
    qg = rng.standard_normal((G, d))
    keys = rng.standard_normal((C * 16, d)) * np.where(np.arange(d) < 4, 8.0, 1.0)
    lev = O.cluster_pyramid(keys, 16, (), a)[0]
    got = O.sim_fxp(qg, lev.r_max, lev.r_min, a, fb) * 2.0 ** -fb
    exact = lev.rep @ qg.sum(0)
    bound = _fxp_bound(qg, lev.r_max, lev.r_min, fb)  # |rep_i| <= max(|r_max_i|, |r_min_i|)
    err = np.abs(got - exact)
    assert np.all(err <= bound * (1 + 1e-9))
    assert err.max() > 0  # the rounding is live
    assert err.max() > bound.max() / 200  # and the bound not vacuous


def test_fxp_ring_wraps_like_two_complement_int64():
    # f = 24 and values near 2^9: products of encodings near 2^66 leave the
    # int64 range; the ring arithmetic must equal Python big integers reduced
    # modulo 2^64 (two's complement), with floor division for truncation
    rng = np.random.default_rng(31)
    G, d, C, f, a = 3, 16, 6, 24, 0.6
    qg = rng.uniform(-600, 600, (G, d))
    rmin = rng.uniform(-600, 0, (C, d))
    rmax = rmin + rng.uniform(0, 600, (C, d))
    M = 1 << 64

    def wrap(v):
        v %= M
        return v - M if v >= 1 << 63 else v

    one = 1 << f
    q = [wrap(sum(round(float(qg[g, i]) * one) for g in range(G))) for i in range(d)]
    ea, eb = round(a * one), round((1 - a) * one)
    want = []
    wrapped = False
    for c in range(C):
        rep = [wrap(wrap(ea * round(float(rmax[c, i]) * one)) // one + wrap(eb * round(float(rmin[c, i]) * one)) // one)
               for i in range(d)]
        full = sum(q[i] * rep[i] for i in range(d))
        wrapped |= abs(full) >= 1 << 63
        want.append(min(max(wrap(full) // one, -(1 << 31)), (1 << 31) - 1))
    assert wrapped  # the case exercises the wrap
    assert O.sim_fxp(qg, rmax, rmin, a, f).tolist() == want


def test_fxp_saturates_to_int32():
    # scores beyond the int32 range of the ranking key saturate (equal keys
    # then rank the lower id first)
    q = np.full((1, 4), 100.0)
    r = np.full((3, 4), 100.0)
    got = O.sim_fxp(q, r, -r, 1.0, 18)
    assert got.tolist() == [(1 << 31) - 1] * 3
    assert O.sim_fxp(q, -r, -r, 1.0, 18).tolist() == [-(1 << 31)] * 3


def test_fxp_ranking_matches_float_away_from_ties():
    # where every cut of the float selection has a margin above twice the
    # rounding bound, the fixed-point selection keeps the same clusters
    n_clear = 0
    for seed in range(8):
        rng = np.random.default_rng(900 + seed)
        G, d = 4, 32
        keys = rng.standard_normal((2048, d))
        qg = rng.standard_normal((G, d))
        fan = (4, 4)
        keep = O.level_keep_fractions(100_000, 3)
        levels = O.cluster_pyramid(keys, 8, fan, 0.6)
        trace = []
        want = O.hierarchical_select(qg, levels, fan, keep, trace=trace)
        got = O.hierarchical_select(qg, levels, fan, keep, metric="fxp", frac_bits=18)
        clear = True
        for lvl, (cand, sim, k) in zip(range(len(levels) - 1, -1, -1), trace):
            srt = np.sort(sim)[::-1]
            band = _fxp_bound(qg, levels[lvl].r_max[cand], levels[lvl].r_min[cand], 18).max()
            clear &= bool(k >= len(srt) or srt[k - 1] - srt[k] > 2 * band)
        if clear:
            n_clear += 1
            assert np.array_equal(got, want), seed
    assert n_clear >= 6  # the comparison is live


@pytest.mark.parametrize("seed", range(4))
def test_bound_equals_eq3_at_alpha_one_for_nonnegative_queries(seed):
    # Eq. 2's max(q r_max, q r_min) is q r_max when q >= 0, which is Eq. 3 at
    # alpha = 1: the two metrics must select the same clusters
    rng = np.random.default_rng(300 + seed)
    keys = rng.standard_normal((400, 16))
    qg = np.abs(rng.standard_normal((2, 16)))
    fan = (4, 2)
    keep = O.level_keep_fractions(150_000, 3)
    levels = O.cluster_pyramid(keys, 4, fan, 1.0)
    a = O.hierarchical_select(qg, levels, fan, keep, metric="bound")
    b = O.hierarchical_select(qg, levels, fan, keep, metric="eq3")
    assert np.array_equal(a, b)
    # and with mixed-sign queries the two generally differ (the test is live)
    qm = rng.standard_normal((2, 16))
    diff = sum(not np.array_equal(O.hierarchical_select(qm * (j + 1) + j, levels, fan, keep, metric="bound"),
                                  O.hierarchical_select(qm * (j + 1) + j, levels, fan, keep, metric="eq3"))
               for j in range(4))
    assert diff >= 1


# ---------------------------------------------------------------- P8 -------

def test_p8_coarse_keep_all_equals_flat():
    rng = np.random.default_rng(8)
    keys = rng.standard_normal((16 * 40, 12))
    qg = rng.standard_normal((2, 12))
    flat = O.hierarchical_select(qg, O.cluster_pyramid(keys, 16, (), 0.6), (), (150_000,))
    for fan in ((4,), (3, 2), (8,)):
        lev = O.cluster_pyramid(keys, 16, fan, 0.6)
        keep = [150_000] + [O.PPM] * len(fan)
        assert np.array_equal(O.hierarchical_select(qg, lev, fan, keep), flat)


# ---------------------------------------------------------------- P9 -------

def _tiny_run(L, m, E=3, G=1, T=40, s=4, seed=9):
    rng = np.random.default_rng(seed)
    Hkv, d = 2, 8
    Hq = Hkv * G
    K = rng.standard_normal((L, Hkv, T, d)); V = rng.standard_normal((L, Hkv, T, d))
    Qw = rng.standard_normal((L, Hq, T, d))
    q = rng.standard_normal((E, L, Hq, d)); kn = rng.standard_normal((E, L, Hkv, d))
    vn = rng.standard_normal((E, L, Hkv, d))
    p = O.Params(keep_ppm=500_000, cluster_size=s, fanouts=(2,), level_keep_ppm=(250_000, 500_000),
                 share_every=m)
    return O.run(lambda l, b: K[l], lambda l, b: V[l], lambda l, b: Qw[l],
                 lambda e, l, b: q[e, l], lambda e, l, b: kn[e, l], lambda e, l, b: vn[e, l],
                 [T], p, steps=E, layers=list(range(L)))


def test_p9_sharing():
    L = 7
    solo = _tiny_run(L, 1)
    for l in range(L):
        assert (0, l, 0, 0) in solo.selected
    shared = _tiny_run(L, 2)
    for e in range(3):
        for l in range(L):
            lead = O.leader_of(l, 2)
            for h in range(2):
                assert np.array_equal(shared.selected[(e, l, 0, h)], shared.selected[(e, lead, 0, h)])
                assert np.array_equal(shared.kept[(l, 0, h)], shared.kept[(lead, 0, h)])
    # leaders are computed from their own inputs: same as the unshared run
    for l in (0, 1, 2, 4, 6):
        for h in range(2):
            assert np.array_equal(shared.selected[(0, l, 0, h)], solo.selected[(0, l, 0, h)])


# ---------------------------------------------------------------- P10 ------

@pytest.mark.slow
def test_p10_sink_token_kept_c1():
    """The GPT-2-small workload's sink (key 0 scaled by 4 under the iid rule)
    draws enough window attention that static eviction keeps it in every
    head (a sanity check of the recipe and of the scoring, not a parity pin)."""
    from paper_2501_06807_gb300 import synth
    from tests import helpers as H
    w = synth.C1
    x = synth.generate(w, H.window_rows_for(w), decode_steps=0)
    res = H.oracle_run(x, 0, [0])
    for h in range(w.n_kv_heads):
        kept = res.kept[(0, 0, h)]
        assert 0 in kept, h
        sc = res.scores[(0, 0, h)]
        assert sc[0] > np.sort(sc)[len(sc) // 2] * 4   # far above the median token


def test_p10_needles_survive_c5_shape():
    """The 32k-token needle workload at full size (layer 0, two kv heads,
    8 decode steps): every planted needle token is kept by static eviction and
    attended at every decode step (inside a selected cluster or the tail).
    At reduced lengths the coarsest level has too few nodes for a passage that
    straddles two of them, so the check needs the real shape."""
    from paper_2501_06807_gb300 import synth
    w = synth.C5.replace(n_layers=1, decode_steps=8)
    T = w.prompt_len
    R = O.window_length(T)
    x = synth.generate(w, R)
    G, s = w.group, w.cluster_size
    d = w.head_dim
    for h in (0, 5):
        K = x.k[0, 0, h, :T].double().numpy()
        qw = x.q_win[0, 0, h * G:(h + 1) * G, R - R:].double().numpy()
        score = O.accumulated_attention(qw, K, 1 / math.sqrt(d))
        kept = O.static_evict(score, O.kept_count(T, w.keep_ppm))
        start = int(x.needle_pos[0, 0, h])
        needles = list(range(start, start + w.needle_len))
        assert set(needles) <= set(kept.tolist())
        cache = K[kept]
        cache_idx = [int(np.searchsorted(kept, t)) for t in needles]
        for e in range(8):
            n_tok = len(kept) + e
            levels = O.cluster_pyramid(cache[:n_tok], s, w.fanouts, w.alpha)
            sel = O.hierarchical_select(x.q[e, 0, 0, h * G:(h + 1) * G].double().numpy(),
                                        levels, w.fanouts, w.level_keep_ppm)
            att = set(O.attended_tokens(n_tok, s, sel).tolist())
            assert set(cache_idx) <= att
            cache = np.vstack([cache, x.k_new[e, 0, 0, h].double().numpy()[None]])


# ---------------------------------------------------------------- P11 ------

def test_p11_commonality():
    idx = [[3, 1, 2], [3, 1, 2], [3, 1, 2], [3, 1, 2]]
    assert O.commonality(idx, 3, 1) == 1.0
    assert O.commonality(idx, 3, 3) == 1.0
    # hand-worked: layers {0,1,2}, {1,2,3}, {2,3,4}; k = 3, m = 1
    # |L0 & L1| = 2, |L1 & L2| = 2 -> (2 + 2) / (3 * 2)
    assert abs(O.commonality([[0, 1, 2], [1, 2, 3], [2, 3, 4]], 3, 1) - 4 / 6) < 1e-15
    run = _tiny_run(6, 2, E=1)
    sel = [list(run.selected[(0, l, 0, 0)]) for l in range(2, 6)]
    k = len(sel[0])
    assert O.commonality([sel[0], sel[1]], k, 1) == 1.0      # layers 2, 3 share


def test_p11_selected_positions_name_the_cached_tokens():
    """The positions of a selected cluster are the tokens its cache rows hold:
    a kept row holds the prompt key at its position, a row appended at
    decode step e holds that step's key, at position prompt_len + e."""
    assert O.selected_positions([3, 7, 9, 12], 14, [1, 2], 2) == [9, 12, 14, 15]
    assert O.selected_positions([0, 5], 6, [], 2) == []
    rng = np.random.default_rng(5)
    L, Hkv, T, d, s, E = 2, 2, 40, 8, 4, 10
    K = rng.standard_normal((L, Hkv, T, d)); V = rng.standard_normal((L, Hkv, T, d))
    Qw = rng.standard_normal((L, Hkv, T, d))
    q = rng.standard_normal((E, L, Hkv, d)); kn = rng.standard_normal((E, L, Hkv, d))
    p = O.Params(keep_ppm=500_000, cluster_size=s, fanouts=(2,), level_keep_ppm=(250_000, 500_000), share_every=1)
    res = O.run(lambda l, b: K[l], lambda l, b: V[l], lambda l, b: Qw[l], lambda e, l, b: q[e, l],
                lambda e, l, b: kn[e, l], lambda e, l, b: V[l][:, 0] * 0, [T], p, steps=E, layers=[0, 1])
    for l in range(L):
        for h in range(Hkv):
            kept = res.kept[(l, 0, h)]
            cache = np.vstack([res.cache_k[(l, 0, h)], kn[:, l, h]])   # every row after E appends
            n_clusters = cache.shape[0] // s
            for c in range(n_clusters):
                pos = O.selected_positions(kept, T, [c], s)
                want = [K[l, h, x] if x < T else kn[x - T, l, h] for x in pos]
                assert np.array_equal(np.array(want), cache[c * s:(c + 1) * s]), (l, h, c)
            assert len(set(O.selected_positions(kept, T, range(n_clusters), s))) == n_clusters * s


def test_mean_summary_composes_by_member_counts():
    """A coarse cluster's mean key is its children's means weighted by their
    token counts (the last cluster of a level may hold fewer children)."""
    rng = np.random.default_rng(77)
    keys = rng.standard_normal((16 * 23 + 5, 8))
    fan = (3, 2)
    levels = O.cluster_pyramid(keys, 16, fan, 0.6)
    for l in (1, 2):
        f = fan[l - 1]
        child = levels[l - 1]
        for c, m in enumerate(levels[l].members):
            kids = range(c * f, min((c + 1) * f, len(child.members)))
            w = np.array([len(child.members[q]) for q in kids], dtype=np.float64)
            want = (w[:, None] * child.mean[list(kids)]).sum(0) / w.sum()
            assert np.allclose(levels[l].mean[c], want, rtol=1e-13, atol=1e-15)
            assert len(m) == w.sum()
