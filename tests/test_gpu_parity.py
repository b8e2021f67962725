"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle.

Tolerances:
* attention outputs: max |o - o_ref| / max |o_ref| per output vector
  <= 1e-5 (fp32 KV) and <= 2e-3 (bf16 KV);
* summaries: r_max / r_min bit-exact, rep within fp32 rounding, the mean key
  within 64 u of the largest member key;
* cache contents: bit-exact;
* scores and index sets: within bands derived from the kernels' fp32
  arithmetic (``static_band`` / ``select_band``); an index set must equal
  the oracle's unless the oracle's margin at a cut is inside the band (a tie
  at the kernel's precision), in which case only its validity is checked.
"""
import ctypes as C
import math

import numpy as np
import pytest
import torch

from oracle import mpcache_oracle as O
from paper_2501_06807_gb300 import mpcache, synth
from tests import helpers as H

pytestmark = pytest.mark.gpu
U = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2501_06807_gb300 import build
    build.build()


def _tol(dtype):
    return 1e-5 if dtype == torch.float32 else 2e-3


def static_band(qw, K, scale, w, G):
    """Relative error bound of the GPU's accumulated scores: fp32 dot products
    over d channels (|error| <= d u sum|q k|), the log2 rescale and the row
    statistic -(m + log2 l) folded into the exponent (four roundings of
    magnitude up to scale log2(e) A, and log2 l <= log2 T), two ex2.approx per
    probability and the row / column sums."""
    A = (np.abs(qw.reshape(-1, qw.shape[-1])) @ np.abs(K).T).max()
    d, T = K.shape[1], K.shape[0]
    return (2 * scale * d * U * A + 4 * U * scale * 1.4427 * A + 3 * U * math.log2(T) + 4 * 2.0 ** -22
            + (T / 64 + w * G / 64 + 64) * U)


def score_stats(got, ref, w, G):
    """Measured error of accumulated scores against the oracle's: the largest
    relative error of one token's score, the mean signed relative error, and
    the relative error of the total mass (the oracle's total is w G, each
    softmax row summing to 1)."""
    pos = ref > 0
    rel = (got[pos] - ref[pos]) / ref[pos]
    mass = float(ref.sum())
    return {"max_rel_err": float(np.abs(rel).max(initial=0.0)), "mean_rel_err": float(rel.mean()) if rel.size else 0.0,
            "mass_rel_err": abs(float(got.sum()) - mass) / max(mass, 1e-300), "mass": w * G}


def score_estimate(qw, K, scale, w, G):
    """Typical relative error of the GPU's accumulated scores, the bound the
    element-wise check uses.  The worst-case band (static_band) grows with d
    u per dot product; rounding errors of d fp32 additions add up like a
    random walk, so this estimate takes sqrt(d) u: the exponent of each
    probability is off by about c sqrt(d) u A (A bounds sum |q k|, c is the
    scale times log2 e), plus one rounding of the row statistic (at most
    c A + log2 T), the ex2 approximation (a few ulp) and the column sum over
    the w G window rows (sqrt(w G) u)."""
    A = (np.abs(qw.reshape(-1, qw.shape[-1])) @ np.abs(K).T).max()
    d, T = K.shape[1], K.shape[0]
    c = scale * 1.4426950408889634
    return math.log(2) * (c * math.sqrt(d) * U * A + U * (c * A + math.log2(max(T, 2)))) + 4 * U + math.sqrt(w * G) * U


def check_scores(got, ref, qw, K, scale, w, G, tau, where):
    """Every score within the estimate of score_estimate of its oracle value
    (the worst-case band tau, 13-21 times wider on the tested workloads,
    only decides which ids count as ties at the budget cut), and no systematic error: the total mass
    (w G, each softmax row sums to 1) and the mean signed relative error
    within 1e-5, so that a score error of 1e-4 in the same direction fails."""
    est = score_estimate(qw, K, scale, w, G)
    assert est < tau
    pos = ref > 0
    assert np.all(np.abs(got - ref) <= est * np.maximum(ref, 1e-30) + 1e-30), (where, est)
    st = score_stats(got, ref, w, G)
    assert st["mass_rel_err"] <= 1e-5, (where, st)
    if pos.sum() >= 64:
        assert abs(st["mean_rel_err"]) <= 1e-5, (where, st)
    return est


def select_band(q_group, levels):
    """Absolute error bound of the GPU's cluster similarities (fp32 q-sum,
    fp32 rep, fp32 dot over d channels), doubled for a pair of candidates."""
    qa = np.abs(q_group).sum(0)
    qs = np.abs(q_group.sum(0))
    d, G = q_group.shape[1], q_group.shape[0]
    b = 0.0
    for lev in levels:
        if len(lev.r_max):
            mag = np.abs(lev.r_max) + np.abs(lev.r_min)
            b = max(b, float(((d + 4) * U * (mag @ qs) + G * U * (mag @ qa)).max()))
    return 2 * b + 1e-30


def unique_selection(trace, band):
    return cut_margin(trace) > band


def cut_margin(trace):
    """Smallest gap, over a selection's levels, between the oracle's k-th and
    (k+1)-th similarity (inf when no level cuts)."""
    m = math.inf
    for cand, sim, k in trace:
        if 0 < k < len(cand):
            srt = np.sort(sim)[::-1]
            m = min(m, float(srt[k - 1] - srt[k]))
    return m


# ------------------------------------------------ attention in isolation ----

ATTN_CASES = [
    # dtype, d, Hq, Hkv, s, fanouts, n_keep, steps
    (torch.float32, 64, 2, 1, 16, (), 83, 20),
    (torch.float32, 128, 8, 1, 32, (2,), 150, 36),
    (torch.bfloat16, 128, 4, 1, 16, (4,), 200, 35),
    (torch.bfloat16, 128, 8, 2, 16, (8, 8), 600, 18),
    (torch.bfloat16, 64, 2, 2, 8, (3,), 77, 17),
    (torch.bfloat16, 128, 16, 1, 4, (2, 2), 61, 9),
    (torch.bfloat16, 64, 1, 1, 1, (4,), 40, 5),
    (torch.bfloat16, 128, 4, 2, 16, (4,), 5, 13),   # starts with no full cluster
]


@pytest.mark.parametrize("dtype,d,Hq,Hkv,s,fan,N,E", ATTN_CASES)
def test_attention_cache_and_seal(dtype, d, Hq, Hkv, s, fan, N, E):
    g = torch.Generator().manual_seed(N * 7 + d)
    L, B, T = 4, 2, N + 37
    G = Hq // Hkv
    keep = tuple([O.PPM] * (1 + len(fan)))
    eng = H.make_engine(synth.Workload("t", L, B, Hq, Hkv, d, "f32" if dtype == torch.float32 else "bf16",
                                       T, T, O.PPM, s, fan, keep, 2, E, "iid"), E)
    K = torch.randn((L, B, Hkv, T, d), generator=g).to(dtype)
    V = torch.randn((L, B, Hkv, T, d), generator=g).to(dtype)
    kept = torch.zeros((eng.n_groups, B, Hkv, N), dtype=torch.int32)
    for idx in np.ndindex(eng.n_groups, B, Hkv):
        kept[idx] = torch.sort(torch.randperm(T, generator=g)[:N]).values.to(torch.int32)
    eng.kept[..., :N] = kept.cuda()
    eng.n_keep.fill_(N)
    eng.build_clusters(K.cuda(), V.cuda())
    torch.cuda.synchronize()
    assert eng.n_tok.tolist() == [N] * B
    # cache rows are the kept rows, bit-exact
    caches = {}
    for l in range(L):
        grp = eng.group_of[l]
        for b in range(B):
            for h in range(Hkv):
                ids = kept[grp, b, h].long()
                got_k = H.unswizzle(eng.kc[l, b, h, :N].cpu())
                got_v = H.unswizzle(eng.vc[l, b, h, :N].cpu())
                assert torch.equal(got_k, K[l, b, h, ids]) and torch.equal(got_v, V[l, b, h, ids])
                caches[(l, b, h)] = [K[l, b, h, ids].double().numpy(), V[l, b, h, ids].double().numpy()]

    def check_pyramid(n_tok):
        for l in eng.leaders:
            grp = eng.group_of[l]
            for b in range(B):
                for h in range(Hkv):
                    lev = O.cluster_pyramid(caches[(l, b, h)][0][:n_tok], s, fan, 0.6)
                    for li, lv in enumerate(lev):
                        n = len(lv.members)
                        rows = slice(_off(eng, li), _off(eng, li) + n)
                        assert np.array_equal(eng.rmax[grp, b, h, rows].cpu().double().numpy(), lv.r_max)
                        assert np.array_equal(eng.rmin[grp, b, h, rows].cpu().double().numpy(), lv.r_min)
                        rep = eng.rep[grp, b, h, rows].cpu().double().numpy()
                        assert np.allclose(rep, lv.rep, rtol=4e-7, atol=4e-7 * np.abs(lv.rep).max(initial=0))
                        # mean key: fp32 sums of s rows, weighted child means and
                        # running means at seals; bounded by 64 u of the largest key
                        mean = eng.mean[grp, b, h, rows].cpu().double().numpy()
                        kmax = np.abs(caches[(l, b, h)][0][:n_tok]).max(initial=0)
                        assert np.allclose(mean, lv.mean, rtol=0, atol=64 * 2.0 ** -24 * kmax)

    check_pyramid(N)
    scale = 1 / math.sqrt(d)
    for e in range(E):
        n_tok = N + e
        C1 = n_tok // s
        k = int(torch.randint(0, min(C1, eng.sel_cap) + 1, (1,), generator=g)) if e % 5 else min(C1, eng.sel_cap)
        sel = torch.full((eng.n_groups, B, Hkv, eng.sel_cap), -1, dtype=torch.int32)
        for idx in np.ndindex(eng.n_groups, B, Hkv):
            sel[idx][:k] = torch.sort(torch.randperm(C1, generator=g)[:k]).values.to(torch.int32)
        eng.sel.copy_(sel.cuda())
        eng.n_sel.fill_(k)
        q = torch.randn((L, B, Hq, d), generator=g).to(dtype)
        kn = torch.randn((L, B, Hkv, d), generator=g).to(dtype)
        vn = torch.randn((L, B, Hkv, d), generator=g).to(dtype)
        eng.attend(q.cuda(), kn.cuda(), vn.cuda(), advance=True)
        out = eng.out.cpu().double().numpy()
        for l in range(L):
            grp = eng.group_of[l]
            for b in range(B):
                for h in range(Hkv):
                    c = caches[(l, b, h)]
                    c[0] = np.vstack([c[0], kn[l, b, h].double().numpy()[None]])
                    c[1] = np.vstack([c[1], vn[l, b, h].double().numpy()[None]])
                    toks = O.attended_tokens(n_tok, s, sel[grp, b, h, :k].numpy())
                    for gg in range(G):
                        ref = O.sparse_attention(q[l, b, h * G + gg].double().numpy(), c[0][toks], c[1][toks], scale)
                        err = H.rel_err(out[l, b, h * G + gg], ref)
                        assert err <= _tol(dtype), (e, l, b, h, gg, err)
        if (n_tok + 1) % s == 0:
            check_pyramid(n_tok + 1)
    torch.cuda.synchronize()
    assert eng.n_tok.tolist() == [N + E] * B
    # appended rows landed in the cache
    for l in range(L):
        got = H.unswizzle(eng.kc[l, 0, 0, :N + E].cpu()).double().numpy()
        assert np.array_equal(got, caches[(l, 0, 0)][0])
    from paper_2501_06807_gb300 import mpcache
    assert mpcache.device_status() == 0


def _off(eng, level):
    cap = eng.cap_tokens // eng.s
    off = 0
    for li in range(level):
        off += cap
        cap = -(-cap // eng.fanouts[li])
    return off


@pytest.mark.parametrize("case", ["bf16_dense", "bf16_paged", "f32_d64"])
def test_prefill_per_group_from_pinned_host_memory(case):
    """Static eviction one leader at a time and gathering per group, with the
    keys of non-leader layers and all values read from pinned host memory
    (only the kept rows cross the host link), equals the one-call prefill
    from device tensors bit for bit."""
    if case == "f32_d64":
        w = synth.C1.replace(n_layers=4, prompt_len=300, prompt_len_min=200, batch=2, n_q_heads=4, n_kv_heads=2,
                             share_every=2, fanouts=(4,), level_keep_ppm=(250_000, 500_000))
    else:
        w = synth.C3.replace(n_layers=6, prompt_len=700, prompt_len_min=300, batch=2, n_q_heads=8, n_kv_heads=2,
                             share_every=2)
    if case == "bf16_paged":
        w = w.replace(page_size=16, paged=True)
    x = synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=1)
    xc = H.to_cuda(x)
    pt = xc.page_table.cuda() if xc.page_table is not None else None
    lens = x.prompt_lens.cuda()
    ref = H.make_engine(w, 1)
    ref.prefill(xc.k, xc.v, xc.q_win, lens, pt, w.page_size)
    eng = H.make_engine(w, 1)
    hk, hv = x.k.pin_memory(), x.v.pin_memory()
    gat = torch.cuda.Stream()
    for lead in eng.leaders:
        eng.static_evict(xc.k, xc.q_win, lens, pt, w.page_size, layers=[lead])
        gat.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(gat):
            members = [l for l in range(w.n_layers) if eng.group_of[l] == eng.group_of[lead] and l != lead]
            eng.build_clusters(xc.k, hv, pt, w.page_size, layers=[lead])
            if members:
                eng.build_clusters(hk, hv, pt, w.page_size, layers=members)
    torch.cuda.current_stream().wait_stream(gat)
    torch.cuda.synchronize()
    for name in ("kept", "n_keep", "n_tok", "kc", "vc", "rmax", "rmin", "rep", "mean"):
        assert torch.equal(getattr(eng, name), getattr(ref, name)), name
    assert torch.equal(eng.scores, ref.scores)
    assert mpcache.device_status() == 0
    # static eviction reads keys through TMA tensor maps: host keys are
    # refused by the binding and, below it, by the C call before any launch
    with pytest.raises(ValueError, match="on the GPU"):
        eng.static_evict(hk, xc.q_win, lens, pt, w.page_size)
    a = eng.static_args(xc.k, xc.q_win, lens, pt, w.page_size)
    a.k.data = hk.data_ptr()
    lib = mpcache.load()
    rc = lib.mpc_static_evict(C.byref(a), None, 0, C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == mpcache.MPC_ERR_INVALID_ARG, lib.mpc_last_error()
    assert b"host memory" in lib.mpc_last_error()
    assert mpcache.device_status() == 0


# ------------------------------------------------- selection in isolation ----

SELECT_CASES = [
    # dtype, d, Hq, Hkv, s, fanouts, keep ppm (finest first), n_tok, batch
    (torch.float32, 64, 3, 3, 16, (), (250_000,), 16 * 37 + 5, 2),
    (torch.bfloat16, 128, 4, 4, 16, (4,), (125_000, 500_000), 1024, 2),
    (torch.bfloat16, 128, 32, 8, 16, (8, 8), (50_000, 250_000, 500_000), 8192 + 7, 2),
    (torch.bfloat16, 128, 8, 2, 16, (8,), (100_000, 500_000), 2048 + 15, 2),
    (torch.bfloat16, 64, 2, 1, 1, (), (30_000,), 3000, 2),       # token-wise (s = 1): sort path
    (torch.float32, 128, 2, 1, 4, (3, 2), (200_000, 400_000, 600_000), 997, 2),
    (torch.bfloat16, 128, 4, 1, 16, (4,), (1_000_000, 1_000_000), 320, 2),  # keep all
    (torch.bfloat16, 128, 2, 1, 4, (), (150_000,), 2003, 2),     # 500 candidates: counting-rank path
    (torch.bfloat16, 128, 40, 20, 16, (4,), (125_000, 500_000), 700, 8),  # 160 units: 8-warp CTAs
    (torch.bfloat16, 64, 40, 40, 16, (4,), (125_000, 500_000), 600, 8),   # 320 units: 4-warp CTAs
    # 320 units (4-warp CTAs, six per SM): 94 coarse rows and 188 children
    # exceed the capped row buffer, so both rounds stage in several batches
    (torch.bfloat16, 128, 40, 40, 16, (4,), (125_000, 500_000), 6000, 8),
    (torch.bfloat16, 128, 8, 2, 16, (4, 4, 2), (60_000, 250_000, 500_000, 500_000), 4096 + 9, 2),  # four levels
]


@pytest.mark.parametrize("metric", ["eq3", "bound", "mean"])
@pytest.mark.parametrize("dtype,d,Hq,Hkv,s,fan,keep,N,B", SELECT_CASES)
def test_selection(dtype, d, Hq, Hkv, s, fan, keep, N, B, metric):
    _check_selection(dtype, d, Hq, Hkv, s, fan, keep, N, B, metric, 0.6)


@pytest.mark.parametrize("alpha", [0.0, 0.25, 1.0])
def test_selection_alpha_sweep(alpha):
    # Eq. 3's weight between r_max and r_min (the paper's alpha ablation):
    # the summaries and the selection follow it
    _check_selection(torch.bfloat16, 128, 8, 2, 16, (8,), (100_000, 500_000), 2048 + 15, 2, "eq3", alpha)


def _check_selection(dtype, d, Hq, Hkv, s, fan, keep, N, B, metric, alpha):
    g = torch.Generator().manual_seed(N + d)
    L = 1
    G = Hq // Hkv
    eng = H.make_engine(synth.Workload("t", L, B, Hq, Hkv, d, "f32" if dtype == torch.float32 else "bf16",
                                       N, N, O.PPM, s, fan, keep, 1, 4, "iid", alpha=alpha), 4)
    # keys with token-wise locality (a slow drift per channel), the structure
    # clustering relies on; iid keys make coarse summaries indistinguishable
    drift = torch.cumsum(torch.randn((L, B, Hkv, N, d), generator=g) * 0.15, dim=3)
    K = ((torch.randn((L, B, Hkv, N, d), generator=g) + drift)
         * torch.rand((1, 1, Hkv, 1, d), generator=g) * 3).to(dtype)
    eng.kept[..., :N] = torch.arange(N, dtype=torch.int32).cuda()
    eng.n_keep.fill_(N)
    eng.build_clusters(K.cuda(), K.cuda())
    ties = near = 0
    ratio = math.inf  # smallest (gap at a cut) / (band) over the units
    for rep_i in range(3):
        q = (torch.randn((L, B, Hq, d), generator=g) * 2).to(dtype)
        eng.select(q.cuda(), {"eq3": mpcache.MPC_SIM_EQ3, "bound": mpcache.MPC_SIM_BOUND,
                              "mean": mpcache.MPC_SIM_MEAN}[metric])
        sel = eng.sel.cpu().numpy()
        n_sel = eng.n_sel.cpu().numpy()
        for b in range(B):
            for h in range(Hkv):
                levels = O.cluster_pyramid(K[0, b, h].double().numpy(), s, fan, alpha)
                qg = q[0, b, h * G:(h + 1) * G].double().numpy()
                tr = []
                ref = O.hierarchical_select(qg, levels, fan, keep, trace=tr, metric=metric)
                got = sel[0, b, h, :n_sel[b]]
                assert n_sel[b] == len(ref)
                assert (sel[0, b, h, n_sel[b]:] == -1).all()
                band = select_band(qg, levels)
                ratio = min(ratio, cut_margin(tr) / band)
                if unique_selection(tr, band):
                    assert np.array_equal(got, ref), (b, h)
                else:
                    near += 1
                    if not np.array_equal(got, ref):
                        ties += 1
                        assert np.all(np.diff(got) > 0) and got.min(initial=0) >= 0
                        assert got.max(initial=-1) < N // s
    H.log_parity("selection", case=f"{str(dtype)[6:]} d{d} Hq{Hq} Hkv{Hkv} s{s} fan{fan} N{N} B{B}", metric=metric,
                 alpha=alpha, units=3 * B * Hkv, units_within_band=near, units_differing=ties,
                 min_gap_over_band=ratio if math.isfinite(ratio) else None)
    assert ties <= max(1, 3 * B * Hkv // 100)


@pytest.mark.parametrize("frac_bits", [18, 5])
@pytest.mark.parametrize("dtype,d,Hq,Hkv,s,fan,keep,N,B", SELECT_CASES)
def test_selection_fixed_point(dtype, d, Hq, Hkv, s, fan, keep, N, B, frac_bits):
    _check_selection_fxp(dtype, d, Hq, Hkv, s, fan, keep, N, B, frac_bits, 1.0)


def test_selection_fixed_point_ring_wraps():
    # f = 24 and large values: the ring sums leave the int64 range and wrap
    # modulo 2^64 on both sides
    _check_selection_fxp(torch.bfloat16, 128, 4, 1, 16, (4,), (125_000, 500_000), 1024, 2, 24, 60.0, wraps=True)


def _check_selection_fxp(dtype, d, Hq, Hkv, s, fan, keep, N, B, frac_bits, scale, wraps=False):
    """Eq. 3 in the fixed-point ring: integer scores, so the selection is
    bit-exact (equal scores rank the lower id first on both sides)."""
    g = torch.Generator().manual_seed(N + d + frac_bits)
    G = Hq // Hkv
    alpha = float(np.float32(0.6))
    eng = H.make_engine(synth.Workload("t", 1, B, Hq, Hkv, d, "f32" if dtype == torch.float32 else "bf16",
                                       N, N, O.PPM, s, fan, keep, 1, 4, "iid"), 4)
    drift = torch.cumsum(torch.randn((1, B, Hkv, N, d), generator=g) * 0.15, dim=3)
    K = ((torch.randn((1, B, Hkv, N, d), generator=g) + drift)
         * torch.rand((1, 1, Hkv, 1, d), generator=g) * 3 * scale).to(dtype)
    eng.kept[..., :N] = torch.arange(N, dtype=torch.int32).cuda()
    eng.n_keep.fill_(N)
    eng.build_clusters(K.cuda(), K.cuda())
    wrapped = False
    for rep_i in range(3):
        q = (torch.randn((1, B, Hq, d), generator=g) * 2 * scale).to(dtype)
        eng.select(q.cuda(), mpcache.MPC_SIM_FXP, frac_bits)
        sel = eng.sel.cpu().numpy()
        n_sel = eng.n_sel.cpu().numpy()
        for b in range(B):
            for h in range(Hkv):
                levels = O.cluster_pyramid(K[0, b, h].double().numpy(), s, fan, alpha)
                qg = q[0, b, h * G:(h + 1) * G].double().numpy()
                ref = O.hierarchical_select(qg, levels, fan, keep, metric="fxp", alpha=alpha, frac_bits=frac_bits)
                assert n_sel[b] == len(ref)
                assert np.array_equal(sel[0, b, h, :n_sel[b]], ref), (b, h)
                assert (sel[0, b, h, n_sel[b]:] == -1).all()
                if wraps:
                    qs = O.fxp_encode(qg, frac_bits).sum(0).astype(object)
                    rep = levels[0].r_max[0] * alpha + levels[0].r_min[0] * (1 - alpha)
                    wrapped |= abs(int(sum(qs * O.fxp_encode(rep, frac_bits).astype(object)))) >= 2 ** 63
    assert wrapped or not wraps


def test_fixed_point_ranking_survives_on_needle_workload():
    """Eq. 3 in the fixed-point ring at the default 18 fractional bits, on the
    needle workload (three-level pyramid, GQA): the selections equal the fp32
    ones almost everywhere, and every cluster of the needle passage that the
    fp32 selection keeps is kept.  Coarser encodings are reported alongside."""
    w = synth.C5.replace(n_layers=3, prompt_len=4096, prompt_len_min=4096, n_q_heads=8, n_kv_heads=2,
                         level_keep_ppm=(100_000, 250_000, 500_000))
    E = 12
    x = synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=E)
    xc = H.to_cuda(x)
    eng = H.make_engine(w, E)
    eng.prefill(xc.k, xc.v, xc.q_win, x.prompt_lens.cuda(), None, w.page_size)
    kept = eng.kept.cpu().numpy()
    same = {18: 0, 8: 0, 5: 0, 3: 0}
    units = needles = needles_kept = 0
    for e in range(E):
        eng.select(xc.q[e])
        ref = eng.sel.cpu().numpy().copy()
        for fb in same:
            eng.select(xc.q[e], mpcache.MPC_SIM_FXP, fb)
            got = eng.sel.cpu().numpy()
            same[fb] += int((got == ref).all(axis=-1).sum())
            if fb != 18:
                continue
            for lead in eng.leaders:
                grp = eng.group_of[lead]
                for b in range(w.batch):
                    for h in range(w.n_kv_heads):
                        p0 = int(x.needle_pos[lead, b, h])
                        pos = kept[grp, b, h]
                        hit = np.nonzero((pos >= p0) & (pos < p0 + w.needle_len))[0]
                        clusters = set((hit // w.cluster_size).tolist())
                        want = clusters & set(ref[grp, b, h].tolist())
                        needles += len(want)
                        needles_kept += len(want & set(got[grp, b, h].tolist()))
        units += ref.shape[0] * ref.shape[1] * ref.shape[2]
        eng.decode_step(xc.q[e], xc.k_new[e], xc.v_new[e])
    frac = {fb: same[fb] / units for fb in same}
    print("identical selections (fraction of units) by fractional bits:", frac,
          "needle clusters kept:", needles_kept, "/", needles)
    assert needles > 0 and needles_kept == needles
    assert frac[18] >= 0.95
    assert mpcache.device_status() == 0


# ----------------------------------------------- static eviction alone ----

STATIC_CASES = [
    # dtype, d, Hq, Hkv, lens, keep_ppm, page size (0: dense keys)
    (torch.float32, 64, 4, 4, (512,), 500_000, 0),
    (torch.bfloat16, 128, 8, 2, (1000,), 250_000, 0),
    (torch.bfloat16, 64, 2, 1, (129, 300, 64), 500_000, 0),
    (torch.bfloat16, 128, 4, 4, (777, 1500), 125_000, 16),
    (torch.float32, 128, 2, 2, (33,), 1_000_000, 0),
    (torch.bfloat16, 128, 4, 1, (1,), 500_000, 0),
    (torch.bfloat16, 128, 4, 2, (300, 1000), 250_000, 4),     # pages smaller than a swizzle atom
    (torch.bfloat16, 64, 8, 2, (777, 129), 500_000, 48),      # pages that do not divide 128
    (torch.bfloat16, 128, 2, 2, (1500,), 125_000, 256),       # pages larger than a key tile
    (torch.float32, 64, 4, 2, (500, 333), 500_000, 32),       # fp32 keys: paged SIMT passes
    (torch.bfloat16, 128, 2, 1, (49152,), 250_000, 0),        # the longest prompt the calls accept
]


@pytest.mark.parametrize("dtype,d,Hq,Hkv,lens,keep,page", STATIC_CASES)
def test_static_eviction(dtype, d, Hq, Hkv, lens, keep, page):
    g = torch.Generator().manual_seed(sum(lens) + d)
    B, T = len(lens), max(lens)
    G = Hq // Hkv
    w = synth.Workload("t", 1, B, Hq, Hkv, d, "f32" if dtype == torch.float32 else "bf16", T, min(lens),
                       keep, 16, (), (O.PPM,), 1, 1, "iid", paged=page > 0)
    eng = H.make_engine(w, 1)
    R = eng.win_rows
    K = torch.zeros((1, B, Hkv, T, d))
    Q = torch.zeros((1, B, Hq, R, d))
    for b, t in enumerate(lens):
        K[0, b, :, :t] = torch.randn((Hkv, t, d), generator=g) * 1.5
        Q[0, b, :, R - min(R, t):] = torch.randn((Hq, min(R, t), d), generator=g) * 1.5
    K, Q = K.to(dtype), Q.to(dtype)
    lens_t = torch.tensor(lens, dtype=torch.int32)
    if page:
        P = page
        n_pages = [(t + P - 1) // P for t in lens]
        perm = torch.randperm(sum(n_pages), generator=g).to(torch.int32)
        pt = torch.full((B, (T + P - 1) // P), -1, dtype=torch.int32)
        pool = torch.zeros((1, sum(n_pages), Hkv, P, d), dtype=dtype)
        o = 0
        for b, t in enumerate(lens):
            pt[b, :n_pages[b]] = perm[o:o + n_pages[b]]
            o += n_pages[b]
            for j in range(n_pages[b]):
                seg = K[0, b, :, j * P:(j + 1) * P]
                pool[0, int(pt[b, j]), :, :seg.shape[1]] = seg
        eng.static_evict(pool.cuda(), Q.cuda(), lens_t.cuda(), pt.cuda(), P)
    else:
        eng.static_evict(K.cuda(), Q.cuda(), lens_t.cuda())
    scores = eng.scores.cpu().double().numpy()
    kept = eng.kept.cpu().numpy()
    assert eng.n_keep.cpu().tolist() == [O.kept_count(t, keep) for t in lens]
    for b, t in enumerate(lens):
        wl = O.window_length(t)
        for h in range(Hkv):
            qw = Q[0, b, h * G:(h + 1) * G, R - wl:].double().numpy()
            kk = K[0, b, h, :t].double().numpy()
            ref = O.accumulated_attention(qw, kk, 1 / math.sqrt(d))
            tau = static_band(qw, kk, 1 / math.sqrt(d), wl, G)
            got = scores[0, b, h, :t]
            est = check_scores(got, ref, qw, kk, 1 / math.sqrt(d), wl, G, tau, (b, h))
            nk = O.kept_count(t, keep)
            ref_kept = O.static_evict(ref, nk)
            assert np.all(kept[0, b, h, nk:] == -1)
            swaps = H.set_parity(kept[0, b, h, :nk], ref_kept, lambda ids: ref[ids], nk,
                                 band=2 * tau * ref[ref_kept].min())
            H.log_parity("static_eviction", case=f"{str(dtype)[6:]} d{d} Hq{Hq} Hkv{Hkv} T{t} page{page}", b=b, h=h,
                         **score_stats(got, ref, wl, G), bound=est, tie_band=tau, swaps_at_cut=swaps, n_keep=nk)


# ------------------------------------------------------- full pipeline ----

def _pipeline(w: synth.Workload, E: int, layers, max_skip=0.02, device="cpu"):
    R = H.window_rows_for(w)
    x = synth.generate(w, R, device=device, decode_steps=E)
    xc = H.to_cuda(x)
    eng = H.make_engine(w, E)
    lens = x.prompt_lens.cuda()
    pt = xc.page_table.cuda() if xc.page_table is not None else None
    eng.prefill(xc.k, xc.v, xc.q_win, lens, pt, w.page_size)
    torch.cuda.synchronize()
    g_scores, g_kept = eng.scores.cpu().double().numpy(), eng.kept.cpu().numpy()
    sels, outs = [], []
    for e in range(E):
        eng.decode_step(xc.q[e], xc.k_new[e], xc.v_new[e])
        sels.append(eng.sel.cpu().numpy().copy())
        outs.append(eng.out.cpu().double().numpy().copy())
    res = H.oracle_run(x, E, layers)
    G = w.group
    diverged = set()   # (l, b, h) whose kept set is a tie-variant
    taus = {}
    units = 0
    worst = {"max_rel_err": 0.0, "mass_rel_err": 0.0, "bound": 0.0, "tie_band": 0.0, "swaps_at_cut": 0,
             "attn_max_rel_err": 0.0, "selection_ties": 0}
    for l in layers:
        lead = O.leader_of(l, w.share_every)
        grp = eng.group_of[l]
        for b in range(w.batch):
            T = int(x.prompt_lens[b])
            for h in range(w.n_kv_heads):
                if lead == l:
                    ref = res.scores[(l, b, h)]
                    kk, _ = x.dense_kv(l, b)
                    qw = x.q_win[l, b, h * G:(h + 1) * G, R - O.window_length(T):].double().numpy()
                    tau = static_band(qw, kk[h].double().numpy(), 1 / math.sqrt(w.head_dim),
                                      O.window_length(T), G)
                    got = g_scores[grp, b, h, :T]
                    est = check_scores(got, ref, qw, kk[h].double().numpy(), 1 / math.sqrt(w.head_dim),
                                       O.window_length(T), G, tau, (l, b, h))
                    worst["bound"] = max(worst["bound"], est)
                    st = score_stats(got, ref, O.window_length(T), G)
                    for key in ("max_rel_err", "mass_rel_err"):
                        worst[key] = max(worst[key], st[key])
                    worst["tie_band"] = max(worst["tie_band"], tau)
                    taus[(l, b, h)] = tau
                nk = len(res.kept[(l, b, h)])
                gk = g_kept[grp, b, h, :nk]
                if not np.array_equal(gk, res.kept[(l, b, h)]):
                    sc = res.scores[(lead, b, h)]
                    worst["swaps_at_cut"] += H.set_parity(gk, res.kept[(l, b, h)], lambda ids: sc[ids], nk,
                                                          band=2 * taus[(lead, b, h)] * sc[res.kept[(l, b, h)]].min())
                    diverged.add((l, b, h))
    skipped = 0
    for e in range(E):
        for l in layers:
            lead = O.leader_of(l, w.share_every)
            grp = eng.group_of[l]
            for b in range(w.batch):
                n_sel = None
                for h in range(w.n_kv_heads):
                    units += 1
                    if (lead, b, h) in diverged or (l, b, h) in diverged:
                        skipped += 1
                        continue
                    ref_sel = res.selected[(e, l, b, h)]
                    got_sel = sels[e][grp, b, h, :len(ref_sel)]
                    if not np.array_equal(got_sel, ref_sel):
                        levels = res.levels[(e, lead, b, h)]
                        qg = x.q[e, lead, b, h * G:(h + 1) * G].double().numpy()
                        tr = []
                        O.hierarchical_select(qg, levels, w.fanouts, w.level_keep_ppm, trace=tr)
                        assert not unique_selection(tr, select_band(qg, levels)), (e, l, b, h, got_sel, ref_sel)
                        skipped += 1
                        worst["selection_ties"] += 1
                        continue
                    for gg in range(G):
                        err = H.rel_err(outs[e][l, b, h * G + gg], res.out[(e, l, b)][h * G + gg])
                        worst["attn_max_rel_err"] = max(worst["attn_max_rel_err"], err)
                        assert err <= (1e-5 if w.dtype == "f32" else 2e-3), (e, l, b, h, gg, err)
    H.log_parity("pipeline", case=w.name, layers=len(layers), steps=E, units=units, tie_skipped_units=skipped, **worst)
    assert skipped <= max_skip * units, (skipped, units)
    from paper_2501_06807_gb300 import mpcache
    assert mpcache.device_status() == 0
    return eng, x, res


def test_pipeline_c1_full():
    """The GPT-2-small workload exactly as configured: 12 heads, 512 tokens,
    fp32, 8 decode steps; the sink token (key 0) is kept in every head."""
    eng, _, _ = _pipeline(synth.C1, synth.C1.decode_steps, [0], max_skip=0.0)
    kept = eng.kept.cpu().numpy()
    n = int(eng.n_keep[0])
    for h in range(synth.C1.n_kv_heads):
        assert 0 in kept[0, 0, h, :n], h


def test_pipeline_llama2_shape_reduced():
    w = synth.C2.replace(n_layers=5, prompt_len=1024, prompt_len_min=1024, n_q_heads=8, n_kv_heads=8)
    _pipeline(w, 21, list(range(5)))


def test_pipeline_gqa_three_levels_needles():
    w = synth.C5.replace(n_layers=3, prompt_len=4096, prompt_len_min=4096, n_q_heads=8, n_kv_heads=2,
                         level_keep_ppm=(100_000, 250_000, 500_000))
    _pipeline(w, 18, [0, 1, 2])


def test_pipeline_paged_ragged_batch():
    w = synth.C4.replace(n_layers=3, batch=3, prompt_len=700, prompt_len_min=300, n_q_heads=4, n_kv_heads=4)
    _pipeline(w, 10, [0, 1, 2])


def test_pipeline_token_wise_without_static_eviction():
    """The LongCache-style comparator (next-rows item 3): no static eviction
    (keep every prompt token) and one token per finest cluster, so selection
    ranks single tokens through a two-level pyramid of token groups."""
    w = synth.C3.replace(n_layers=2, prompt_len=1024, prompt_len_min=1024, n_q_heads=8, n_kv_heads=2,
                         keep_ppm=1_000_000, cluster_size=1, fanouts=(16,), level_keep_ppm=(50_000, 250_000),
                         share_every=1)
    _pipeline(w, 6, [0, 1])


# ------------------------------------------------- commonality score ----

@pytest.mark.parametrize("L,m,k,n_clusters,overlap", [(6, 1, 12, 200, 0.8), (10, 3, 26, 512, 0.6),
                                                      (4, 3, 5, 33, 1.0), (32, 2, 64, 4000, 0.3)])
def test_commonality_synthetic(L, m, k, n_clusters, overlap):
    """mpc_commonality against the oracle's commonality (Sec. 2, Obs. 3) on
    index sets with a controlled share of common ids; totals are exact."""
    from paper_2501_06807_gb300 import mpcache
    rng = np.random.default_rng(L * 100 + k)
    B, Hkv, cap = 2, 3, k + 4
    sel = np.full((L, B, Hkv, cap), -1, dtype=np.int32)
    sets = {}
    for b in range(B):
        for h in range(Hkv):
            base = rng.choice(n_clusters, k, replace=False)
            for l in range(L):
                keep = base[rng.random(k) < overlap]
                fresh = rng.choice(np.setdiff1d(np.arange(n_clusters), keep), k - len(keep), replace=False)
                ids = np.sort(np.concatenate([keep, fresh]))
                sel[l, b, h, :k] = ids
                sets[(b, h, l)] = list(ids)
    total, score = mpcache.commonality(torch.from_numpy(sel).cuda(), k, m, n_clusters)
    total, score = total.cpu().numpy(), score.cpu().numpy()
    for b in range(B):
        for h in range(Hkv):
            ref = O.commonality([sets[(b, h, l)] for l in range(L)], k, m)
            assert total[b, h] == round(ref * k * (L - m))
            assert abs(score[b, h] - ref) <= 1e-6 * max(ref, 1e-6)


def test_commonality_of_unshared_selections():
    """Every layer its own leader (m = 1 sharing): the commonality of the
    engine's per-layer selections equals the oracle's on the same sets."""
    from paper_2501_06807_gb300 import mpcache
    w = synth.C3.replace(n_layers=6, prompt_len=2048, prompt_len_min=2048, share_every=1, decode_steps=2)
    R = mpcache.window_rows_bound(w.prompt_len, w.window_ppm, w.long_window_ppm, w.long_prompt_threshold)
    x = synth.generate(w, R, device="cuda", decode_steps=2)
    eng = H.make_engine(w, 2)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda())
    eng.select(x.q[0])
    torch.cuda.synchronize()
    n_sel = int(eng.n_sel[0])
    sel = eng.sel[:, :, :, :]                    # [L (each its own group)][B][Hkv][sel_cap]
    assert sel.shape[0] == w.n_layers
    n_clusters = int(eng.n_tok[0]) // w.cluster_size
    for m in (1, 2):
        total, score = mpcache.commonality(sel.contiguous(), n_sel, m, n_clusters)
        s_cpu = sel.cpu().numpy()
        for b in range(w.batch):
            for h in range(w.n_kv_heads):
                ref = O.commonality([list(s_cpu[l, b, h, :n_sel]) for l in range(w.n_layers)], n_sel, m)
                assert int(total[b, h]) == round(ref * n_sel * (w.n_layers - m))


def test_adaptive_sharing_loop():
    """Adaptive cross-layer index sharing end to end (Sec. 2 Obs. 3, Sec. 3.4):
    every layer its own leader, the commonality of the selected tokens on the
    GPU for windows of 2 .. 4 layers at every decode step (exact totals
    against the oracle's commonality of the same selections as positions, and
    against the oracle's own pipeline where its kept sets and selections are
    the GPU's), the group size from mpc_choose_share_every against the rule
    worked by hand, then the method run with that group size against the
    oracle.  Adjacent layers are correlated (rho = 0.95) as a residual stream
    would make them; on these inputs the oracle's commonality is about 0.37,
    0.15 and 0.09 for windows of 2, 3 and 4 layers, so a threshold of 0.25
    shares between pairs of layers."""
    from paper_2501_06807_gb300 import mpcache
    w = synth.C3.replace(n_layers=6, prompt_len=2048, prompt_len_min=2048, n_q_heads=8, n_kv_heads=2,
                         keep_ppm=500_000, share_every=1, layer_rho_ppm=950_000)
    E, L, s, Hkv = 3, w.n_layers, w.cluster_size, w.n_kv_heads
    R = H.window_rows_for(w)
    x = synth.generate(w, R, device="cpu", decode_steps=E)
    xc = H.to_cuda(x)
    eng = H.make_engine(w, E)
    eng.prefill(xc.k, xc.v, xc.q_win, x.prompt_lens.cuda())
    res = H.oracle_run(x, E, list(range(L)))
    T = int(x.prompt_lens[0])
    ms = (1, 2, 3)
    scores = {m: [] for m in ms}
    units = same = 0
    for e in range(E):
        eng.decode_step(xc.q[e], xc.k_new[e], xc.v_new[e])
        torch.cuda.synchronize()
        sel, kept = eng.sel.cpu().numpy(), eng.kept.cpu().numpy()
        n_sel, nk = int(eng.n_sel[0]), int(eng.n_keep[0])
        assert n_sel >= 1
        prev_total = None
        for m in ms:
            total, score = eng.commonality(m)
            total, score = total.cpu().numpy(), score.cpu().numpy()
            for h in range(Hkv):
                pos = [O.selected_positions(kept[l, 0, h, :nk], T, sel[l, 0, h, :n_sel], s) for l in range(L)]
                ref = O.commonality(pos, n_sel * s, m)
                assert total[0, h] == round(ref * n_sel * s * (L - m)), (e, m, h)
                assert abs(score[0, h] - ref) <= 1e-6
                agree = all(np.array_equal(kept[l, 0, h, :nk], res.kept[(l, 0, h)]) and
                            np.array_equal(sel[l, 0, h, :n_sel], res.selected[(e, l, 0, h)]) for l in range(L))
                units += 1
                if agree:
                    same += 1
                    pos_o = [O.selected_positions(res.kept[(l, 0, h)], T, res.selected[(e, l, 0, h)], s)
                             for l in range(L)]
                    assert O.commonality(pos_o, n_sel * s, m) == ref
                scores[m].append(float(score[0, h]))
            # a window of m + 1 layers shares no more than its first m
            if prev_total is not None:
                assert (total <= prev_total).all()
            prev_total = total
    assert same >= 0.9 * units, (same, units)
    mean = {m: float(np.mean(v)) for m, v in scores.items()}
    for thr in (0.0, 0.25, 0.5, 0.75, 1.0):
        want = max([1] + [m + 1 for m in ms if mean[m] >= thr])
        assert mpcache.choose_share_every(mean, thr) == want, (thr, mean)
    chosen = mpcache.choose_share_every(mean, 0.25)
    H.log_parity("adaptive_sharing", case=w.name, rho_ppm=w.layer_rho_ppm, commonality=mean, threshold=0.25,
                 chosen_share_every=chosen, units_matching_oracle=same, units=units)
    assert chosen >= 2, mean
    _pipeline(w.replace(share_every=chosen), E, list(range(L)))


def test_commonality_positions_cover_sealed_clusters():
    """mpc_commonality's token positions for clusters sealed while decoding
    (R25: row r >= n_keep holds position T + r - n_keep): every cluster is
    selected (ratio 1 at both levels), 20 steps seal one cluster of appended
    rows, and the GPU's totals equal the oracle's commonality of the same
    selections mapped by selected_positions."""
    w = synth.C3.replace(n_layers=4, prompt_len=512, prompt_len_min=512, n_q_heads=4, n_kv_heads=2,
                         keep_ppm=500_000, share_every=1, level_keep_ppm=(1_000_000, 1_000_000))
    E, L, s = 20, w.n_layers, w.cluster_size
    x = H.to_cuda(synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=E))
    eng = H.make_engine(w, E)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda())
    for e in range(E):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
    eng.select(x.q[E - 1])  # selections over the cache after the last append
    torch.cuda.synchronize()
    T, nk, n_sel = int(x.prompt_lens[0]), int(eng.n_keep[0]), int(eng.n_sel[0])
    assert n_sel == (nk + E) // s and n_sel * s > nk   # a sealed cluster of appended rows is selected
    sel, kept = eng.sel.cpu().numpy(), eng.kept.cpu().numpy()
    for m in (1, 2, 3):
        total, _ = eng.commonality(m)
        for h in range(w.n_kv_heads):
            pos = [O.selected_positions(kept[l, 0, h, :nk], T, sel[l, 0, h, :n_sel], s) for l in range(L)]
            assert max(max(p) for p in pos) >= T                   # appended positions take part
            ref = O.commonality(pos, n_sel * s, m)
            assert int(total[0, h]) == round(ref * n_sel * s * (L - m)), (m, h)


# ------------------------------------------ full size, sampled outputs ----

def _full_size_sampled(w, E, pick):
    """Runs a workload at full size, in the launch configuration the
    benchmark times, for E decode steps, and checks sampled (leader,
    sequence, kv head) units against the oracle one by one: window scores and
    the kept set, the cluster summaries, every step's selection, and the
    attention outputs of the leader and of its group's last layer.
    Downstream checks start from the GPU's kept set and selections, so a tie
    at one cut does not mask the next stage.  ``pick(eng, x)`` names the
    sampled units."""
    R = H.window_rows_for(w)
    x = synth.generate(w, R, device="cuda", decode_steps=E)
    eng = H.make_engine(w, E)
    pt = x.page_table.cuda() if x.page_table is not None else None
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda(), pt, w.page_size)
    torch.cuda.synchronize()
    G, d, s = w.group, w.head_dim, w.cluster_size
    scale = 1 / math.sqrt(d)
    samples = pick(eng, x)
    members = {lead: [l for l in range(w.n_layers) if eng.group_of[l] == eng.group_of[lead]] for lead, _, _ in samples}
    watch = sorted({(l, b) for lead, b, _ in samples for l in (lead, members[lead][-1])})
    scores = eng.scores.cpu().double().numpy()
    kept = eng.kept.cpu().numpy()
    rmax, rmin, rep = eng.rmax.cpu().numpy(), eng.rmin.cpu().numpy(), eng.rep.cpu().numpy()
    sels, outs = [], []
    for e in range(E):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
        sels.append(eng.sel.cpu().numpy().copy())
        outs.append({lb: eng.out[lb[0], lb[1]].cpu().double().numpy() for lb in watch})
    assert mpcache.device_status() == 0
    dense = {}

    def kv(l, b):
        if (l, b) not in dense:
            k, v = x.dense_kv(l, b)
            dense[(l, b)] = (k.double().cpu().numpy(), v.double().cpu().numpy())
        return dense[(l, b)]

    for lead, b, h in samples:
        grp = eng.group_of[lead]
        T = int(x.prompt_lens[b])
        wl = O.window_length(T, w.window_ppm, w.long_window_ppm, w.long_prompt_threshold)
        n_keep = O.kept_count(T, w.keep_ppm)
        K = kv(lead, b)[0][h]
        qw = x.q_win[lead, b, h * G:(h + 1) * G, R - wl:].double().cpu().numpy()
        # static eviction
        ref = O.accumulated_attention(qw, K, scale)
        tau = static_band(qw, K, scale, wl, G)
        got = scores[grp, b, h, :T]
        est = check_scores(got, ref, qw, K, scale, wl, G, tau, (lead, b, h))
        ref_kept = O.static_evict(ref, n_keep)
        gk = kept[grp, b, h, :n_keep]
        swaps = H.set_parity(gk, ref_kept, lambda ids: ref[ids], n_keep, band=2 * tau * ref[ref_kept].min())
        rec = dict(case=w.name, lead=lead, b=b, h=h, **score_stats(got, ref, wl, G), bound=est, tie_band=tau,
                   swaps_at_cut=swaps,
                   steps=E, selection_ties=0, attn_max_rel_err=0.0, seals=0)
        # summaries of the GPU's kept keys, as gathered at prefill
        levels = O.cluster_pyramid(K[gk], s, w.fanouts, w.alpha)
        for li, lv in enumerate(levels):
            rows = slice(_off(eng, li), _off(eng, li) + len(lv.members))
            assert np.array_equal(rmax[grp, b, h, rows].astype(np.float64), lv.r_max), (lead, b, h, li)
            assert np.array_equal(rmin[grp, b, h, rows].astype(np.float64), lv.r_min), (lead, b, h, li)
            assert np.allclose(rep[grp, b, h, rows], lv.rep, rtol=4e-7, atol=4e-7 * np.abs(lv.rep).max(initial=0))
        for e in range(E):
            n_tok = n_keep + e  # cache rows before this step's append
            lead_cache = np.concatenate([K[gk], x.k_new[:e, lead, b, h].double().cpu().numpy()])
            lv_e = O.cluster_pyramid(lead_cache[:n_tok], s, w.fanouts, w.alpha)
            qg = x.q[e, lead, b, h * G:(h + 1) * G].double().cpu().numpy()
            tr = []
            ref_sel = O.hierarchical_select(qg, lv_e, w.fanouts, w.level_keep_ppm, trace=tr)
            got_sel = sels[e][grp, b, h, :len(ref_sel)]
            C1 = n_tok // s
            if n_tok % s == 0 and e > 0:
                rec["seals"] += 1  # the previous step's append sealed a cluster
            if unique_selection(tr, select_band(qg, lv_e)):
                assert np.array_equal(got_sel, ref_sel), (lead, b, h, e)
            else:
                rec["selection_ties"] += 1
                assert np.all(np.diff(got_sel) > 0) and got_sel.min(initial=0) >= 0 and got_sel.max(initial=-1) < C1
            rows = np.concatenate([np.arange(c * s, (c + 1) * s) for c in got_sel] + [np.arange(C1 * s, n_tok)])
            for l in (lead, members[lead][-1]):
                Kl, Vl = kv(l, b)
                cache_k = np.concatenate([Kl[h][gk], x.k_new[:e, l, b, h].double().cpu().numpy()])
                cache_v = np.concatenate([Vl[h][gk], x.v_new[:e, l, b, h].double().cpu().numpy()])
                Ka = np.concatenate([cache_k[rows], x.k_new[e, l, b, h][None].double().cpu().numpy()])
                Va = np.concatenate([cache_v[rows], x.v_new[e, l, b, h][None].double().cpu().numpy()])
                for g in range(G):
                    hq = h * G + g
                    q = x.q[e, l, b, hq].double().cpu().numpy()
                    o_ref = O.sparse_attention(q, Ka, Va, scale)
                    err = H.rel_err(outs[e][(l, b)][hq], o_ref)
                    rec["attn_max_rel_err"] = max(rec["attn_max_rel_err"], err)
                    assert err <= 2e-3, (lead, b, h, e, l, hq)
        H.log_parity("full_size_sampled", **rec)


def test_full_size_32k_sampled():
    """The 32k-token LLaMA-3-8B GQA workload at full size (32 layers, 8 kv
    heads, 8192 kept tokens, a three-level pyramid), 20 decode steps: the
    16th append fills the first tail cluster, so the selections of the last
    four steps read a pyramid the decode step sealed."""
    _full_size_sampled(synth.C5, 20, lambda eng, x: [(eng.leaders[2], 0, 3), (eng.leaders[-1], 0, 7)])


def test_needles_survive_at_32k():
    """The 32k-token workload's check: every planted needle token of every
    leader layer and kv head is kept by the static eviction, and its cluster
    is selected at every one of the 256 decode steps (10 leaders x 8 kv heads
    x 256 steps, all on the GPU path the benchmark times)."""
    w = synth.C5
    E = w.decode_steps
    x = synth.generate(w, H.window_rows_for(w), device="cuda", decode_steps=E)
    eng = H.make_engine(w, E)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda())
    sels = torch.empty((E,) + tuple(eng.sel.shape), dtype=torch.int32, device="cuda")
    for e in range(E):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
        sels[e].copy_(eng.sel)
    assert mpcache.device_status() == 0
    kept = eng.kept.cpu().numpy()
    sels = sels.cpu().numpy()
    n_keep = int(eng.n_keep[0])
    missing_kept = missing_sel = units = 0
    for lead in eng.leaders:
        grp = eng.group_of[lead]
        for h in range(w.n_kv_heads):
            p0 = int(x.needle_pos[lead, 0, h])
            pos = kept[grp, 0, h, :n_keep]
            rows = np.searchsorted(pos, np.arange(p0, p0 + w.needle_len))
            found = (rows < n_keep) & (pos[np.minimum(rows, n_keep - 1)] == np.arange(p0, p0 + w.needle_len))
            missing_kept += int((~found).sum())
            clusters = np.unique(rows[found] // w.cluster_size)
            for e in range(E):
                units += 1
                missing_sel += len(set(clusters.tolist()) - set(sels[e, grp, 0, h].tolist()))
    H.log_parity("needles_32k", leaders=len(eng.leaders), kv_heads=w.n_kv_heads, steps=E, units=units,
                 needle_tokens_not_kept=missing_kept, needle_clusters_not_selected=missing_sel)
    assert missing_kept == 0
    assert missing_sel == 0


def test_full_size_batch32_paged_sampled():
    """The batch-32 paged LLaMA-2-7B workload at full size (32 sequences of
    1024-4096 tokens, pages of 16 with a shuffled page table, 17 leaders),
    three decode steps; the sampled sequences are the shortest and the
    longest of the batch."""
    def pick(eng, x):
        lens = x.prompt_lens.tolist()
        bs, bl = lens.index(min(lens)), lens.index(max(lens))
        return [(eng.leaders[3], bs, 5), (eng.leaders[-1], bl, 30)]
    _full_size_sampled(synth.C4, 3, pick)


def test_full_size_2k_mha_sampled():
    """The 2k-token LLaMA-2-7B MHA workload at full size (32 layers, 32 kv
    heads, a two-level pyramid, groups of two layers), three decode steps."""
    _full_size_sampled(synth.C2, 3, lambda eng, x: [(eng.leaders[1], 0, 0), (eng.leaders[-1], 0, 31)])


def test_full_size_8k_gqa_sampled():
    """The 8k-token LLaMA-3-8B GQA workload at full size (32 layers, 8 kv
    heads, a two-level pyramid, groups of four layers), 20 decode steps (a
    tail cluster is sealed at the 16th)."""
    _full_size_sampled(synth.C3, 20, lambda eng, x: [(eng.leaders[0], 0, 1), (eng.leaders[-2], 0, 6)])


@pytest.mark.parametrize("batch", [1, 4, 16])
def test_full_size_paged_batches_sampled(batch):
    """The paged LLaMA-2-7B workload at the sweep's other batch sizes (prompts
    of 1024-4096 tokens, pages of 16 with a shuffled page table), four decode
    steps; the sampled sequences are the shortest and the longest."""
    def pick(eng, x):
        lens = x.prompt_lens.tolist()
        bs, bl = lens.index(min(lens)), lens.index(max(lens))
        return [(eng.leaders[1], bs, 2), (eng.leaders[-1], bl, 29)]
    _full_size_sampled(synth.WORKLOADS[f"c4_llama2_7b_paged_b{batch}"], 4, pick)


def test_pipeline_prompt_shorter_than_a_cluster():
    """Degenerate start: 12 prompt tokens (< s = 16), so the pyramid is empty
    and selection has no candidate; attention covers the tail alone until the
    decode appends seal the first cluster (step 4), after which it becomes
    selectable."""
    w = synth.C3.replace(n_layers=2, prompt_len=12, prompt_len_min=12, n_q_heads=4, n_kv_heads=2,
                         keep_ppm=1_000_000, fanouts=(2,), share_every=1)
    _pipeline(w, 24, [0, 1], max_skip=0.0)


def test_decode_past_capacity_is_refused_and_flagged():
    """A decode step with no cache row left for its append is refused on the
    device: no row is written, the token count stays, and the status word
    reports it (flag 2) until read."""
    w = synth.C3.replace(n_layers=1, prompt_len=32, prompt_len_min=32, n_q_heads=2, n_kv_heads=1,
                         keep_ppm=1_000_000, fanouts=(), level_keep_ppm=(500_000,), share_every=1)
    x = H.to_cuda(synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=34))
    eng = H.make_engine(w, 2)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda(), None, w.page_size)
    cap = eng.cap_tokens
    steps = cap - 32
    for e in range(steps):
        eng.decode_step(x.q[e], x.k_new[e], x.v_new[e])
    assert mpcache.device_status() == 0
    assert int(eng.n_tok[0]) == cap
    kc = eng.kc.clone()
    eng.decode_step(x.q[steps], x.k_new[steps], x.v_new[steps])
    assert mpcache.device_status() & 2
    assert int(eng.n_tok[0]) == cap
    assert torch.equal(eng.kc, kc)
    assert mpcache.device_status() == 0  # read and cleared


def test_corrupt_indices_are_reported_not_followed():
    """Indices outside their range (a selected cluster id past the sealed
    clusters, a kept position past the prompt) are reported in the device
    status word (flag 4) and never used as addresses: the outputs stay
    finite and the status clears once read."""
    w = synth.C3.replace(n_layers=1, prompt_len=256, prompt_len_min=256, n_q_heads=2, n_kv_heads=1,
                         keep_ppm=1_000_000, fanouts=(), level_keep_ppm=(250_000,), share_every=1)
    x = H.to_cuda(synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=2))
    eng = H.make_engine(w, 2)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda(), None, w.page_size)
    assert mpcache.device_status() == 0
    # a selected id past the 16 sealed clusters
    eng.select(x.q[0])
    eng.sel[0, 0, 0, 0] = 1_000_000
    eng.attend(x.q[0], x.k_new[0], x.v_new[0], advance=False)
    assert mpcache.device_status() & 4
    assert torch.isfinite(eng.out).all()
    assert mpcache.device_status() == 0
    # a kept position past the prompt
    eng.kept[0, 0, 0, 5] = 1_000_000
    eng.build_clusters(x.k, x.v, None, w.page_size)
    assert mpcache.device_status() & 4
    assert mpcache.device_status() == 0


@pytest.mark.parametrize("kind", [0, 1])
def test_bounded_wait_runs_out_and_reports(kind):
    """A wait that nothing satisfies (an mbarrier, or a flag that nothing
    sets) gives up after its limit, sets flag 1 of the status word and
    returns; the context stays usable for the next call."""
    never = torch.zeros(1, dtype=torch.int32, device="cuda")
    assert mpcache.device_status() == 0
    mpcache.selftest_wait(kind, 2000, never)
    assert mpcache.device_status() & 1
    assert mpcache.device_status() == 0
    x = torch.arange(8, device="cuda") * 2  # the context still runs work
    assert int(x.sum()) == 56
