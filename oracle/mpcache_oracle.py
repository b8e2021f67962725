"""Plain fp64 CPU oracle of the MPCache decode path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  It shares no code with the CUDA library or its Python binding; it reads
inputs drawn by the seeded generator and computes every step of the method in
float64 with numpy, in the order of the paper's Algorithm 2:

Step 1 (prefill, once):
  * look-once static eviction (Sec. 3.2 "Look-once static KV cache eviction";
    App. E "Static eviction"): softmax attention map of the last 20% prompt
    queries (10% for prompts longer than 24k tokens) against all keys, summed
    per key column; the highest-scoring tokens are kept, the rest dropped;
  * leader layers score, the other layers of a sharing group reuse the
    leader's kept set (cross-layer index sharing, Sec. 3.4);
  * the kept keys/values are gathered (token gathering, Alg. 1).
Step 2 (every decode step e, every layer l):
  * append k, v to the cache (decoding stage, App. A);
  * leader layers: cluster similarity Sim(q, K_c) = q . (alpha r_max +
    (1 - alpha) r_min) (linearised and reordered bound, Eq. 3) with r_max /
    r_min the per-channel max / min of the cluster keys (Sec. 3.3), hierarchical
    top-k from the coarsest to the finest level among the children of the kept
    parents (Sec. 3.3 "Hierarchical KV cache clustering"); other layers reuse
    the leader's ids (Sec. 3.4);
  * softmax(q K'^T / sqrt(d)) V' over the gathered tokens (Alg. 1).

Readings of points the paper leaves open (the same readings as the CUDA
path's, each implemented here on its own):
  * the static map uses the model's own 1/sqrt(d) scale and a causal mask;
  * window w = ceil(rho_w T), rho_w = 0.2, or 0.1 when T > 24576;
  * one kept set per (sequence, kv head); GQA sums the group's query heads;
  * counts are n = min(N, max(1, ceil(ratio N))), ratios in parts per million;
  * ties rank the lower index first;
  * clusters are consecutive runs of s kept tokens in position order; the
    partial remainder (< s tokens) is the tail, always attended and not
    selectable; coarser levels group f consecutive children, the last group
    may be partial; a coarse summary is the max / min over all member tokens;
  * GQA selection scores (sum_g q_g) . rep once per kv head;
  * sharing: layers 0 and 1 lead themselves; for l >= 2 the leader is
    2 + m * floor((l - 2) / m);
  * fixed-point Eq. 3 (the ring arithmetic of App. B emulated on plaintext
    values): f = 18 fractional bits unless given, enc(x) = rint(x 2^f) with
    ties to even, truncation by floor after each product and once per dot
    product, alpha and 1 - alpha encoded as public constants, scores
    saturated to int32 for ranking.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np

PPM = 10 ** 6


# ---------------------------------------------------------------- counts ----

def ceil_ratio(n: int, ppm: int) -> int:
    """ceil(n * ppm / 1e6) in exact integer arithmetic."""
    return -(-int(n) * int(ppm) // PPM)


def window_length(T: int, window_ppm: int = 200_000, long_ppm: int = 100_000,
                  long_threshold: int = 24_576) -> int:
    """Rows of the static-eviction window: the last 20% of the prompt, 10% when
    the prompt is longer than 24k tokens (Sec. 3.2; App. E "Static eviction")."""
    ppm = long_ppm if T > long_threshold else window_ppm
    return min(T, max(1, ceil_ratio(T, ppm)))


def kept_count(T: int, keep_ppm: int) -> int:
    """Static budget: tokens kept out of T (Alg. 2 Step 1)."""
    if T == 0:
        return 0
    return min(T, max(1, ceil_ratio(T, keep_ppm)))


def selected_count(n_clusters: int, keep_ppm: int, n_candidates: int) -> int:
    """Clusters kept at one level: k = ceil(size * eta) (Alg. 2 topk), clamped
    to the candidates that the coarser level left."""
    if n_clusters == 0 or n_candidates == 0:
        return 0
    return min(n_candidates, max(1, ceil_ratio(n_clusters, keep_ppm)))


def leader_of(layer: int, share_every: int) -> int:
    """Cross-layer index sharing (Sec. 3.4): groups of ``share_every`` adjacent
    layers reuse the first layer's indices; the first two layers lead
    themselves."""
    if share_every <= 1 or layer < 2:
        return layer
    return 2 + share_every * ((layer - 2) // share_every)


def level_keep_fractions(eta_ppm: int, n_levels: int) -> List[int]:
    """Cumulative kept fraction per level, finest first (App. E "KV cache
    clustering configuration": coarse levels drop half of their clusters when
    the final ratio is below 0.5).  Level l >= 2 keeps max(eta, 0.5^(n-l+1)),
    the finest level keeps eta."""
    out = [int(eta_ppm)]
    for lvl in range(2, n_levels + 1):
        half_pow = PPM >> (n_levels - lvl + 1)
        out.append(max(int(eta_ppm), half_pow))
    return out


# ------------------------------------------------------ static eviction ----

def accumulated_attention(q_win: np.ndarray, k: np.ndarray, scale: float,
                          row_chunk: int = 512) -> np.ndarray:
    """Accumulated window attention per key (Sec. 3.2; Alg. 2 Step 1).

    q_win: [G][w][d] queries of prompt positions T-w .. T-1 (all query heads
    of one kv group); k: [T][d].  Returns score[T] = sum over the group's heads
    and the window rows i of softmax_j(q_i . k_j * scale), j <= T - w + i.
    """
    q_win = np.asarray(q_win, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    G, w, _ = q_win.shape
    T = k.shape[0]
    score = np.zeros(T, dtype=np.float64)
    cols = np.arange(T)
    for g in range(G):
        for r0 in range(0, w, row_chunk):
            r1 = min(w, r0 + row_chunk)
            pos = T - w + np.arange(r0, r1)
            logits = (q_win[g, r0:r1] @ k.T) * scale
            logits = np.where(cols[None, :] <= pos[:, None], logits, -np.inf)
            logits -= logits.max(axis=1, keepdims=True)
            p = np.exp(logits)
            p /= p.sum(axis=1, keepdims=True)
            score += p.sum(axis=0)
    return score


def rank_desc(scores: np.ndarray, ids: Optional[np.ndarray] = None) -> np.ndarray:
    """Order of ``ids`` by score descending, lower id first on equal scores."""
    scores = np.asarray(scores, dtype=np.float64)
    if ids is None:
        ids = np.arange(len(scores))
    return np.asarray(ids)[np.lexsort((np.asarray(ids), -scores))]


def static_evict(score: np.ndarray, n_keep: int) -> np.ndarray:
    """Keep the n_keep highest accumulated scores (drop the UIA tokens);
    positions returned in ascending order (Alg. 2 static_evict)."""
    return np.sort(rank_desc(score)[:n_keep])


# --------------------------------------------------- cluster summaries ----

@dataclass
class Level:
    members: List[np.ndarray]   # token indices (into the kept cache) per cluster
    r_max: np.ndarray           # [C][d]
    r_min: np.ndarray           # [C][d]
    rep: np.ndarray             # [C][d] alpha r_max + (1 - alpha) r_min
    mean: np.ndarray = None     # [C][d] mean of the member keys (average baseline)


def cluster_pyramid(keys: np.ndarray, s: int, fanouts: Sequence[int],
                    alpha: float) -> List[Level]:
    """Hierarchical clusters of the cache keys, finest level first.

    keys: [N][d] cache keys in position order.  Level 1: cluster c holds
    tokens [c s, (c+1) s) for c < floor(N / s) (adjacent tokens, Sec. 3.3; the
    partial remainder is the tail).  Level l+1 groups f_l consecutive level-l
    clusters.  r_max / r_min are the channel-wise max / min over all member
    tokens (Sec. 3.3, Eq. 2), rep the reordered representative of Eq. 3 and
    mean the average member key (the average baseline of App. G).
    """
    keys = np.asarray(keys, dtype=np.float64)
    n_full = keys.shape[0] // s
    members = [np.arange(c * s, (c + 1) * s) for c in range(n_full)]
    levels: List[Level] = []
    for lvl in range(1 + len(fanouts)):
        d = keys.shape[1]
        if members:
            r_max = np.stack([keys[m].max(axis=0) for m in members])
            r_min = np.stack([keys[m].min(axis=0) for m in members])
            mean = np.stack([keys[m].mean(axis=0) for m in members])
        else:
            r_max = np.zeros((0, d))
            r_min = np.zeros((0, d))
            mean = np.zeros((0, d))
        rep = alpha * r_max + (1.0 - alpha) * r_min
        levels.append(Level(members, r_max, r_min, rep, mean))
        if lvl < len(fanouts):
            f = fanouts[lvl]
            n_up = -(-len(members) // f)
            members = [np.concatenate(members[p * f:(p + 1) * f]) for p in range(n_up)]
    return levels


# ------------------------------------------- fixed-point emulation ----
# The MPC runtime evaluates Eq. 3 on secret shares of fixed-point values in
# the ring Z_{2^64} (App. B: arithmetic sharing with l = 64).  In plaintext
# the shares add up to the value itself, so the arithmetic is emulated here
# on the values: x is encoded as rint(x 2^f) (f fractional bits, the ring's
# two's-complement representative), sums are ring sums, and a product of two
# encodings carries 2f fractional bits until one truncation (an arithmetic
# shift right by f, i.e. floor) brings it back to f.  A dot product is one
# ring sum of products truncated once.

FXP_FRAC_BITS = 18  # default fractional bits of the encoding


def fxp_encode(x, frac_bits: int = FXP_FRAC_BITS) -> np.ndarray:
    """rint(x 2^f) (round half to even) as int64; |x| must stay below 2^(62-f)."""
    v = np.rint(np.asarray(x, dtype=np.float64) * float(1 << frac_bits))
    if np.any(np.abs(v) >= 2.0 ** 62):
        raise ValueError("value out of the fixed-point range")
    return v.astype(np.int64)


def fxp_dot(a: np.ndarray, b: np.ndarray, frac_bits: int = FXP_FRAC_BITS) -> np.ndarray:
    """Truncated ring dot product over the last axis: floor((sum_i a_i b_i
    mod 2^64) / 2^f).  numpy int64 products and sums wrap modulo 2^64, and
    >> on int64 is the arithmetic (floor) shift."""
    with np.errstate(over="ignore"):
        return (np.asarray(a, dtype=np.int64) * np.asarray(b, dtype=np.int64)).sum(axis=-1) >> frac_bits


def sim_fxp(q_group: np.ndarray, r_max: np.ndarray, r_min: np.ndarray, alpha: float,
            frac_bits: int = FXP_FRAC_BITS) -> np.ndarray:
    """Eq. 3 in the ring, per cluster c (rows of r_max / r_min, [C][d]):
      q_i     = sum_g enc(q_gi)                         (ring sum)
      rep_ci  = dot(enc(alpha), enc(r_max_ci)) + dot(enc(1 - alpha), enc(r_min_ci))
      sim_c   = dot(q, rep_c)
    with alpha and 1 - alpha public constants encoded like any value (each
    product of rep is a one-term dot, truncated on its own).  Returns the
    int64 scores (units of 2^-f) saturated to the int32 range."""
    d = np.shape(q_group)[-1]
    q = fxp_encode(q_group, frac_bits).reshape(-1, d).sum(axis=0)
    ea = fxp_encode([alpha], frac_bits)
    eb = fxp_encode([1.0 - alpha], frac_bits)
    emax = fxp_encode(r_max, frac_bits).reshape(-1, d)
    emin = fxp_encode(r_min, frac_bits).reshape(-1, d)
    rep = fxp_dot(emax[..., None], ea[None], frac_bits) + fxp_dot(emin[..., None], eb[None], frac_bits)
    sc = fxp_dot(q[None, :], rep, frac_bits)
    return np.clip(sc, -(1 << 31), (1 << 31) - 1)


def hierarchical_select(q_group: np.ndarray, levels: List[Level],
                        fanouts: Sequence[int], level_keep_ppm: Sequence[int],
                        trace: Optional[list] = None, metric: str = "eq3",
                        alpha: float = 0.6, frac_bits: int = FXP_FRAC_BITS) -> np.ndarray:
    """Coarse-to-fine cluster selection (Sec. 3.3; Alg. 2 Sim + topk).

    q_group: [G][d] decode queries of one kv group, scored through their sum
    q = sum_g q_g.  The similarity of cluster c is q . rep_c (Eq. 3, the
    default); with metric="bound", the upper bound of Eq. 2,
    sum_i max(q_i r_max_ci, q_i r_min_ci), evaluated on the same summed query;
    with metric="mean", q . mean_c (the average-key baseline of App. G);
    with metric="fxp", Eq. 3 in the fixed-point ring (sim_fxp, weight
    ``alpha``, ``frac_bits`` fractional bits), ranked as integers.
    At the coarsest level every cluster is a candidate; at each finer level
    the candidates are the children of the kept parents.  Returns the kept
    finest-level ids in ascending order.  ``trace``, if given, receives per
    level (coarsest first) the candidate ids, their similarities and k, for
    tests that need the margin at each cut.
    """
    if metric not in ("eq3", "bound", "mean", "fxp"):
        raise ValueError(metric)
    qsum = np.asarray(q_group, dtype=np.float64).sum(axis=0)
    n = len(levels)
    cand = np.arange(levels[-1].rep.shape[0])
    kept = cand
    for lvl in range(n - 1, -1, -1):
        lev = levels[lvl]
        if not len(cand):
            sim = np.zeros(0)
        elif metric == "eq3":
            sim = lev.rep[cand] @ qsum
        elif metric == "mean":
            sim = lev.mean[cand] @ qsum
        elif metric == "fxp":
            sim = sim_fxp(q_group, lev.r_max[cand], lev.r_min[cand], alpha, frac_bits).astype(np.float64)
        else:
            sim = np.maximum(lev.r_max[cand] * qsum, lev.r_min[cand] * qsum).sum(axis=1)
        k = selected_count(lev.rep.shape[0], level_keep_ppm[lvl], len(cand))
        if trace is not None:
            trace.append((np.asarray(cand), np.asarray(sim), k))
        kept = np.sort(rank_desc(sim, cand)[:k]) if k else np.zeros(0, dtype=np.int64)
        if lvl > 0:
            f = fanouts[lvl - 1]
            n_child = levels[lvl - 1].rep.shape[0]
            cand = np.array([c for p in kept for c in range(p * f, min((p + 1) * f, n_child))],
                            dtype=np.int64)
    return kept.astype(np.int64)


# ---------------------------------------------------- sparse attention ----

def sparse_attention(q: np.ndarray, k_sel: np.ndarray, v_sel: np.ndarray,
                     scale: float) -> np.ndarray:
    """softmax(q K'^T * scale) V' over the gathered tokens (Alg. 1)."""
    q = np.asarray(q, dtype=np.float64)
    logits = (np.asarray(k_sel, dtype=np.float64) @ q) * scale
    logits -= logits.max()
    p = np.exp(logits)
    p /= p.sum()
    return p @ np.asarray(v_sel, dtype=np.float64)


def attended_tokens(n_tok: int, s: int, sel: np.ndarray) -> np.ndarray:
    """Cache indices attended at a step whose cache held n_tok tokens before
    the append: every token of the selected clusters plus the tail, which
    includes the token appended at this step."""
    n_full = n_tok // s
    toks = [np.arange(c * s, (c + 1) * s) for c in np.asarray(sel, dtype=np.int64)]
    toks.append(np.arange(n_full * s, n_tok + 1))
    return np.concatenate(toks).astype(np.int64)


# ------------------------------------------------------ metric variants ----

def sim_max_dot(q: np.ndarray, keys: np.ndarray) -> float:
    """Exact maximum dot product of a cluster (Eq. 1, left side)."""
    return float((np.asarray(keys, np.float64) @ np.asarray(q, np.float64)).max())


def sim_bound(q: np.ndarray, r_max: np.ndarray, r_min: np.ndarray) -> float:
    """Upper bound of Eq. 2: sum_i max(q_i r_max_i, q_i r_min_i)."""
    q = np.asarray(q, np.float64)
    return float(np.maximum(q * r_max, q * r_min).sum())


def sim_linear(q: np.ndarray, r_max: np.ndarray, r_min: np.ndarray, alpha: float) -> float:
    """Linearised similarity before reordering: sum_i alpha q_i r_max_i +
    (1 - alpha) q_i r_min_i (Sec. 3.3, the step before Eq. 3)."""
    q = np.asarray(q, np.float64)
    return float((alpha * q * r_max + (1.0 - alpha) * q * r_min).sum())


def sim_average(q: np.ndarray, keys: np.ndarray) -> float:
    """Average-key similarity, the rejected baseline (App. G, Fig. avg vs MP)."""
    return float(np.asarray(q, np.float64) @ np.asarray(keys, np.float64).mean(axis=0))


def commonality(indices: Sequence[Sequence[int]], k: int, m: int) -> float:
    """Commonality score of m adjacent layers (Sec. 2, Observation 3):
    1 / (k (L - m)) * sum_l |intersection_{i=l}^{l+m} idx_i[:k]|."""
    L = len(indices)
    total = 0
    for l in range(L - m):
        inter = set(list(indices[l])[:k])
        for i in range(l + 1, l + m + 1):
            inter &= set(list(indices[i])[:k])
        total += len(inter)
    return total / (k * (L - m))


def selected_positions(kept: Sequence[int], prompt_len: int, selected: Sequence[int], s: int) -> List[int]:
    """Token positions of the selected clusters (the idx sets of the
    commonality score, Sec. 2 Observation 3, for a layer with its own static
    eviction): cluster c holds cache rows c s .. c s + s - 1; a row r below
    len(kept) is the kept prompt token kept[r], a later row is the token
    appended at position prompt_len + r - len(kept) (App. A decode append)."""
    n_keep = len(kept)
    out = []
    for c in selected:
        for r in range(int(c) * s, int(c) * s + s):
            out.append(int(kept[r]) if r < n_keep else prompt_len + r - n_keep)
    return sorted(out)


# ------------------------------------------------------- full pipeline ----

@dataclass
class Params:
    """Hyper-parameters of one run (same meaning as the workload fields)."""
    keep_ppm: int
    cluster_size: int
    fanouts: Sequence[int]
    level_keep_ppm: Sequence[int]
    share_every: int
    alpha: float = 0.6
    window_ppm: int = 200_000
    long_window_ppm: int = 100_000
    long_prompt_threshold: int = 24_576
    scale: Optional[float] = None


@dataclass
class Result:
    scores: Dict[tuple, np.ndarray] = field(default_factory=dict)      # (l, b, h) leaders
    kept: Dict[tuple, np.ndarray] = field(default_factory=dict)        # (l, b, h) all layers
    selected: Dict[tuple, np.ndarray] = field(default_factory=dict)    # (e, l, b, h) all layers
    out: Dict[tuple, np.ndarray] = field(default_factory=dict)         # (e, l, b) -> [Hq][d]
    levels: Dict[tuple, List[Level]] = field(default_factory=dict)     # (e, l, b, h) leaders
    cache_k: Dict[tuple, np.ndarray] = field(default_factory=dict)     # (l, b, h) after prefill


def run(prompt_k, prompt_v, q_win, q, k_new, v_new, prompt_lens, p: Params,
        steps: Optional[int] = None, layers: Optional[Sequence[int]] = None,
        keep_levels: bool = False) -> Result:
    """Whole method on one batch, following Alg. 2.

    prompt_k/prompt_v: callables (l, b) -> [Hkv][T_b][d] arrays;
    q_win: callable (l, b) -> [Hq][R][d] with row r at position T_b - R + r;
    q, k_new, v_new: callables (e, l, b) -> [H][d].
    ``layers`` restricts Step 2 to a subset (their leaders are always run).
    """
    res = Result()
    n_layers_total = None
    lens = [int(t) for t in prompt_lens]
    B = len(lens)
    if layers is None:
        raise ValueError("pass the layer list")
    want = sorted(set(layers) | {leader_of(l, p.share_every) for l in layers})
    s = p.cluster_size

    # Step 1: look-once static eviction during prefill
    caches = {}
    for l in want:
        lead = leader_of(l, p.share_every)
        for b in range(B):
            K = np.asarray(prompt_k(l, b), dtype=np.float64)
            V = np.asarray(prompt_v(l, b), dtype=np.float64)
            Hkv, T, d = K.shape
            scale = p.scale if p.scale is not None else 1.0 / np.sqrt(d)
            for h in range(Hkv):
                if lead == l:
                    Q = np.asarray(q_win(l, b), dtype=np.float64)
                    Hq, R = Q.shape[0], Q.shape[1]
                    G = Hq // Hkv
                    w = window_length(T, p.window_ppm, p.long_window_ppm, p.long_prompt_threshold)
                    qg = Q[h * G:(h + 1) * G, R - w:R]
                    score = accumulated_attention(qg, K[h], scale)
                    res.scores[(l, b, h)] = score
                    res.kept[(l, b, h)] = static_evict(score, kept_count(T, p.keep_ppm))
                else:
                    res.kept[(l, b, h)] = res.kept[(lead, b, h)]
                idx = res.kept[(l, b, h)]
                caches[(l, b, h)] = [K[h][idx].copy(), V[h][idx].copy()]
                res.cache_k[(l, b, h)] = caches[(l, b, h)][0].copy()

    # Step 2: query-aware dynamic selection during decoding
    E = steps if steps is not None else 0
    for e in range(E):
        for l in want:
            lead = leader_of(l, p.share_every)
            for b in range(B):
                Qd = np.asarray(q(e, l, b), dtype=np.float64)
                kn = np.asarray(k_new(e, l, b), dtype=np.float64)
                vn = np.asarray(v_new(e, l, b), dtype=np.float64)
                Hq, d = Qd.shape
                Hkv = kn.shape[0]
                G = Hq // Hkv
                scale = p.scale if p.scale is not None else 1.0 / np.sqrt(d)
                out = np.zeros((Hq, d))
                for h in range(Hkv):
                    ck, cv = caches[(l, b, h)]
                    n_tok = ck.shape[0]
                    ck = np.vstack([ck, kn[h][None]])
                    cv = np.vstack([cv, vn[h][None]])
                    caches[(l, b, h)] = [ck, cv]
                    if lead == l:
                        levels = cluster_pyramid(ck[:n_tok], s, p.fanouts, p.alpha)
                        sel = hierarchical_select(Qd[h * G:(h + 1) * G], levels,
                                                  p.fanouts, p.level_keep_ppm)
                        if keep_levels:
                            res.levels[(e, l, b, h)] = levels
                    else:
                        sel = res.selected[(e, lead, b, h)]
                    res.selected[(e, l, b, h)] = sel
                    toks = attended_tokens(n_tok, s, sel)
                    for g in range(G):
                        out[h * G + g] = sparse_attention(Qd[h * G + g], ck[toks], cv[toks], scale)
                res.out[(e, l, b)] = out
    return res
