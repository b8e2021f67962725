"""Seeded synthetic workloads for the MPCache decode path.

This module only *draws inputs*: prompt keys/values, the window queries of the
prompt's last rows, and the per-step decode query/key/value.  It contains none
of the method's arithmetic (no softmax, no ranking, no clustering), so both the
CUDA path and the fp64 oracle may take their inputs from it.

The five workloads mirror the model shapes the paper evaluates on (GPT-2 small,
LLaMA-2-7B, LLaMA-3-8B GQA; Sec. 5 and App. E) with activations replaced by the
seeded distributions described in ``Workload.rule``:

* ``iid``      Q, K, V ~ N(0, 1); key 0 scaled by 4 as an attention sink.
* ``outlier``  K ~ N(0, 1) with 4 seeded outlier channels per (layer, kv head)
               scaled by 8; V ~ N(0, 1).  Each (layer, b, kv head) owns a seeded
               5% subset S of prompt positions; every window/decode query is
               q = 0.7 * k_j + 0.714 * n with j ~ U(S), n ~ N(0, I).
* ``needle``   ``outlier`` plus, per (layer, b, kv head), one contiguous 64-token
               passage at a seeded depth in [0.1 T, 0.9 T) whose keys are
               3 u + 0.5 n, u a random direction of norm sqrt(d); every query is
               q = 0.35 * k_j + 0.7 * u + 0.622 * n (the needle direction
               dominates, as a question about the planted passage would).

``layer_rho_ppm`` = rho > 0 (``outlier`` and ``needle``) chains the layers of
a sequence the way a residual stream would (Sec. 2, Observation 3): layer l's
keys are rho K_{l-1} + sqrt(1 - rho^2) K_fresh (after the outlier scaling),
slot i of its subset S keeps layer l-1's position with probability rho (else
a fresh position), and the slot each window/decode query targets is drawn
from one stream per sequence, shared by all layers.  rho = 0 (the default)
draws every layer independently.

Layouts (all row-major, head_dim innermost):

* dense prompt K/V: ``[L][B][Hkv][T_max][d]``; positions >= T_b are zero.
* paged prompt K/V: pool ``[L][n_pages][Hkv][page][d]`` plus
  ``page_table[B][max_pages]`` (int32, shuffled page ids, -1 unused).
* window queries: ``[L][B][Hq][R][d]``; row r holds the query of prompt position
  ``T_b - R + r`` (rows aligned to the end of every prompt).
* decode tensors: ``q[E][L][B][Hq][d]``, ``k_new``/``v_new`` ``[E][L][B][Hkv][d]``.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass
from typing import Optional, Tuple

import torch

PPM = 1_000_000


@dataclass(frozen=True)
class Workload:
    """Shape and hyper-parameters of one synthetic MPCache workload.

    Ratios are integers in parts per million so that every count derived from
    them is exact integer arithmetic on both sides of the parity tests.
    ``level_keep_ppm[i]`` is the fraction of level-(i+1) clusters that survive
    selection (level 1 = finest, s tokens per cluster); ``fanouts[i]`` is the
    number of level-(i+1) clusters grouped under one level-(i+2) cluster.
    """

    name: str
    n_layers: int
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    dtype: str                      # "f32" or "bf16"
    prompt_len: int                 # T (max T when ragged)
    prompt_len_min: int             # == prompt_len unless ragged
    keep_ppm: int                   # static budget rho_s
    cluster_size: int               # s
    fanouts: Tuple[int, ...]        # children per coarser cluster, levels 2..n
    level_keep_ppm: Tuple[int, ...] # kept fraction per level, finest first
    share_every: int                # cross-layer sharing group size m
    decode_steps: int               # E
    rule: str                       # "iid" | "outlier" | "needle"
    paged: bool = False
    page_size: int = 16
    seed: int = 1000
    window_ppm: int = 200_000       # last 20% of the prompt
    long_window_ppm: int = 100_000  # 10% for long prompts
    long_prompt_threshold: int = 24_576
    alpha: float = 0.6
    needle_len: int = 64
    layer_rho_ppm: int = 0          # cross-layer correlation (0: independent layers)

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def n_levels(self) -> int:
        return 1 + len(self.fanouts)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads: GPT-2-small, LLaMA-2-7B, LLaMA-3-8B GQA, batched paged
# LLaMA-2-7B, 32k-token LLaMA-3-8B GQA with needles.
C1 = Workload("c1_gpt2_small_t512", 1, 1, 12, 12, 64, "f32", 512, 512,
              500_000, 16, (), (250_000,), 1, 8, "iid", seed=1001)
C2 = Workload("c2_llama2_7b_t2048", 32, 1, 32, 32, 128, "bf16", 2048, 2048,
              500_000, 16, (4,), (125_000, 500_000), 2, 64, "outlier", seed=1002)
C3 = Workload("c3_llama3_8b_gqa_t8192", 32, 1, 32, 8, 128, "bf16", 8192, 8192,
              250_000, 16, (8,), (100_000, 500_000), 4, 128, "outlier", seed=1003)
C4 = Workload("c4_llama2_7b_paged_b32", 32, 32, 32, 32, 128, "bf16", 4096, 1024,
              500_000, 16, (4,), (125_000, 500_000), 2, 32, "outlier",
              paged=True, seed=1004)
C5 = Workload("c5_llama3_8b_gqa_t32768_needles", 32, 1, 32, 8, 128, "bf16",
              32768, 32768, 250_000, 16, (8, 8), (50_000, 250_000, 500_000), 4,
              256, "needle", seed=1005)

C4_BATCHES = (1, 4, 16, 32)
# the batched paged workload at its other batch sizes (same seed and rule)
C4_VARIANTS = tuple(C4.replace(name=f"c4_llama2_7b_paged_b{b}", batch=b) for b in C4_BATCHES if b != C4.batch)
# The token-wise comparator (LongCache-style dynamic selection of single
# tokens, no static eviction) on the 8k and 32k shapes: every prompt token
# kept, clusters of one token under groups of 16, and as many selected tokens
# as the clustered workload attends in selected clusters (13 and 26 clusters
# of 16); the groups' level keeps 10% (8k) or 5% (32k) of them.
C3_TOKENWISE = C3.replace(name="c3_tokenwise_t8192", keep_ppm=1_000_000, cluster_size=1, fanouts=(16,),
                          level_keep_ppm=(25_391, 100_000))
C5_TOKENWISE = C5.replace(name="c5_tokenwise_t32768_needles", keep_ppm=1_000_000, cluster_size=1, fanouts=(16,),
                          level_keep_ppm=(12_695, 50_000))
WORKLOADS = {w.name: w for w in (C1, C2, C3, C4, C5) + C4_VARIANTS + (C3_TOKENWISE, C5_TOKENWISE)}


@dataclass
class Inputs:
    """Tensors of one workload (see the module docstring for layouts)."""

    work: Workload
    prompt_lens: torch.Tensor          # int32 [B] (host)
    k: torch.Tensor                    # dense [L][B][Hkv][T][d] or pool
    v: torch.Tensor
    page_table: Optional[torch.Tensor] # int32 [B][max_pages] or None
    q_win: torch.Tensor                # [L][B][Hq][R][d]
    q: torch.Tensor                    # [E][L][B][Hq][d]
    k_new: torch.Tensor                # [E][L][B][Hkv][d]
    v_new: torch.Tensor
    needle_pos: Optional[torch.Tensor] # int32 [L][B][Hkv] start of the passage

    def dense_kv(self, layer: int, b: int):
        """Prompt K/V of (layer, b) as [Hkv][T_b][d] (gathered from pages)."""
        T = int(self.prompt_lens[b])
        if self.page_table is None:
            return self.k[layer, b, :, :T], self.v[layer, b, :, :T]
        P = self.work.page_size
        n = (T + P - 1) // P
        pages = self.page_table[b, :n].long().to(self.k.device)
        kk = self.k[layer, pages].permute(1, 0, 2, 3).reshape(self.k.shape[2], n * P, -1)
        vv = self.v[layer, pages].permute(1, 0, 2, 3).reshape(self.v.shape[2], n * P, -1)
        return kk[:, :T], vv[:, :T]


def _torch_dtype(name: str) -> torch.dtype:
    return {"f32": torch.float32, "bf16": torch.bfloat16}[name]


class _Streams:
    """One independent torch generator per (layer, tensor) stream."""

    def __init__(self, seed: int, device: torch.device):
        self.seed = seed
        self.device = device

    def gen(self, layer: int, tensor: int) -> torch.Generator:
        g = torch.Generator(device=self.device)
        g.manual_seed((self.seed * 1_000_003 + layer * 7919 + tensor * 104_729) % (2**62))
        return g


def prompt_lengths(work: Workload) -> torch.Tensor:
    """Per-sequence prompt lengths (uniform in [min, max] when ragged)."""
    if work.prompt_len_min == work.prompt_len:
        return torch.full((work.batch,), work.prompt_len, dtype=torch.int32)
    g = torch.Generator().manual_seed(work.seed * 31 + 7)
    return torch.randint(work.prompt_len_min, work.prompt_len + 1, (work.batch,),
                         generator=g, dtype=torch.int64).to(torch.int32)


def generate(work: Workload, window_rows: int, device="cpu",
             decode_steps: Optional[int] = None) -> Inputs:
    """Draw every input tensor of ``work`` on ``device``.

    ``window_rows`` (R) is how many trailing prompt rows of queries to draw per
    sequence; the caller passes at least the longest window it will score.
    ``decode_steps`` overrides ``work.decode_steps`` (tests use fewer steps).
    """
    device = torch.device(device)
    E = work.decode_steps if decode_steps is None else decode_steps
    L, B, Hq, Hkv, d = work.n_layers, work.batch, work.n_q_heads, work.n_kv_heads, work.head_dim
    G = Hq // Hkv
    T_max = work.prompt_len
    R = int(window_rows)
    lens = prompt_lengths(work)
    dt = _torch_dtype(work.dtype)
    st = _Streams(work.seed, device)
    f32 = dict(dtype=torch.float32, device=device)

    k_dense = torch.zeros((L, B, Hkv, T_max, d), dtype=dt, device=device)
    v_dense = torch.zeros((L, B, Hkv, T_max, d), dtype=dt, device=device)
    q_win = torch.zeros((L, B, Hq, R, d), dtype=dt, device=device)
    q_dec = torch.empty((E, L, B, Hq, d), dtype=dt, device=device)
    k_new = torch.empty((E, L, B, Hkv, d), dtype=dt, device=device)
    v_new = torch.empty((E, L, B, Hkv, d), dtype=dt, device=device)
    needle_pos = None
    if work.rule == "needle":
        needle_pos = torch.zeros((L, B, Hkv), dtype=torch.int32)

    rho = work.layer_rho_ppm / PPM
    prev = {}  # b -> (scaled keys, S) of the previous layer (rho > 0)
    for l in range(L):
        for b in range(B):
            T = int(lens[b])
            gk = st.gen(l, 1 + 16 * b)
            gv = st.gen(l, 2 + 16 * b)
            gq = st.gen(l, 3 + 16 * b)
            gs = st.gen(l, 4 + 16 * b)
            gd = st.gen(l, 5 + 16 * b)
            K = torch.randn((Hkv, T, d), generator=gk, **f32)
            V = torch.randn((Hkv, T, d), generator=gv, **f32)
            if work.rule == "iid":
                K[:, 0, :] *= 4.0
                k_dense[l, b, :, :T] = K.to(dt)
                v_dense[l, b, :, :T] = V.to(dt)
                rows = min(R, T)
                q_win[l, b, :, R - rows:] = torch.randn((Hq, rows, d), generator=gq, **f32).to(dt)
                q_dec[:, l, b] = torch.randn((E, Hq, d), generator=gd, **f32).to(dt)
                k_new[:, l, b] = torch.randn((E, Hkv, d), generator=gd, **f32).to(dt)
                v_new[:, l, b] = torch.randn((E, Hkv, d), generator=gd, **f32).to(dt)
                continue
            # outlier channels: 4 per kv head, scaled by 8 (prompt and decode keys)
            ch = torch.stack([torch.randperm(d, generator=gs, device=device)[:4] for _ in range(Hkv)])
            scale = torch.ones((Hkv, d), **f32)
            scale.scatter_(1, ch, 8.0)
            K = K * scale[:, None, :]
            if rho > 0 and b in prev:
                K = rho * prev[b][0] + (1.0 - rho * rho) ** 0.5 * K
            u = None
            if work.rule == "needle":
                u = torch.randn((Hkv, d), generator=gs, **f32)
                u = u / u.norm(dim=1, keepdim=True) * (d ** 0.5)
                lo = T // 10
                hi = max(lo + 1, (9 * T) // 10 - work.needle_len)
                start = torch.randint(lo, hi, (Hkv,), generator=gs, device=device)
                for h in range(Hkv):
                    s0 = int(start[h])
                    n = torch.randn((work.needle_len, d), generator=gs, **f32)
                    K[h, s0:s0 + work.needle_len] = 3.0 * u[h] + 0.5 * n
                    needle_pos[l, b, h] = s0
            Kq = K.to(dt)
            k_dense[l, b, :, :T] = Kq
            v_dense[l, b, :, :T] = V.to(dt)
            # 5% seeded position subset per kv head; queries follow its keys
            n_s = max(1, (T * 5 + 99) // 100)
            S = torch.stack([torch.randperm(T, generator=gs, device=device)[:n_s] for _ in range(Hkv)])
            if rho > 0:
                if b in prev:
                    stay = torch.rand((Hkv, n_s), generator=gs, device=device) < rho
                    S = torch.where(stay, prev[b][1], S)
                prev[b] = (K, S)
            Kf = Kq.float()
            # rho > 0: the targeted slots come from one stream per sequence
            gp = {"q": st.gen(0, 6 + 16 * b), "d": st.gen(0, 7 + 16 * b)} if rho > 0 else None

            def draw_q(count: int, gen: torch.Generator, which: str) -> torch.Tensor:
                # [Hq][count][d]: q = 0.7 k_j (+ 0.35 u) + noise
                pick = torch.randint(0, n_s, (Hq, count), generator=gen if gp is None else gp[which],
                                     device=device)
                kvh = torch.arange(Hq, device=device) // G
                j = S[kvh[:, None], pick]
                kj = Kf[kvh[:, None], j]
                noise = torch.randn((Hq, count, d), generator=gen, **f32)
                if u is None:
                    return 0.7 * kj + 0.714 * noise
                return 0.35 * kj + 0.7 * u[kvh][:, None, :] + 0.622 * noise

            rows = min(R, T)
            q_win[l, b, :, R - rows:] = draw_q(rows, gq, "q").to(dt)
            q_dec[:, l, b] = draw_q(E, gd, "d").permute(1, 0, 2).to(dt)
            kn = torch.randn((E, Hkv, d), generator=gd, **f32) * scale[None]
            k_new[:, l, b] = kn.to(dt)
            v_new[:, l, b] = torch.randn((E, Hkv, d), generator=gd, **f32).to(dt)

    page_table = None
    k_out, v_out = k_dense, v_dense
    if work.paged:
        P = work.page_size
        n_pages_b = [(int(t) + P - 1) // P for t in lens]
        total = sum(n_pages_b)
        max_pages = (T_max + P - 1) // P
        g = torch.Generator().manual_seed(work.seed * 131 + 3)
        perm = torch.randperm(total, generator=g).to(torch.int32)
        page_table = torch.full((B, max_pages), -1, dtype=torch.int32)
        k_out = torch.zeros((L, total, Hkv, P, d), dtype=dt, device=device)
        v_out = torch.zeros((L, total, Hkv, P, d), dtype=dt, device=device)
        off = 0
        for b in range(B):
            n = n_pages_b[b]
            ids = perm[off:off + n]
            off += n
            page_table[b, :n] = ids
            pad = n * P
            kb = torch.zeros((L, Hkv, pad, d), dtype=dt, device=device)
            vb = torch.zeros((L, Hkv, pad, d), dtype=dt, device=device)
            T = int(lens[b])
            kb[:, :, :T] = k_dense[:, b, :, :T]
            vb[:, :, :T] = v_dense[:, b, :, :T]
            idx = ids.long().to(device)
            k_out[:, idx] = kb.reshape(L, Hkv, n, P, d).permute(0, 2, 1, 3, 4)
            v_out[:, idx] = vb.reshape(L, Hkv, n, P, d).permute(0, 2, 1, 3, 4)
        del k_dense, v_dense

    return Inputs(work, lens, k_out, v_out, page_table, q_win, q_dec, k_new, v_new, needle_pos)
