"""The seeded input recipe of the synthetic workloads, checked on small shapes:
the sink key of the iid rule, the outlier channels, the contiguous needle
passage and its direction, window queries aligned to the end of each prompt,
the paged pool (a shuffled page table over the same keys as the dense
layout), and that equal seeds give equal inputs.  CPU only."""
import torch

from paper_2501_06807_gb300 import synth


def _small(w, **kw):
    return w.replace(n_layers=2, decode_steps=3, **kw)


def test_same_seed_same_inputs():
    w = _small(synth.C3, prompt_len=256, prompt_len_min=256, batch=1)
    a, b = synth.generate(w, 64), synth.generate(w, 64)
    for name in ("k", "v", "q_win", "q", "k_new", "v_new"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
    c = synth.generate(w.replace(seed=w.seed + 1), 64)
    assert not torch.equal(a.k, c.k)


def test_iid_rule_sink_key():
    w = _small(synth.C1, prompt_len=512, prompt_len_min=512)
    x = synth.generate(w, 103)
    norms = x.k.float().norm(dim=-1)             # [L][B][Hkv][T]
    # key 0 is drawn x4: its norm is about 4 sqrt(d), the others about sqrt(d)
    assert (norms[..., 0] > 2.5 * norms[..., 1:].median()).all()


def test_outlier_rule_four_channels_per_head():
    w = _small(synth.C2, prompt_len=2048, prompt_len_min=2048, batch=1, n_q_heads=4, n_kv_heads=4)
    x = synth.generate(w, 16)
    std = x.k.float().std(dim=3)                  # [L][B][Hkv][d] over positions
    for l in range(w.n_layers):
        for h in range(w.n_kv_heads):
            big = (std[l, 0, h] > 4.0).nonzero().flatten()
            assert len(big) == 4, (l, h, big)     # four channels scaled x8
            assert std[l, 0, h, big].min() > 6.0 and std[l, 0, h].median() < 1.2


def test_needle_passage_is_contiguous_and_directional():
    w = _small(synth.C5, prompt_len=4096, prompt_len_min=4096, n_q_heads=8, n_kv_heads=2)
    x = synth.generate(w, 410)
    T, L = w.prompt_len, w.needle_len
    d = w.head_dim
    for l in range(w.n_layers):
        for h in range(w.n_kv_heads):
            s0 = int(x.needle_pos[l, 0, h])
            assert T // 10 <= s0 and s0 + L <= (9 * T) // 10
            kk = x.k[l, 0, h].float()
            seg = kk[s0:s0 + L]
            u = seg.mean(dim=0)
            # 3u with |u| = sqrt(d), plus 0.5 n: the passage mean has norm ~3 sqrt(d)
            assert abs(float(u.norm()) / d ** 0.5 - 3.0) < 0.3
            cos = (kk @ u) / (kk.norm(dim=1) * u.norm())
            inside = cos[s0:s0 + L]
            outside = torch.cat([cos[:s0], cos[s0 + L:]])
            assert float(inside.min()) > 0.9 and float(outside.abs().max()) < 0.5
    # the queries of a needle layer point at the passage direction
    qd = x.q[:, 0, 0].float()                     # [E][Hq][d]
    u0 = x.k[0, 0, 0, int(x.needle_pos[0, 0, 0]):int(x.needle_pos[0, 0, 0]) + L].float().mean(dim=0)
    cos_q = (qd[:, :w.group] @ u0) / (qd[:, :w.group].norm(dim=-1) * u0.norm())
    assert float(cos_q.mean()) > 0.4


def test_window_queries_aligned_to_the_prompt_end():
    w = _small(synth.C4.replace(name="t"), batch=4, prompt_len=512, prompt_len_min=64,
               n_q_heads=2, n_kv_heads=2)
    R = 200
    x = synth.generate(w, R)
    for b in range(w.batch):
        T = int(x.prompt_lens[b])
        rows = min(R, T)
        nz = x.q_win[0, b].float().abs().sum(dim=(0, 2)) > 0   # [R]
        assert not nz[:R - rows].any() and nz[R - rows:].all(), (b, T)


def test_paged_pool_holds_the_dense_keys():
    w = _small(synth.C4, batch=3, prompt_len=300, prompt_len_min=40, n_q_heads=2, n_kv_heads=2)
    xp = synth.generate(w, 60)
    xd = synth.generate(w.replace(paged=False), 60)
    P = w.page_size
    n_pages = [(int(t) + P - 1) // P for t in xp.prompt_lens]
    ids = torch.cat([xp.page_table[b, :n] for b, n in enumerate(n_pages)])
    assert sorted(ids.tolist()) == list(range(sum(n_pages)))   # a permutation of the pool
    assert (xp.page_table[xp.page_table >= 0].numel() == sum(n_pages))
    for l in range(w.n_layers):
        for b in range(w.batch):
            T = int(xp.prompt_lens[b])
            kk, vv = xp.dense_kv(l, b)
            assert torch.equal(kk[:, :T], xd.k[l, b, :, :T])
            assert torch.equal(vv[:, :T], xd.v[l, b, :, :T])
