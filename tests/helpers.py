"""Shared helpers of the test-suite (no method arithmetic of their own)."""
from __future__ import annotations

import json
import os

import numpy as np
import torch

from oracle import mpcache_oracle as O
from paper_2501_06807_gb300 import synth


def oracle_params(w: synth.Workload) -> O.Params:
    return O.Params(keep_ppm=w.keep_ppm, cluster_size=w.cluster_size, fanouts=w.fanouts,
                    level_keep_ppm=w.level_keep_ppm, share_every=w.share_every, alpha=w.alpha,
                    window_ppm=w.window_ppm, long_window_ppm=w.long_window_ppm,
                    long_prompt_threshold=w.long_prompt_threshold)


def window_rows_for(w: synth.Workload) -> int:
    """Rows of window queries to draw: the longest window of any prompt
    length up to T_max (computed with the oracle's rule)."""
    return max(O.window_length(t, w.window_ppm, w.long_window_ppm, w.long_prompt_threshold)
               for t in {w.prompt_len, min(w.prompt_len, w.long_prompt_threshold)})


def oracle_run(x: synth.Inputs, steps: int, layers):
    """Runs the oracle on the generator's tensors (widened to float64)."""
    w = x.work
    f = lambda t: t.detach().to("cpu").double().numpy()
    dense = {}

    def kv(l, b):
        if (l, b) not in dense:
            k, v = x.dense_kv(l, b)
            dense[(l, b)] = (f(k), f(v))
        return dense[(l, b)]

    return O.run(lambda l, b: kv(l, b)[0], lambda l, b: kv(l, b)[1],
                 lambda l, b: f(x.q_win[l, b]), lambda e, l, b: f(x.q[e, l, b]),
                 lambda e, l, b: f(x.k_new[e, l, b]), lambda e, l, b: f(x.v_new[e, l, b]),
                 [int(t) for t in x.prompt_lens], oracle_params(w), steps=steps, layers=layers,
                 keep_levels=True)


def make_engine(w: synth.Workload, steps: int, layers=None):
    from paper_2501_06807_gb300 import mpcache
    return mpcache.Engine(n_layers=w.n_layers, batch=w.batch, n_q_heads=w.n_q_heads,
                          n_kv_heads=w.n_kv_heads, head_dim=w.head_dim,
                          dtype=torch.float32 if w.dtype == "f32" else torch.bfloat16,
                          t_max=w.prompt_len, keep_ppm=w.keep_ppm, cluster_size=w.cluster_size,
                          fanouts=w.fanouts, level_keep_ppm=w.level_keep_ppm,
                          share_every=w.share_every, max_decode_steps=steps, alpha=w.alpha,
                          window_ppm=w.window_ppm, long_window_ppm=w.long_window_ppm,
                          long_prompt_threshold=w.long_prompt_threshold, layers=layers)


def to_cuda(x: synth.Inputs) -> synth.Inputs:
    import dataclasses
    kw = {}
    for fld in dataclasses.fields(x):
        v = getattr(x, fld.name)
        if isinstance(v, torch.Tensor) and fld.name not in ("prompt_lens", "needle_pos"):
            v = v.cuda()
        kw[fld.name] = v
    return synth.Inputs(**kw)


def set_parity(gpu, ref_sorted_ids, ref_scores_of, k, band):
    """Compares a GPU index set with the oracle's top-k set.

    ``ref_scores_of(ids)`` gives the oracle's float64 scores of ids.  Sets may
    differ only by ids whose oracle scores lie within ``band`` (absolute) of
    the oracle's k-th score: those are ties at the kernel's precision.
    Returns the number of such tie swaps."""
    g = set(int(i) for i in gpu)
    r = set(int(i) for i in ref_sorted_ids)
    assert len(g) == len(gpu) == k, (len(g), len(gpu), k)
    if g == r:
        return 0
    ref_ids = np.array(sorted(r))
    cut = float(np.min(ref_scores_of(ref_ids))) if len(ref_ids) else 0.0
    diff = np.array(sorted(g ^ r))
    sc = ref_scores_of(diff)
    bad = diff[np.abs(sc - cut) > band]
    assert len(bad) == 0, f"ids {bad[:8]} differ beyond the tie band {band:g} (cut {cut:g})"
    return len(g - r)


def rel_err(a, b):
    """max |a - b| / max |b| (a vector's error relative to its largest entry)."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.abs(a - b).max() / max(np.abs(b).max(), 1e-300))


def unswizzle(cache_rows: torch.Tensor) -> torch.Tensor:
    """Undoes the 16-byte chunk permutation of the cluster-major cache:
    [..., rows, d] in storage order -> logical order."""
    rows, d = cache_rows.shape[-2], cache_rows.shape[-1]
    E = 16 // cache_rows.element_size()
    n_ch = d // E
    r = torch.arange(rows).view(rows, 1)
    ch = torch.arange(n_ch).view(1, n_ch)
    src = (ch ^ (r & 7))  # logical chunk ch is stored at ch ^ (r & 7)
    x = cache_rows.reshape(*cache_rows.shape[:-1], n_ch, E)
    idx = src.to(cache_rows.device).view(*([1] * (x.dim() - 3)), rows, n_ch, 1).expand_as(x)
    return torch.gather(x, -2, idx).reshape(cache_rows.shape)


def log_parity(test: str, **fields):
    """Reports one parity record (measured errors, the bands they are held to,
    counts of tie swaps and skipped units): printed (shown with ``pytest -rP``
    or ``-s``) and, when the environment variable MPC_PARITY_LOG names a file,
    appended to it as a JSON line."""
    rec = {"test": test}
    for k, v in fields.items():
        if isinstance(v, (np.floating, np.integer)):
            v = v.item()
        rec[k] = v
    line = json.dumps(rec)
    print("parity", line)
    path = os.environ.get("MPC_PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(line + "\n")
