"""mpc_decode_step (one call per decode step) against the two calls it fuses.

With ``fuse`` = 1 the step runs the leaders' selection and every layer's
attention in one persistent kernel (the automatic setting launches the two
kernels of mpc_select and mpc_sparse_decode_attn, also checked here).  It is specified to give the selections of mpc_select
followed by mpc_sparse_decode_attn: the same fp32 similarity arithmetic and
ranking (so the selected ids are identical, no tie band), the same appended
rows and seals (so caches and pyramids are bit-identical), and the same
attention products summed in another order (outputs agree to fp32 rounding:
a relative error of 2e-5 per output vector is asserted, against 2e-3 for the
bf16 tolerance the oracle tests use).  Two engines are fed the same inputs;
one decodes with ``Engine.decode_step`` (the fused call), the other with
``Engine.decode_step_two_calls``.  Every shape crosses at least one tail seal.
The fused call's parity with the oracle itself is covered by the pipeline and
full-size tests of test_gpu_parity.py, whose engines decode through it.
"""
import ctypes as C

import numpy as np
import pytest
import torch

from paper_2501_06807_gb300 import mpcache, synth
from tests import helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2501_06807_gb300 import build
    build.build()


def _twin(w, E, device="cpu", **step_kw):
    """Runs the same workload through the fused and the two-call decode and
    compares every step."""
    R = H.window_rows_for(w)
    x = H.to_cuda(synth.generate(w, R, device=device, decode_steps=E))
    pt = x.page_table.cuda() if x.page_table is not None else None
    lens = x.prompt_lens.cuda()
    fused, ref = H.make_engine(w, E), H.make_engine(w, E)
    for eng in (fused, ref):
        eng.prefill(x.k, x.v, x.q_win, lens, pt, w.page_size)
    torch.cuda.synchronize()
    assert torch.equal(fused.rep, ref.rep) and torch.equal(fused.kc, ref.kc)
    worst = 0.0
    metric = step_kw.pop("metric", mpcache.MPC_SIM_EQ3)
    step_kw.setdefault("fuse", 1)
    for e in range(E):
        fused.decode_step(x.q[e], x.k_new[e], x.v_new[e], metric=metric, **step_kw)
        ref.select(x.q[e], metric=metric)
        ref.attend(x.q[e], x.k_new[e], x.v_new[e], advance=True)
        torch.cuda.synchronize()
        assert torch.equal(fused.sel, ref.sel), e
        assert torch.equal(fused.n_sel, ref.n_sel), e
        a, b = fused.out.double(), ref.out.double()
        err = ((a - b).abs().amax(-1) / b.abs().amax(-1).clamp_min(1e-30)).max().item()
        worst = max(worst, err)
        assert err <= 2e-5, (e, err)
    assert torch.equal(fused.n_tok, ref.n_tok)
    assert torch.equal(fused.kc, ref.kc) and torch.equal(fused.vc, ref.vc)
    for name in ("rmax", "rmin", "rep", "mean"):
        assert torch.equal(getattr(fused, name), getattr(ref, name)), name
    assert mpcache.device_status() == 0
    print(f"fused vs two calls: {E} steps, ids identical, max relative output difference {worst:.2e}")
    return fused


CASES = [
    # name, workload, steps, step kwargs
    ("gqa4_three_levels", synth.C5.replace(n_layers=6, prompt_len=4096, prompt_len_min=4096, n_q_heads=8,
                                            n_kv_heads=2, level_keep_ppm=(100_000, 250_000, 500_000)), 20, {}),
    ("mha_paged_ragged", synth.C4.replace(n_layers=3, batch=3, prompt_len=900, prompt_len_min=300, n_q_heads=4,
                                          n_kv_heads=4), 18, {}),
    ("gqa16", synth.C3.replace(n_layers=3, prompt_len=2048, prompt_len_min=2048, n_q_heads=16, n_kv_heads=1),
     17, {}),
    ("d64", synth.C3.replace(n_layers=3, prompt_len=1024, prompt_len_min=1024, n_q_heads=8, n_kv_heads=4,
                             head_dim=64), 17, {}),
    ("s8_gather_rows", synth.C3.replace(n_layers=2, prompt_len=1024, prompt_len_min=1024, n_q_heads=4,
                                        n_kv_heads=2, cluster_size=8, fanouts=(4,)), 18, {}),
    ("s32_two_tail_tiles", synth.C3.replace(n_layers=2, prompt_len=2048, prompt_len_min=2048, n_q_heads=4,
                                            n_kv_heads=2, cluster_size=32, fanouts=(4,)), 34, {}),
    ("token_wise_s1", synth.C3.replace(n_layers=2, prompt_len=1024, prompt_len_min=1024, n_q_heads=8,
                                       n_kv_heads=2, keep_ppm=1_000_000, cluster_size=1, fanouts=(16,),
                                       level_keep_ppm=(50_000, 250_000), share_every=1), 6, {}),
    ("no_speculative_round", synth.C3.replace(n_layers=5, prompt_len=2048, prompt_len_min=2048,
                                              n_q_heads=8, n_kv_heads=2), 17, dict(speculate=0)),
    ("speculative_round", synth.C3.replace(n_layers=5, prompt_len=2048, prompt_len_min=2048,
                                           n_q_heads=8, n_kv_heads=2), 17, dict(speculate=1)),
    ("all_static_ranges", synth.C3.replace(n_layers=5, prompt_len=2048, prompt_len_min=2048,
                                           n_q_heads=8, n_kv_heads=2), 17, dict(static_ppm=1_000_000)),
    ("half_dynamic_one_tile_slices", synth.C3.replace(n_layers=5, prompt_len=2048, prompt_len_min=2048,
                                                      n_q_heads=8, n_kv_heads=2), 17,
     dict(static_ppm=500_000, slice_tiles=1)),
    ("all_dynamic_slices", synth.C5.replace(n_layers=6, prompt_len=4096, prompt_len_min=4096, n_q_heads=8,
                                            n_kv_heads=2, level_keep_ppm=(100_000, 250_000, 500_000)), 20,
     dict(static_ppm=1, slice_tiles=3)),
    ("bound_metric", synth.C3.replace(n_layers=3, prompt_len=2048, prompt_len_min=2048, n_q_heads=8,
                                      n_kv_heads=2), 17, dict(metric=mpcache.MPC_SIM_BOUND)),
    ("mean_metric", synth.C3.replace(n_layers=3, prompt_len=2048, prompt_len_min=2048, n_q_heads=8,
                                     n_kv_heads=2), 17, dict(metric=mpcache.MPC_SIM_MEAN)),
    ("prompt_shorter_than_a_cluster", synth.C3.replace(n_layers=2, prompt_len=12, prompt_len_min=12,
                                                       n_q_heads=4, n_kv_heads=2, keep_ppm=1_000_000,
                                                       fanouts=(2,), share_every=1), 24, {}),
    ("automatic_two_launches", synth.C5.replace(n_layers=6, prompt_len=4096, prompt_len_min=4096, n_q_heads=8,
                                                n_kv_heads=2, level_keep_ppm=(100_000, 250_000, 500_000)), 20,
     dict(fuse=-1)),
    ("fp32_two_launch_path", synth.C1.replace(n_layers=2, prompt_len=300, prompt_len_min=300), 18, {}),
    ("fixed_point_two_launch_path", synth.C3.replace(n_layers=3, prompt_len=1024, prompt_len_min=1024,
                                                     n_q_heads=8, n_kv_heads=2), 17,
     dict(metric=mpcache.MPC_SIM_FXP)),
]


@pytest.mark.parametrize("name,w,E,kw", CASES, ids=[c[0] for c in CASES])
def test_fused_step_equals_two_calls(name, w, E, kw):
    _twin(w, E, **dict(kw))


def test_fused_step_equals_two_calls_at_32k():
    """The 32k-token needle workload at full size, 20 decode steps (one tail
    seal per unit): the fused kernel the benchmark times beside the default
    form gives the two calls' ids, caches and pyramids exactly."""
    _twin(synth.C5, 20, device="cuda")


@pytest.mark.parametrize("fuse", [1, -1])
def test_decode_step_replays_in_a_graph(fuse):
    """The decode step replays inside a CUDA graph (fused: one kernel per
    step, the published selections and counters of the workspace carried
    from replay to replay; automatic: the selection and attention launches)
    and gives the eager run's outputs bit for bit (static splits and fixed
    merge orders make them deterministic)."""
    w = synth.C3.replace(n_layers=6, prompt_len=2048, prompt_len_min=2048, n_q_heads=8, n_kv_heads=2)
    E = 20
    x = H.to_cuda(synth.generate(w, H.window_rows_for(w), device="cpu", decode_steps=E))
    lens = x.prompt_lens.cuda()
    eager, graphed = H.make_engine(w, E), H.make_engine(w, E)
    outs_e = torch.empty((E,) + eager.out.shape, device="cuda")
    outs_g = torch.empty_like(outs_e)
    for eng in (eager, graphed):
        eng.prefill(x.k, x.v, x.q_win, lens)
    for e in range(E):
        eager.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=outs_e[e], fuse=fuse)
    graphed.decode_step(x.q[0], x.k_new[0], x.v_new[0], out=outs_g[0], fuse=fuse)  # allocates the workspace
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for e in range(1, E):
            graphed.decode_step(x.q[e], x.k_new[e], x.v_new[e], out=outs_g[e], fuse=fuse)
    g.replay()
    torch.cuda.synchronize()
    diff = (outs_g - outs_e).abs().amax(dim=(2, 3, 4))  # [step][layer]
    bad = [(e, l, float(diff[e, l])) for e, l in zip(*torch.nonzero(diff).T.tolist())]
    assert not bad, bad[:12]
    assert torch.equal(graphed.kc, eager.kc) and torch.equal(graphed.rep, eager.rep)
    assert mpcache.device_status() == 0


def test_fused_step_refuses_a_group_without_its_leader():
    w = synth.C3.replace(n_layers=6, prompt_len=512, prompt_len_min=512, n_q_heads=4, n_kv_heads=2)
    eng = H.make_engine(w, 2)
    q = torch.zeros((6, 1, 4, 128), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((6, 1, 2, 128), dtype=torch.bfloat16, device="cuda")
    a = eng.step_args(q, kv, kv)
    refs = (mpcache.LayerRef * 2)(mpcache.LayerRef(3, 2, 0), mpcache.LayerRef(4, 2, 0))
    a.attn.n_refs, a.attn.refs = 2, C.cast(refs, C.POINTER(mpcache.LayerRef))
    n = C.c_size_t(0)
    lib = mpcache.load()
    assert lib.mpc_decode_step_workspace_size(C.byref(a), C.byref(n)) == mpcache.MPC_ERR_INVALID_ARG
    assert b"leader" in lib.mpc_last_error()
