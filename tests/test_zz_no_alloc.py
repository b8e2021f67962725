"""The allocation-free decode entry point.

mpc_sparse_decode_attn_static_scratch serves callers that cannot allocate
device memory: it keeps its split-K scratch in a fixed array inside the
library instead of a caller workspace.  These tests call it through the C ABI
and check it against the regular entry point and against the oracle's
sparse attention over the same cache rows and selection (same tolerance as
the other attention tests), twice in a row so that state left in the shared
array by the first call cannot leak into the second.  The file sorts last so
that a run stopping at the first failure has already run every other test.
"""
import ctypes as C
import math

import numpy as np
import pytest
import torch

from oracle import mpcache_oracle as O
from paper_2501_06807_gb300 import synth
from tests import helpers as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    from paper_2501_06807_gb300 import build, mpcache
    build.build()
    return mpcache.load()


def _static_call(lib, eng, q, kn, vn, advance):
    a = eng.attn_args(q, kn, vn, advance=advance)
    rc = lib.mpc_sparse_decode_attn_static_scratch(C.byref(a), C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0, lib.mpc_last_error()


def _oracle_worst(eng, x, e, w, got):
    """The largest relative error of ``got`` ([layer][b][Hq][d]) against the
    oracle's sparse attention (Alg. 1) over the engine's cache rows (the
    appended row included) and its selection, for sequence 0."""
    G, d, s = w.group, w.head_dim, w.cluster_size
    n = int(eng.n_tok[0])  # rows before this step's append
    n_sel = int(eng.n_sel[0])
    sel = eng.sel.cpu().numpy()
    worst = 0.0
    for l in range(w.n_layers):
        for h in range(w.n_kv_heads):
            K = H.unswizzle(eng.kc[l, 0, h, :n + 1].cpu()).double().numpy()
            V = H.unswizzle(eng.vc[l, 0, h, :n + 1].cpu()).double().numpy()
            toks = O.attended_tokens(n, s, sel[eng.group_of[l], 0, h, :n_sel])
            for g in range(G):
                q = x.q[e, l, 0, h * G + g].double().cpu().numpy()
                ref = O.sparse_attention(q, K[toks], V[toks], 1 / math.sqrt(d))
                worst = max(worst, H.rel_err(got[l, 0, h * G + g].double().cpu().numpy(), ref))
    return worst


@pytest.mark.parametrize("Hq,Hkv,n_layers", [(8, 2, 3), (4, 4, 1)])
def test_static_scratch_matches_workspace_path(lib, Hq, Hkv, n_layers):
    from paper_2501_06807_gb300 import mpcache
    w = synth.C5.replace(n_layers=n_layers, prompt_len=2048, prompt_len_min=2048, n_q_heads=Hq,
                         n_kv_heads=Hkv, level_keep_ppm=(250_000, 500_000, 1_000_000))
    E = 3
    x = H.to_cuda(synth.generate(w, H.window_rows_for(w), decode_steps=E))
    eng = H.make_engine(w, E)
    eng.prefill(x.k, x.v, x.q_win, x.prompt_lens.cuda())
    tol = 2e-3
    for e in range(E):
        eng.select(x.q[e])
        eng.attend(x.q[e], x.k_new[e], x.v_new[e], advance=False)
        ref = eng.out.clone()
        for _ in range(2):  # two calls in a row on the same state
            eng.out.zero_()
            _static_call(lib, eng, x.q[e], x.k_new[e], x.v_new[e], advance=False)
            got = eng.out.clone()
            err = (got - ref).abs().amax(dim=-1) / ref.abs().amax(dim=-1)
            assert float(err.max()) <= tol
            assert _oracle_worst(eng, x, e, w, got) <= tol
        _static_call(lib, eng, x.q[e], x.k_new[e], x.v_new[e], advance=True)
    torch.cuda.synchronize()
    assert eng.n_tok.tolist() == [int(eng.n_keep[0]) + E]
    assert mpcache.device_status() == 0


def test_static_scratch_rejects_oversize(lib):
    from paper_2501_06807_gb300 import mpcache
    # 16 query heads per kv head and few units: many splits, ~6 MB of partials
    w = synth.C2.replace(n_layers=8, batch=2, n_q_heads=32, n_kv_heads=2,
                         level_keep_ppm=(1_000_000, 1_000_000))
    eng = H.make_engine(w, 4)
    q = torch.zeros((8, 2, 32, 128), dtype=torch.bfloat16, device="cuda")
    kv = torch.zeros((8, 2, 2, 128), dtype=torch.bfloat16, device="cuda")
    a = eng.attn_args(q, kv, kv)
    n = C.c_size_t(0)
    assert lib.mpc_sparse_decode_attn_workspace_size(C.byref(a), C.byref(n)) == 0
    assert n.value > 4 << 20
    rc = lib.mpc_sparse_decode_attn_static_scratch(C.byref(a), None)
    assert rc == mpcache.MPC_ERR_WORKSPACE
    assert b"4 MiB" in lib.mpc_last_error()
