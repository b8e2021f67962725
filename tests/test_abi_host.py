"""Host-side checks of the C ABI (no GPU needed): the library loads and
exports every entry point of include/mpcache.h, the ctypes mirrors of the
argument structs match the C layout, and argument validation rejects bad
input with the documented codes before any CUDA call."""
import ctypes as C
import os
import re
import subprocess

import pytest
import torch

from oracle import mpcache_oracle as O
from paper_2501_06807_gb300 import build, mpcache

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "mpcache.h")


@pytest.fixture(scope="module")
def lib():
    build.build()
    return mpcache.load()


def test_exports_every_declared_symbol(lib):
    text = open(HEADER).read()
    names = re.findall(r"MPC_API\s+[\w\s\*]+?\b(mpc_\w+)\s*\(", text)
    assert len(names) >= 12
    assert set(names) == set(mpcache.ENTRY_POINTS)
    for n in names:
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", mpcache.library_path()],
                         capture_output=True, text=True).stdout
    exported = set(re.findall(r"\b(mpc_\w+)\b", out))
    assert set(names) <= exported
    assert lib.mpc_abi_version() == mpcache.ABI_VERSION == 7


def test_struct_layout_matches_c(tmp_path):
    structs = {"mpc_layer_ref": mpcache.LayerRef, "mpc_kv_tensor": mpcache.KvTensor,
               "mpc_static_args": mpcache.StaticArgs, "mpc_cluster_args": mpcache.ClusterArgs,
               "mpc_select_args": mpcache.SelectArgs, "mpc_attn_args": mpcache.AttnArgs,
               "mpc_commonality_args": mpcache.CommonalityArgs, "mpc_decode_args": mpcache.DecodeArgs}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "mpcache.h"', 'int main(void){']
    for cname, py in structs.items():
        lines.append(f'printf("{cname} size %zu\\n", sizeof({cname}));')
        for fname, _ in py._fields_:
            lines.append(f'printf("{cname} {fname} %zu\\n", offsetof({cname}, {fname}));')
    lines.append("return 0;}")
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)], check=True)
    got = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    for line in got:
        if not line:
            continue
        cname, field, val = line.split()
        py = structs[cname]
        want = C.sizeof(py) if field == "size" else getattr(py, field).offset
        assert int(val) == want, (cname, field, val, want)


def _attn_args(**over):
    a = mpcache.AttnArgs()
    a.struct_size = C.sizeof(mpcache.AttnArgs)
    refs = (mpcache.LayerRef * 2)(mpcache.LayerRef(0, 0, 1), mpcache.LayerRef(1, 0, 0))
    a.n_refs, a.refs = 2, C.cast(refs, C.POINTER(mpcache.LayerRef))
    a.batch, a.n_q_heads, a.n_kv_heads, a.head_dim, a.dtype = 1, 8, 2, 128, mpcache.MPC_BF16
    a.kc = a.vc = a.q = a.k_new = a.v_new = 4096
    a.cap_tokens, a.sel_cap, a.summary_rows = 512, 4, 64
    a.cluster_size, a.n_levels = 16, 2
    a.fanout[0] = 4
    a.alpha = 0.6
    for k, v in over.items():
        setattr(a, k, v)
    a._refs = refs
    return a


def _ws(lib, fn, a):
    n = C.c_size_t(0)
    rc = getattr(lib, fn)(C.byref(a), C.byref(n))
    return rc, n.value


def test_attn_validation(lib):
    rc, n = _ws(lib, "mpc_sparse_decode_attn_workspace_size", _attn_args())
    assert rc == 0 and n > 0
    cases = [
        (dict(struct_size=8), mpcache.MPC_ERR_INVALID_ARG),
        (dict(head_dim=96), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(dtype=7), mpcache.MPC_ERR_INVALID_ARG),
        (dict(n_q_heads=7), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(n_refs=0), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(cap_tokens=500), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(cluster_size=0), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(n_levels=5), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(alpha=1.5), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(kc=4100), mpcache.MPC_ERR_INVALID_ARG),
        (dict(n_q_heads=2 * 17, n_kv_heads=2), mpcache.MPC_ERR_BAD_SHAPE),
    ]
    for over, code in cases:
        rc, _ = _ws(lib, "mpc_sparse_decode_attn_workspace_size", _attn_args(**over))
        assert rc == code, (over, rc, lib.mpc_last_error())
        assert lib.mpc_last_error()
    a = _attn_args()
    a.fanout[0] = 1
    assert _ws(lib, "mpc_sparse_decode_attn_workspace_size", a)[0] == mpcache.MPC_ERR_BAD_SHAPE
    # the call itself rejects a missing workspace before launching anything
    a = _attn_args()
    a.n_tok = a.out = a.sel = a.n_sel = 8192
    assert lib.mpc_sparse_decode_attn(C.byref(a), None, 0, None) == mpcache.MPC_ERR_WORKSPACE
    assert lib.mpc_sparse_decode_attn(None, None, 0, None) == mpcache.MPC_ERR_INVALID_ARG


def test_select_and_static_validation(lib):
    s = mpcache.SelectArgs()
    s.struct_size = C.sizeof(mpcache.SelectArgs)
    refs = (mpcache.LayerRef * 1)(mpcache.LayerRef(0, 0, 0))
    s.n_refs, s.refs = 1, C.cast(refs, C.POINTER(mpcache.LayerRef))
    s.batch, s.n_q_heads, s.n_kv_heads, s.head_dim, s.dtype = 1, 4, 4, 64, mpcache.MPC_F32
    s.rep, s.cap_tokens, s.cluster_size, s.n_levels = 4096, 256, 16, 1
    s.summary_rows, s.sel_cap = 16, 4
    s.level_keep_ppm[0] = 250_000
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_INVALID_ARG  # not a leader
    refs[0].leader = 1
    assert _ws(lib, "mpc_select_workspace_size", s) == (0, 0)
    s.metric = 7                       # not a metric
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_INVALID_ARG
    s.metric, s.r_max, s.r_min = mpcache.MPC_SIM_BOUND, 4100, 8192  # r_max misaligned
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_INVALID_ARG
    s.r_max = 4096
    assert _ws(lib, "mpc_select_workspace_size", s) == (0, 0)
    s.q, s.n_tok, s.out_sel, s.out_n_sel, s.r_min = 8192, 8192, 8192, 8192, None
    assert lib.mpc_select(C.byref(s), None, 0, None) == mpcache.MPC_ERR_INVALID_ARG  # bound needs r_min
    # the fixed-point metric reads r_max and r_min and checks alpha and f
    s.metric, s.r_min, s.alpha, s.frac_bits = mpcache.MPC_SIM_FXP, 8192, 0.6, 18
    assert _ws(lib, "mpc_select_workspace_size", s) == (0, 0)
    for alpha, fb in ((1.5, 18), (-0.1, 18), (float("nan"), 18), (0.6, 0), (0.6, 25)):
        s.alpha, s.frac_bits = alpha, fb
        assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_BAD_SHAPE, (alpha, fb)
    s.alpha, s.frac_bits, s.r_max = 0.6, 24, 4100
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_INVALID_ARG  # misaligned
    s.r_max, s.r_min = 4096, None
    assert lib.mpc_select(C.byref(s), None, 0, None) == mpcache.MPC_ERR_INVALID_ARG  # needs r_min
    s.metric, s.r_max, s.r_min, s.q, s.n_tok, s.out_sel, s.out_n_sel = mpcache.MPC_SIM_EQ3, None, None, None, None, None, None
    s.sel_cap = 3
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_BAD_SHAPE
    s.sel_cap = 4
    s.level_keep_ppm[0] = 0
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_BAD_SHAPE
    s.level_keep_ppm[0] = 250_000
    s.summary_rows = 15
    assert _ws(lib, "mpc_select_workspace_size", s)[0] == mpcache.MPC_ERR_BAD_SHAPE

    a = mpcache.StaticArgs()
    a.struct_size = C.sizeof(mpcache.StaticArgs)
    a.n_refs, a.refs = 1, C.cast(refs, C.POINTER(mpcache.LayerRef))
    a.batch, a.n_q_heads, a.n_kv_heads, a.head_dim, a.dtype = 2, 8, 2, 128, mpcache.MPC_BF16
    a.t_max, a.win_rows, a.keep_cap = 32768, 4916, 8192
    a.window_ppm, a.long_window_ppm, a.long_prompt_threshold, a.keep_ppm = 200_000, 100_000, 24576, 250_000
    rc, n = _ws(lib, "mpc_static_evict_workspace_size", a)
    # row statistics per (ref, b, query head), rows padded to a multiple of
    # 128 (4916 -> 4992): fp32 -(m + log2 l), plus a 16-byte bf16 row
    assert rc == 0 and n == 1 * 2 * 8 * 4992 * (4 + 16)
    a.win_rows = 4915      # the longest window (T = 24576) needs 4916 rows
    assert _ws(lib, "mpc_static_evict_workspace_size", a)[0] == mpcache.MPC_ERR_BAD_SHAPE
    a.win_rows, a.keep_cap = 4916, 8191
    assert _ws(lib, "mpc_static_evict_workspace_size", a)[0] == mpcache.MPC_ERR_BAD_SHAPE
    # paged bf16 keys: the statistics, then the dense copy of the refs' keys
    # (n_refs * batch * n_kv_heads * t_max * d bf16) the tensor-core passes read
    a.keep_cap = 8192
    pt = (C.c_int32 * 1)(0)
    a.k.page_table, a.k.page_size, a.k.max_pages = C.cast(pt, C.c_void_p), 16, 2048
    rc, n = _ws(lib, "mpc_static_evict_workspace_size", a)
    assert rc == 0 and n == 1 * 2 * 8 * 4992 * (4 + 16) + 1 * 2 * 2 * 32768 * 128 * 2
    a.dtype = mpcache.MPC_F32  # fp32 keys stay paged (SIMT passes): no copy
    rc, n = _ws(lib, "mpc_static_evict_workspace_size", a)
    assert rc == 0 and n == 1 * 2 * 8 * 4992 * (4 + 16)


def test_summary_rows(lib):
    assert mpcache.summary_rows(8192 + 512, 16, (8, 8)) == 544 + 68 + 9
    assert mpcache.summary_rows(256, 16, ()) == 16
    arr = (C.c_int32 * 4)(1, 0, 0, 0)
    assert lib.mpc_summary_rows(256, 16, 2, arr) == mpcache.MPC_ERR_BAD_SHAPE


def test_host_rules_match_oracle():
    from oracle import mpcache_oracle as O
    for t in (1, 7, 512, 1000, 2048, 24_576, 24_577, 32_768):
        for ppm in (1, 50_000, 125_000, 200_000, 333_333, 1_000_000):
            assert mpcache.ppm_count(t, ppm) == O.kept_count(t, ppm)
    for m in (1, 2, 4):
        for l in range(40):
            assert mpcache.sharing_leader(l, m) == O.leader_of(l, m)


def test_missing_library_fails_loudly(tmp_path):
    with pytest.raises(OSError):
        mpcache.load(str(tmp_path / "nope.so"))


def test_selftest_wait_validation(lib):
    # checked before any launch: kind, the limit's range, the flag pointer
    assert lib.mpc_selftest_wait(2, 1000, None, None) == mpcache.MPC_ERR_INVALID_ARG
    assert lib.mpc_selftest_wait(0, 0, None, None) == mpcache.MPC_ERR_BAD_SHAPE
    assert lib.mpc_selftest_wait(0, 1_000_001, None, None) == mpcache.MPC_ERR_BAD_SHAPE
    assert lib.mpc_selftest_wait(1, 1000, None, None) == mpcache.MPC_ERR_INVALID_ARG


def test_commonality_validation(lib):
    a = mpcache.CommonalityArgs()
    a.struct_size = C.sizeof(mpcache.CommonalityArgs)
    a.n_layers, a.batch, a.n_kv_heads, a.sel_cap, a.n_clusters, a.k, a.m = 4, 2, 3, 8, 100, 8, 1
    a.sel_layer_stride = 2 * 3 * 8
    a.sel = a.out_total = a.out_score = None
    assert lib.mpc_commonality(C.byref(a), None) == mpcache.MPC_ERR_INVALID_ARG  # NULL pointers
    for field, bad in (("m", 0), ("m", 4), ("k", 9), ("n_layers", 1), ("sel_layer_stride", 47)):
        b = mpcache.CommonalityArgs.from_buffer_copy(a)
        setattr(b, field, bad)
        assert lib.mpc_commonality(C.byref(b), None) == mpcache.MPC_ERR_BAD_SHAPE, field
    # the position map: checked before any launch (the fake pointers are never read)
    a.sel, a.out_total, a.out_score = 16, 32, 48
    a.kept, a.kept_layer_stride, a.kept_cap, a.cluster_size = 64, 2 * 3 * 40, 40, 16
    assert lib.mpc_commonality(C.byref(a), None) == mpcache.MPC_ERR_INVALID_ARG  # no n_keep / prompt_len
    a.n_keep, a.prompt_len = 80, 96
    for field, bad in (("cluster_size", 0), ("kept_cap", 0), ("kept_layer_stride", 2 * 3 * 40 - 1)):
        b = mpcache.CommonalityArgs.from_buffer_copy(a)
        setattr(b, field, bad)
        assert lib.mpc_commonality(C.byref(b), None) == mpcache.MPC_ERR_BAD_SHAPE, field
    a.struct_size = 3
    assert lib.mpc_commonality(C.byref(a), None) == mpcache.MPC_ERR_INVALID_ARG


def test_choose_share_every_binding():
    assert mpcache.choose_share_every({1: 0.95, 2: 0.9, 3: 0.6}, 0.85) == 3   # groups of 3 layers
    assert mpcache.choose_share_every({1: 0.5}, 0.85) == 1                     # no sharing


def test_engine_rejects_unsupported_dtype():
    """The kernels take float32 or bfloat16 only; any other dtype is refused
    before any buffer is allocated, not passed on under the float32 code."""
    with pytest.raises(TypeError):
        mpcache.Engine(n_layers=2, batch=1, n_q_heads=2, n_kv_heads=1, head_dim=64, dtype=torch.float16,
                       t_max=64, keep_ppm=500_000, cluster_size=16, fanouts=(), level_keep_ppm=(500_000,),
                       share_every=2, max_decode_steps=4)


def test_input_checks_refuse_what_the_calls_would_misread():
    chk = mpcache._check_input
    t = torch.zeros((3, 2, 4, 8), dtype=torch.bfloat16)
    # host memory only where allowed, and then pinned (checked last, so the
    # layout checks below run on CPU tensors)
    with pytest.raises(ValueError, match="on the GPU"):
        chk(t, "q", torch.bfloat16, (None, 2, 4, 8))
    with pytest.raises(TypeError, match="dtype"):
        chk(t, "q", torch.float32, (None, 2, 4, 8))
    with pytest.raises(ValueError, match="shape"):
        chk(t, "q", torch.bfloat16, (None, 2, 4, 16))
    with pytest.raises(ValueError, match="shape"):
        chk(t[0], "q", torch.bfloat16, (None, 2, 4, 8))
    with pytest.raises(ValueError, match="layers"):
        chk(t, "q", torch.bfloat16, (None, 2, 4, 8), min_layers=4)
    # a transposed view has the right sizes but not the layout
    u = torch.zeros((3, 2, 8, 4), dtype=torch.bfloat16).transpose(2, 3)
    with pytest.raises(ValueError, match="contiguous"):
        chk(u, "q", torch.bfloat16, (None, 2, 4, 8))
    # a layer stride of its own is fine (a slice along dim 0 of a larger buffer)
    big = torch.zeros((6, 2, 4, 8), dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="on the GPU"):   # layout accepted, only the memory refused
        chk(big[::2], "q", torch.bfloat16, (None, 2, 4, 8), min_layers=3)


def test_static_args_need_the_engines_window_rows():
    """Window queries with fewer rows than the longest window the engine's
    prompts can have are refused before the C call (which refuses them too)."""
    eng = mpcache.Engine.__new__(mpcache.Engine)   # no device buffers needed
    eng.win_rows = 52
    with pytest.raises(ValueError, match="window rows"):
        eng.static_args(torch.zeros(1), torch.zeros((1, 1, 2, 51, 64), dtype=torch.bfloat16), torch.zeros(1))


def _step_args(**over):
    a = mpcache.DecodeArgs()
    a.struct_size = C.sizeof(mpcache.DecodeArgs)
    att = _attn_args()
    a.attn = att
    a._refs = att._refs
    a.level_keep_ppm[0], a.level_keep_ppm[1] = 125_000, 500_000
    a.metric, a.speculate = mpcache.MPC_SIM_EQ3, -1
    for k, v in over.items():
        setattr(a, k, v)
    return a


def test_decode_step_validation(lib):
    """mpc_decode_step checks the attention arguments like
    mpc_sparse_decode_attn, the selection settings like mpc_select, and that
    every ref's group is led by a ref of the call, before any CUDA call."""
    rc, n = _ws(lib, "mpc_decode_step_workspace_size", _step_args())
    assert rc == 0 and n > 0, lib.mpc_last_error()
    cases = [
        (dict(struct_size=8), mpcache.MPC_ERR_INVALID_ARG),
        (dict(speculate=2), mpcache.MPC_ERR_BAD_SHAPE),
        (dict(metric=9), mpcache.MPC_ERR_INVALID_ARG),
    ]
    for over, code in cases:
        rc, _ = _ws(lib, "mpc_decode_step_workspace_size", _step_args(**over))
        assert rc == code, (over, rc, lib.mpc_last_error())
    a = _step_args()
    a.level_keep_ppm[1] = 0
    assert _ws(lib, "mpc_decode_step_workspace_size", a)[0] == mpcache.MPC_ERR_BAD_SHAPE
    a = _step_args()
    a.attn.head_dim = 96  # the embedded attention arguments are checked too
    assert _ws(lib, "mpc_decode_step_workspace_size", a)[0] == mpcache.MPC_ERR_BAD_SHAPE
    # a group whose leader is not among the refs, and a group with two leaders
    for pairs in (((1, 0, 0), (2, 0, 0)), ((0, 0, 1), (1, 0, 1))):
        a = _step_args()
        refs = (mpcache.LayerRef * 2)(*[mpcache.LayerRef(*p) for p in pairs])
        a.attn.refs = C.cast(refs, C.POINTER(mpcache.LayerRef))
        assert _ws(lib, "mpc_decode_step_workspace_size", a)[0] == mpcache.MPC_ERR_INVALID_ARG
        assert b"leader" in lib.mpc_last_error()
    # the form a call takes: two launches unless the fused kernel is asked for
    # or chosen (305-1216 selection units); the fixture has 2 units
    for fuse, want in ((0, 2), (-1, 2), (1, 1)):
        n = C.c_int32(0)
        assert lib.mpc_decode_step_plan(C.byref(_step_args(fuse=fuse)), C.byref(n)) == 0, lib.mpc_last_error()
        assert n.value == want, (fuse, n.value)
    assert lib.mpc_decode_step_plan(C.byref(_step_args(fuse=2)), C.byref(C.c_int32(0))) == mpcache.MPC_ERR_BAD_SHAPE
    # automatic: the fused kernel from 305 to 1216 selection units (leader
    # refs x batch x kv heads; the fixture has 1 leader ref and 2 kv heads)
    for batch, want in ((152, 2), (153, 1), (512, 1)):
        a = _step_args(fuse=-1)
        a.attn.batch = batch
        n = C.c_int32(0)
        assert lib.mpc_decode_step_plan(C.byref(a), C.byref(n)) == 0, lib.mpc_last_error()
        assert n.value == want, (batch, n.value)
    a = _step_args(fuse=-1)
    a.attn.refs[1].leader = 1
    a.attn.refs[1].group = 1      # two leader refs: 4 units per sequence
    a.attn.batch = 400            # 1600 units: two launches again
    n = C.c_int32(0)
    assert lib.mpc_decode_step_plan(C.byref(a), C.byref(n)) == 0, lib.mpc_last_error()
    assert n.value == 2
    # the call rejects a missing workspace before launching anything
    a = _step_args()
    a.attn.n_tok = a.attn.out = a.attn.sel = a.attn.n_sel = 8192
    a.attn.rep = a.attn.r_max = a.attn.r_min = 16384
    assert lib.mpc_decode_step(C.byref(a), None, 0, None) == mpcache.MPC_ERR_WORKSPACE
    assert lib.mpc_decode_step(None, None, 0, None) == mpcache.MPC_ERR_INVALID_ARG


def test_layer_refs_follow_the_sharing_rule(lib):
    """mpc_layer_refs (Sec. 3.4): the first two layers lead themselves, later
    layers reuse the first layer of their group of share_every; leaders are
    the oracle's (leader_of, pinned by hand values), groups are numbered in
    layer order."""
    for L in (1, 2, 3, 6, 32, 33, 128):
        for m in (1, 2, 3, 4, 7):
            arr = (mpcache.LayerRef * L)()
            g = lib.mpc_layer_refs(L, m, arr)
            leaders = sorted({O.leader_of(l, m) for l in range(L)})
            assert g == len(leaders)
            for l in range(L):
                lead = O.leader_of(l, m)
                assert arr[l].layer == l
                assert arr[l].group == leaders.index(lead)
                assert arr[l].leader == (1 if lead == l else 0)
    # the 32-layer workloads: groups of two (17 leaders) and of four (10 leaders)
    assert lib.mpc_layer_refs(32, 2, (mpcache.LayerRef * 32)()) == 17
    assert lib.mpc_layer_refs(32, 4, (mpcache.LayerRef * 32)()) == 10
    bad = (mpcache.LayerRef * 4)()
    assert lib.mpc_layer_refs(0, 2, bad) == mpcache.MPC_ERR_INVALID_ARG
    assert lib.mpc_layer_refs(4, 0, bad) == mpcache.MPC_ERR_INVALID_ARG
    assert lib.mpc_layer_refs(129, 2, (mpcache.LayerRef * 129)()) == mpcache.MPC_ERR_INVALID_ARG
    assert lib.mpc_layer_refs(4, 2, None) == mpcache.MPC_ERR_INVALID_ARG


def test_choose_share_every(lib):
    """mpc_choose_share_every: the largest window (m + 1 layers) whose
    commonality reaches the threshold, else no sharing."""
    def choose(scores, thr):
        arr = (C.c_float * len(scores))(*scores)
        return lib.mpc_choose_share_every(len(scores), arr, thr)
    assert choose([0.9, 0.7, 0.5], 0.6) == 3
    assert choose([0.9, 0.7, 0.5], 0.5) == 4
    assert choose([0.4, 0.3, 0.2], 0.5) == 1
    assert choose([0.4, 0.8, 0.2], 0.5) == 3   # a later window may reach it alone
    assert choose([1.0], 1.0) == 2
    assert mpcache.choose_share_every({1: 0.9, 2: 0.7, 3: 0.5}, 0.6) == 3
    assert choose([0.5], 1.5) == mpcache.MPC_ERR_INVALID_ARG
    assert lib.mpc_choose_share_every(0, (C.c_float * 1)(0.5), 0.5) == mpcache.MPC_ERR_INVALID_ARG
