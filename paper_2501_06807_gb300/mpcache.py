"""Python binding of libmpcache.so (include/mpcache.h).

Argument marshalling only: every step of the method runs in the library's
CUDA kernels.  Tensors are torch tensors on the current CUDA device; calls
are queued on torch's current stream.  The library must have been built
(``paper_2501_06807_gb300.build.build()``); importing this module without it
raises, there is no fallback.

``Engine`` owns the device buffers of one batch (cluster-major cache, summary
pyramid, selections, workspaces) and runs the method: ``prefill`` (static
eviction of the leader layers, then gathering and clustering of every layer)
and ``decode_step`` (selection for the leaders, then append + sparse attention
for every layer, all layers of a step in one launch each).
"""
from __future__ import annotations

import ctypes as C
import math
import os
from typing import List, Optional, Sequence

import torch

from . import build as _build

MPC_OK, MPC_ERR_INVALID_ARG, MPC_ERR_BAD_SHAPE, MPC_ERR_WORKSPACE, MPC_ERR_CUDA = 0, -1, -2, -3, -4
MPC_F32, MPC_BF16 = 0, 1
MPC_SIM_EQ3, MPC_SIM_BOUND, MPC_SIM_MEAN, MPC_SIM_FXP = 0, 1, 2, 3
FXP_FRAC_BITS = 18
MAX_LEVELS = 4
ABI_VERSION = 7
MAX_REFS = 128
PPM = 1_000_000


class LayerRef(C.Structure):
    """mpc_layer_ref: a processed layer's index, its sharing group and whether it leads."""
    _fields_ = [("layer", C.c_int32), ("group", C.c_int32), ("leader", C.c_int32)]


class KvTensor(C.Structure):
    """mpc_kv_tensor: prompt keys or values, dense or as a page pool with its page table."""
    _fields_ = [("data", C.c_void_p), ("layer_stride", C.c_int64), ("page_table", C.c_void_p),
                ("page_size", C.c_int32), ("max_pages", C.c_int32)]


class StaticArgs(C.Structure):
    """mpc_static_args: the arguments of mpc_static_evict, field for field."""
    _fields_ = [("struct_size", C.c_uint32), ("n_refs", C.c_int32), ("refs", C.POINTER(LayerRef)),
                ("batch", C.c_int32), ("n_q_heads", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("dtype", C.c_int32), ("t_max", C.c_int32),
                ("prompt_lens", C.c_void_p), ("q_win", C.c_void_p), ("q_win_layer_stride", C.c_int64),
                ("win_rows", C.c_int32), ("k", KvTensor), ("window_ppm", C.c_int32),
                ("long_window_ppm", C.c_int32), ("long_prompt_threshold", C.c_int32),
                ("keep_ppm", C.c_int32), ("scale", C.c_float), ("keep_cap", C.c_int32),
                ("out_scores", C.c_void_p), ("out_kept", C.c_void_p), ("out_n_keep", C.c_void_p)]


class ClusterArgs(C.Structure):
    """mpc_cluster_args: the arguments of mpc_build_clusters, field for field."""
    _fields_ = [("struct_size", C.c_uint32), ("n_refs", C.c_int32), ("refs", C.POINTER(LayerRef)),
                ("batch", C.c_int32), ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32),
                ("dtype", C.c_int32), ("t_max", C.c_int32), ("k", KvTensor), ("v", KvTensor),
                ("kept", C.c_void_p), ("keep_cap", C.c_int32), ("n_keep", C.c_void_p),
                ("kc", C.c_void_p), ("vc", C.c_void_p), ("cache_layer_stride", C.c_int64),
                ("cap_tokens", C.c_int32), ("r_max", C.c_void_p), ("r_min", C.c_void_p),
                ("rep", C.c_void_p), ("summary_rows", C.c_int32), ("cluster_size", C.c_int32),
                ("n_levels", C.c_int32), ("fanout", C.c_int32 * MAX_LEVELS), ("alpha", C.c_float),
                ("out_n_tok", C.c_void_p), ("mean", C.c_void_p)]


class SelectArgs(C.Structure):
    """mpc_select_args: the arguments of mpc_select, field for field."""
    _fields_ = [("struct_size", C.c_uint32), ("n_refs", C.c_int32), ("refs", C.POINTER(LayerRef)),
                ("batch", C.c_int32), ("n_q_heads", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("dtype", C.c_int32), ("q", C.c_void_p),
                ("q_layer_stride", C.c_int64), ("rep", C.c_void_p), ("summary_rows", C.c_int32),
                ("cap_tokens", C.c_int32), ("n_tok", C.c_void_p), ("cluster_size", C.c_int32),
                ("n_levels", C.c_int32), ("fanout", C.c_int32 * MAX_LEVELS),
                ("level_keep_ppm", C.c_int32 * MAX_LEVELS), ("sel_cap", C.c_int32),
                ("out_sel", C.c_void_p), ("out_n_sel", C.c_void_p), ("metric", C.c_int32),
                ("r_max", C.c_void_p), ("r_min", C.c_void_p), ("mean", C.c_void_p),
                ("alpha", C.c_float), ("frac_bits", C.c_int32)]


class CommonalityArgs(C.Structure):
    """mpc_commonality_args: the arguments of mpc_commonality, field for field."""
    _fields_ = [("struct_size", C.c_uint32), ("n_layers", C.c_int32), ("batch", C.c_int32),
                ("n_kv_heads", C.c_int32), ("sel", C.c_void_p), ("sel_layer_stride", C.c_int64),
                ("sel_cap", C.c_int32), ("n_clusters", C.c_int32), ("k", C.c_int32), ("m", C.c_int32),
                ("out_total", C.c_void_p), ("out_score", C.c_void_p), ("kept", C.c_void_p),
                ("kept_layer_stride", C.c_int64), ("kept_cap", C.c_int32), ("cluster_size", C.c_int32),
                ("n_keep", C.c_void_p), ("prompt_len", C.c_void_p)]


class AttnArgs(C.Structure):
    """mpc_attn_args: the arguments of mpc_sparse_decode_attn, field for field."""
    _fields_ = [("struct_size", C.c_uint32), ("n_refs", C.c_int32), ("refs", C.POINTER(LayerRef)),
                ("batch", C.c_int32), ("n_q_heads", C.c_int32), ("n_kv_heads", C.c_int32),
                ("head_dim", C.c_int32), ("dtype", C.c_int32), ("q", C.c_void_p),
                ("k_new", C.c_void_p), ("v_new", C.c_void_p), ("q_layer_stride", C.c_int64),
                ("kv_new_layer_stride", C.c_int64), ("kc", C.c_void_p), ("vc", C.c_void_p),
                ("cache_layer_stride", C.c_int64), ("cap_tokens", C.c_int32), ("sel", C.c_void_p),
                ("n_sel", C.c_void_p), ("sel_cap", C.c_int32), ("r_max", C.c_void_p),
                ("r_min", C.c_void_p), ("rep", C.c_void_p), ("summary_rows", C.c_int32),
                ("cluster_size", C.c_int32), ("n_levels", C.c_int32), ("fanout", C.c_int32 * MAX_LEVELS),
                ("alpha", C.c_float), ("n_tok", C.c_void_p), ("advance", C.c_int32),
                ("scale", C.c_float), ("out", C.c_void_p), ("out_layer_stride", C.c_int64),
                ("mean", C.c_void_p)]


class DecodeArgs(C.Structure):
    """mpc_decode_args: the arguments of mpc_decode_step (attention arguments plus selection settings)."""
    _fields_ = [("struct_size", C.c_uint32), ("attn", AttnArgs), ("level_keep_ppm", C.c_int32 * MAX_LEVELS),
                ("metric", C.c_int32), ("frac_bits", C.c_int32), ("speculate", C.c_int32),
                ("static_ppm", C.c_int32), ("slice_tiles", C.c_int32), ("fuse", C.c_int32)]


ENTRY_POINTS = ("mpc_static_evict_workspace_size", "mpc_build_clusters_workspace_size",
                "mpc_select_workspace_size", "mpc_sparse_decode_attn_workspace_size",
                "mpc_static_evict", "mpc_build_clusters", "mpc_select", "mpc_sparse_decode_attn",
                "mpc_summary_rows", "mpc_last_error", "mpc_device_status", "mpc_abi_version",
                "mpc_sparse_decode_attn_static_scratch", "mpc_commonality", "mpc_selftest_wait",
                "mpc_decode_step_workspace_size", "mpc_decode_step", "mpc_decode_step_plan", "mpc_layer_refs",
                "mpc_choose_share_every")

_LIB = None


def library_path() -> str:
    """Path of the in-tree libmpcache.so."""
    return _build.LIB


def load(path: Optional[str] = None) -> C.CDLL:
    """Load libmpcache.so (raises OSError if it has not been built)."""
    global _LIB
    if _LIB is not None and path is None:
        return _LIB
    p = path or library_path()
    if not os.path.exists(p):
        raise OSError(f"libmpcache.so not found at {p}; run paper_2501_06807_gb300.build.build()")
    lib = C.CDLL(p)
    for name in ("mpc_static_evict_workspace_size", "mpc_build_clusters_workspace_size",
                 "mpc_select_workspace_size", "mpc_sparse_decode_attn_workspace_size",
                 "mpc_decode_step_workspace_size"):
        getattr(lib, name).restype = C.c_int
        getattr(lib, name).argtypes = [C.c_void_p, C.POINTER(C.c_size_t)]
    for name in ("mpc_static_evict", "mpc_build_clusters", "mpc_select", "mpc_sparse_decode_attn",
                 "mpc_decode_step"):
        getattr(lib, name).restype = C.c_int
        getattr(lib, name).argtypes = [C.c_void_p, C.c_void_p, C.c_size_t, C.c_void_p]
    lib.mpc_summary_rows.restype = C.c_int64
    lib.mpc_summary_rows.argtypes = [C.c_int32, C.c_int32, C.c_int32, C.POINTER(C.c_int32)]
    lib.mpc_last_error.restype = C.c_char_p
    lib.mpc_device_status.restype = C.c_int
    lib.mpc_device_status.argtypes = [C.POINTER(C.c_int)]
    lib.mpc_abi_version.restype = C.c_int
    lib.mpc_sparse_decode_attn_static_scratch.restype = C.c_int
    lib.mpc_sparse_decode_attn_static_scratch.argtypes = [C.c_void_p, C.c_void_p]
    lib.mpc_commonality.restype = C.c_int
    lib.mpc_commonality.argtypes = [C.c_void_p, C.c_void_p]
    lib.mpc_selftest_wait.restype = C.c_int
    lib.mpc_selftest_wait.argtypes = [C.c_int32, C.c_int32, C.c_void_p, C.c_void_p]
    lib.mpc_layer_refs.restype = C.c_int
    lib.mpc_layer_refs.argtypes = [C.c_int32, C.c_int32, C.c_void_p]
    lib.mpc_choose_share_every.restype = C.c_int
    lib.mpc_choose_share_every.argtypes = [C.c_int32, C.POINTER(C.c_float), C.c_float]
    lib.mpc_decode_step_plan.restype = C.c_int
    lib.mpc_decode_step_plan.argtypes = [C.c_void_p, C.POINTER(C.c_int32)]
    if lib.mpc_abi_version() != ABI_VERSION:
        raise MPCError(MPC_ERR_INVALID_ARG,
                       f"libmpcache ABI {lib.mpc_abi_version()} does not match the binding's {ABI_VERSION}")
    if path is None:
        _LIB = lib
    return lib


class MPCError(RuntimeError):
    """A call returned a negative MPC_ERR_* code; ``code`` holds it, the message is the library's."""

    def __init__(self, code: int, msg: str):
        super().__init__(f"mpcache error {code}: {msg}")
        self.code = code


def _check(rc: int) -> None:
    if rc != MPC_OK:
        raise MPCError(rc, load().mpc_last_error().decode())


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def _dtype_code(dtype: torch.dtype) -> int:
    if dtype == torch.float32:
        return MPC_F32
    if dtype == torch.bfloat16:
        return MPC_BF16
    raise TypeError(f"unsupported dtype {dtype}: the kernels take float32 or bfloat16")


def _check_input(t: torch.Tensor, name: str, dtype: torch.dtype, shape: Sequence[Optional[int]],
                 min_layers: int = 0, host_ok: bool = False) -> None:
    """Refuses a tensor that the calls would misread: a dtype other than
    ``dtype``, sizes other than ``shape`` (None: any size; with
    ``min_layers``, dim 0 indexes layers and needs at least that many), a
    layout that is not contiguous after dim 0 (the calls take a stride for
    dim 0 only), or memory the call cannot read (host memory only where
    ``host_ok``, and then pinned)."""
    if t.dtype != dtype:
        raise TypeError(f"{name}: dtype {t.dtype}, expected {dtype}")
    want = tuple("*" if e is None else e for e in shape)
    if t.dim() != len(shape) or any(e is not None and e != n for e, n in zip(shape, t.shape)):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {want}")
    if min_layers and t.shape[0] < min_layers:
        raise ValueError(f"{name}: {t.shape[0]} layers along dim 0, the refs need {min_layers}")
    step = 1
    for n, st in zip(reversed(t.shape[1:]), reversed(t.stride()[1:])):
        if n > 1 and st != step:
            raise ValueError(f"{name}: dims after the first must be contiguous (strides {t.stride()})")
        step *= n
    if not t.is_cuda and not (host_ok and t.is_pinned()):
        raise ValueError(f"{name}: must be on the GPU" + (" or in pinned host memory" if host_ok else ""))


def _refs(refs: Sequence[tuple]):
    arr = (LayerRef * len(refs))(*[LayerRef(int(l), int(g), int(bool(ld))) for l, g, ld in refs])
    return arr


def _fan(fanouts: Sequence[int]):
    a = (C.c_int32 * MAX_LEVELS)()
    for i, f in enumerate(fanouts):
        a[i] = int(f)
    return a


def _ws_zero(nbytes: int, cache: dict, key) -> torch.Tensor:
    ws = cache.get(key)
    if ws is None or ws.numel() < nbytes:
        ws = torch.zeros(max(nbytes, 256), dtype=torch.uint8, device="cuda")
        cache[key] = ws
    return ws


# ----------------------------------------------------------- host rules ----

def ppm_count(n: int, ppm: int) -> int:
    """min(n, max(1, ceil(n * ppm / 1e6))), 0 for n = 0 (the library's rule)."""
    if n <= 0:
        return 0
    return min(n, max(1, (n * ppm + PPM - 1) // PPM))


def window_rows_bound(t_max: int, window_ppm: int, long_ppm: int, threshold: int) -> int:
    """Longest static-eviction window over prompt lengths 1..t_max."""
    a = ppm_count(min(t_max, threshold), window_ppm)
    b = ppm_count(t_max, long_ppm) if t_max > threshold else 0
    return max(a, b)


def layer_refs(n_layers: int, share_every: int):
    """mpc_layer_refs: [(layer, group, is_leader)] for layers 0 .. n_layers - 1
    under cross-layer index sharing with groups of ``share_every``."""
    arr = (LayerRef * n_layers)()
    g = load().mpc_layer_refs(n_layers, max(1, share_every), arr)
    _check(min(g, 0))
    return [(r.layer, r.group, bool(r.leader)) for r in arr]


def sharing_leader(layer: int, share_every: int) -> int:
    """Leader layer of ``layer`` under cross-layer index sharing (from
    mpc_layer_refs: layers 0 and 1 lead themselves, later layers form groups
    of ``share_every``)."""
    refs = layer_refs(layer + 1, share_every)
    group = refs[layer][1]
    return next(l for l, g, leads in refs if leads and g == group)


def commonality(sel: torch.Tensor, k: int, m: int, n_clusters: int, kept: Optional[torch.Tensor] = None,
                cluster_size: int = 1, n_keep: Optional[torch.Tensor] = None,
                prompt_len: Optional[torch.Tensor] = None):
    """Commonality of per-layer selections (Sec. 2, Observation 3; mpc_commonality).

    sel: int32 [L][B][Hkv][sel_cap] selections of consecutive layers, each its
    own leader (ids ascending, -1 padded).  Returns (total, score), each
    [B][Hkv]: total = sum over l < L - m of |S_l n ... n S_{l+m}| over the
    first k ids of each list, score = total / (k (L - m)).  With ``kept``
    (int32 [L][B][Hkv][kept_cap], each layer's kept positions) the sets are
    the token positions of the selected clusters' rows (``n_keep`` and
    ``prompt_len``, int32 [B], place the rows appended while decoding), the
    score divides by k s (L - m), and ``n_clusters`` bounds the positions.
    """
    L, B, Hkv, cap = sel.shape
    total = torch.zeros((B, Hkv), dtype=torch.int32, device=sel.device)
    score = torch.zeros((B, Hkv), dtype=torch.float32, device=sel.device)
    a = CommonalityArgs()
    a.struct_size = C.sizeof(CommonalityArgs)
    a.n_layers, a.batch, a.n_kv_heads = L, B, Hkv
    a.sel, a.sel_layer_stride, a.sel_cap = _ptr(sel), sel.stride(0), cap
    a.n_clusters, a.k, a.m = n_clusters, k, m
    a.out_total, a.out_score = _ptr(total), _ptr(score)
    if kept is not None:
        _check_input(kept, "kept", torch.int32, (L, B, Hkv, None))
        _check_input(n_keep, "n_keep", torch.int32, (B,))
        _check_input(prompt_len, "prompt_len", torch.int32, (B,))
        a.kept, a.kept_layer_stride, a.kept_cap = _ptr(kept), kept.stride(0), kept.shape[3]
        a.cluster_size, a.n_keep, a.prompt_len = cluster_size, _ptr(n_keep), _ptr(prompt_len)
    _check(load().mpc_commonality(C.byref(a), C.c_void_p(_stream())))
    return total, score


def choose_share_every(scores: dict, threshold: float) -> int:
    """mpc_choose_share_every: the adaptive sharing-group size, the largest
    m + 1 whose commonality score of m + 1 adjacent layers (``scores[m]``, e.g.
    the mean over sequences and kv heads, for m = 1 .. n) reaches
    ``threshold``, else 1 (no sharing)."""
    n = max(scores) if scores else 0
    if n < 1:
        return 1
    arr = (C.c_float * n)(*[float(scores.get(m, -1.0)) for m in range(1, n + 1)])
    r = load().mpc_choose_share_every(n, arr, float(threshold))
    _check(min(r, 0))
    return r


def summary_rows(cap_tokens: int, s: int, fanouts: Sequence[int]) -> int:
    """Rows of one summary pyramid (all levels) for ``cap_tokens`` cache rows."""
    arr = (C.c_int32 * MAX_LEVELS)(*([int(f) for f in fanouts] + [0] * (MAX_LEVELS - len(fanouts))))
    r = load().mpc_summary_rows(cap_tokens, s, 1 + len(fanouts), arr)
    if r < 0:
        _check(int(r))
    return int(r)


def device_status() -> int:
    """Synchronizes the device, then reads and clears the device status word
    (1: a bounded wait gave up, 2: a decode step had no row left, 4: an index
    out of range was skipped)."""
    v = C.c_int(0)
    _check(load().mpc_device_status(C.byref(v)))
    return v.value


def selftest_wait(kind: int, limit_us: int, never_set: Optional[torch.Tensor] = None) -> None:
    """Launches the failure-path self-test: a wait that is never satisfied
    (kind 0: an mbarrier; kind 1: ``never_set``, a device int32 kept 0) gives
    up after ``limit_us`` and sets flag 1 of the device status word."""
    _check(load().mpc_selftest_wait(kind, limit_us, C.c_void_p(_ptr(never_set)), C.c_void_p(_stream())))


# -------------------------------------------------------------- engine ----

class Engine:
    """Device state of one batch of the MPCache decode path."""

    def __init__(self, *, n_layers: int, batch: int, n_q_heads: int, n_kv_heads: int, head_dim: int,
                 dtype: torch.dtype, t_max: int, keep_ppm: int, cluster_size: int,
                 fanouts: Sequence[int], level_keep_ppm: Sequence[int], share_every: int,
                 max_decode_steps: int, alpha: float = 0.6, window_ppm: int = 200_000,
                 long_window_ppm: int = 100_000, long_prompt_threshold: int = 24_576,
                 scale: float = 0.0, layers: Optional[Sequence[int]] = None):
        load()
        self.L, self.B, self.Hq, self.Hkv, self.d = n_layers, batch, n_q_heads, n_kv_heads, head_dim
        self.dtype = dtype
        self.dcode = _dtype_code(dtype)
        self.t_max, self.keep_ppm, self.s = t_max, keep_ppm, cluster_size
        self.fanouts = tuple(fanouts)
        self.n_levels = 1 + len(self.fanouts)
        self.level_keep_ppm = tuple(level_keep_ppm)
        assert len(self.level_keep_ppm) == self.n_levels
        self.share_every = share_every
        self.alpha, self.scale = alpha, scale
        self.window_ppm, self.long_window_ppm, self.long_threshold = window_ppm, long_window_ppm, long_prompt_threshold
        self.layers = list(range(n_layers)) if layers is None else list(layers)
        full = layer_refs(n_layers, share_every)  # (layer, group, leads) from mpc_layer_refs
        lead_of_group = {g: l for l, g, leads in full if leads}
        lead = [lead_of_group[g] for _, g, _ in full]
        self.leaders = sorted(set(lead[l] for l in self.layers))
        self.group_of = {l: self.leaders.index(lead[l]) for l in self.layers}
        self.refs_all = [(l, self.group_of[l], lead[l] == l) for l in self.layers]
        self.refs_lead = [(l, self.group_of[l], True) for l in self.leaders]
        missing = [l for l in self.leaders if l not in self.layers]
        if missing:
            raise ValueError(f"leader layers {missing} must be among the processed layers")
        self.n_groups = len(self.leaders)
        self.win_rows = window_rows_bound(t_max, window_ppm, long_window_ppm, long_prompt_threshold)
        self.keep_cap = ppm_count(t_max, keep_ppm)
        s = cluster_size
        self.cap_tokens = ((self.keep_cap + max_decode_steps + s - 1) // s) * s + s
        self.rows = summary_rows(self.cap_tokens, s, self.fanouts)
        self.sel_cap = max(1, ppm_count(self.cap_tokens // s, self.level_keep_ppm[0]))
        dev = "cuda"
        f32, i32 = dict(dtype=torch.float32, device=dev), dict(dtype=torch.int32, device=dev)
        G, B, Hkv, d = self.n_groups, batch, n_kv_heads, head_dim
        self.scores = torch.zeros((G, B, Hkv, t_max), **f32)
        self.kept = torch.zeros((G, B, Hkv, self.keep_cap), **i32)
        self.n_keep = torch.zeros((B,), **i32)
        self.kc = torch.zeros((n_layers, B, Hkv, self.cap_tokens, d), dtype=dtype, device=dev)
        self.vc = torch.zeros_like(self.kc)
        self.rmax = torch.zeros((G, B, Hkv, self.rows, d), **f32)
        self.mean = torch.zeros((G, B, Hkv, self.rows, d), **f32)  # mean member key per cluster
        self.rmin = torch.zeros_like(self.rmax)
        self.rep = torch.zeros_like(self.rmax)
        self.n_tok = torch.zeros((B,), **i32)
        self.sel = torch.full((G, B, Hkv, self.sel_cap), -1, **i32)
        self.n_sel = torch.zeros((B,), **i32)
        self.out = torch.zeros((n_layers, B, n_q_heads, d), **f32)
        self.prompt_lens = None  # the lens of the last static eviction (device int32 [B])
        self._ws = {}

    def check_status(self) -> int:
        """Synchronizes, then reads and clears the device status word (see
        ``device_status``).  A bounded wait that gave up (flag 1) can leave the
        split-merge counters of a decode workspace nonzero, and the calls
        require a zero-filled workspace again after that, so this engine's
        workspaces are cleared before the flags are returned."""
        st = device_status()
        if st & 1:
            for ws in self._ws.values():
                ws.zero_()
            torch.cuda.synchronize()
        return st

    # --------------------------------------------------------- prefill ----
    @staticmethod
    def _subset(refs_list, layers):
        """The refs of ``layers`` (all refs when None)."""
        if layers is None:
            return refs_list
        keep = set(int(l) for l in layers)
        return [r for r in refs_list if r[0] in keep]

    def static_args(self, k: torch.Tensor, q_win: torch.Tensor, lens: torch.Tensor,
                    page_table: Optional[torch.Tensor] = None, page_size: int = 16,
                    layers: Optional[Sequence[int]] = None) -> StaticArgs:
        """The checked mpc_static_args of the leader layers (of ``layers``
        only, if given); the returned struct keeps its refs array alive."""
        # the C call refuses fewer window rows than the longest window of a
        # t_max-token prompt too; this names the tensor in the message
        if q_win.dim() == 5 and q_win.shape[3] < self.win_rows:
            raise ValueError(f"q_win: {q_win.shape[3]} window rows, the engine's prompts need up to "
                             f"{self.win_rows}")
        lead = self._subset(self.refs_lead, layers)
        span = 1 + max((r[0] for r in lead), default=-1)
        self._check_kv(k, "k", page_table, page_size, span, host_ok=False)
        _check_input(q_win, "q_win", self.dtype, (None, self.B, self.Hq, None, self.d), span)
        _check_input(lens, "lens", torch.int32, (self.B,))
        refs = _refs(lead)
        a = StaticArgs()
        a.struct_size = C.sizeof(StaticArgs)
        a.n_refs = len(lead)
        a.refs = C.cast(refs, C.POINTER(LayerRef))
        a.batch, a.n_q_heads, a.n_kv_heads, a.head_dim, a.dtype = self.B, self.Hq, self.Hkv, self.d, self.dcode
        a.t_max = self.t_max
        a.prompt_lens = _ptr(lens)
        a.q_win = _ptr(q_win)
        a.q_win_layer_stride = q_win.stride(0)
        a.win_rows = q_win.shape[3]
        a.k = self._kv(k, page_table, page_size)
        a.window_ppm, a.long_window_ppm, a.long_prompt_threshold = (self.window_ppm, self.long_window_ppm,
                                                                   self.long_threshold)
        a.keep_ppm = self.keep_ppm
        a.scale = self.scale
        a.keep_cap = self.keep_cap
        a.out_scores, a.out_kept, a.out_n_keep = _ptr(self.scores), _ptr(self.kept), _ptr(self.n_keep)
        a._refs = refs
        return a

    def _check_kv(self, t: torch.Tensor, name: str, page_table, page_size: int, span: int, host_ok: bool):
        """Prompt keys or values: dense [layer][b][kv head][t_max][d], or a
        page pool [layer][page][kv head][page_size][d] with its page table
        [b][max_pages] (int32, on the GPU)."""
        if page_table is None:
            _check_input(t, name, self.dtype, (None, self.B, self.Hkv, self.t_max, self.d), span, host_ok)
        else:
            _check_input(t, name, self.dtype, (None, None, self.Hkv, page_size, self.d), span, host_ok)
            _check_input(page_table, "page_table", torch.int32, (self.B, None))

    def _kv(self, t: torch.Tensor, page_table, page_size) -> KvTensor:
        kv = KvTensor()
        kv.data = _ptr(t)
        kv.layer_stride = t.stride(0)
        if page_table is not None:
            kv.page_table = _ptr(page_table)
            kv.page_size = page_size
            kv.max_pages = page_table.shape[1]
        return kv

    def static_evict(self, k, q_win, lens, page_table=None, page_size=16, layers=None):
        """Static eviction of the leader layers (of ``layers`` only, if given)."""
        lib = load()
        a = self.static_args(k, q_win, lens, page_table, page_size, layers)
        n = C.c_size_t(0)
        _check(lib.mpc_static_evict_workspace_size(C.byref(a), C.byref(n)))
        ws = _ws_zero(n.value, self._ws, "static")
        _check(lib.mpc_static_evict(C.byref(a), C.c_void_p(_ptr(ws)), n.value, C.c_void_p(_stream())))
        self.prompt_lens = lens

    def build_clusters(self, k, v, page_table=None, page_size=16, layers=None):
        """Gathering and clustering of every layer (of ``layers`` only, if
        given).  k and v may be pinned host tensors: the gather then reads
        only the kept rows across the host link."""
        lib = load()
        sub = self._subset(self.refs_all, layers)
        span = 1 + max((r[0] for r in sub), default=-1)
        self._check_kv(k, "k", page_table, page_size, span, host_ok=True)
        self._check_kv(v, "v", page_table, page_size, span, host_ok=True)
        refs = _refs(sub)
        a = ClusterArgs()
        a.struct_size = C.sizeof(ClusterArgs)
        a.n_refs = len(sub)
        a.refs = C.cast(refs, C.POINTER(LayerRef))
        a.batch, a.n_kv_heads, a.head_dim, a.dtype = self.B, self.Hkv, self.d, self.dcode
        a.t_max = self.t_max
        a.k = self._kv(k, page_table, page_size)
        a.v = self._kv(v, page_table, page_size)
        a.kept, a.keep_cap, a.n_keep = _ptr(self.kept), self.keep_cap, _ptr(self.n_keep)
        a.kc, a.vc, a.cache_layer_stride, a.cap_tokens = _ptr(self.kc), _ptr(self.vc), self.kc.stride(0), self.cap_tokens
        a.r_max, a.r_min, a.rep, a.summary_rows = _ptr(self.rmax), _ptr(self.rmin), _ptr(self.rep), self.rows
        a.mean = _ptr(self.mean)
        a.cluster_size, a.n_levels, a.fanout, a.alpha = self.s, self.n_levels, _fan(self.fanouts), self.alpha
        a.out_n_tok = _ptr(self.n_tok)
        _check(lib.mpc_build_clusters(C.byref(a), None, 0, C.c_void_p(_stream())))

    def prefill(self, k, v, q_win, lens, page_table=None, page_size=16):
        """Static eviction (leaders) + gathering and clustering (all layers)."""
        self.static_evict(k, q_win, lens, page_table, page_size)
        self.build_clusters(k, v, page_table, page_size)

    # ---------------------------------------------------------- decode ----
    def select(self, q: torch.Tensor, metric: int = MPC_SIM_EQ3, frac_bits: int = FXP_FRAC_BITS):
        """q: [L][B][Hq][d] queries of this step (only the leaders' are read);
        metric MPC_SIM_EQ3 (Eq. 3 with rep), MPC_SIM_BOUND (Eq. 2 bound),
        MPC_SIM_MEAN (mean member key) or MPC_SIM_FXP (Eq. 3 in the
        fixed-point ring with ``frac_bits`` fractional bits and the cache's alpha)."""
        lib = load()
        _check_input(q, "q", self.dtype, (None, self.B, self.Hq, self.d), 1 + max(self.leaders))
        refs = _refs(self.refs_lead)
        a = SelectArgs()
        a.struct_size = C.sizeof(SelectArgs)
        a.n_refs = len(self.refs_lead)
        a.refs = C.cast(refs, C.POINTER(LayerRef))
        a.batch, a.n_q_heads, a.n_kv_heads, a.head_dim, a.dtype = self.B, self.Hq, self.Hkv, self.d, self.dcode
        a.q, a.q_layer_stride = _ptr(q), q.stride(0)
        a.rep, a.summary_rows, a.cap_tokens, a.n_tok = _ptr(self.rep), self.rows, self.cap_tokens, _ptr(self.n_tok)
        a.cluster_size, a.n_levels, a.fanout = self.s, self.n_levels, _fan(self.fanouts)
        a.level_keep_ppm = _fan(self.level_keep_ppm)
        a.sel_cap, a.out_sel, a.out_n_sel = self.sel_cap, _ptr(self.sel), _ptr(self.n_sel)
        a.metric, a.r_max, a.r_min, a.mean = metric, _ptr(self.rmax), _ptr(self.rmin), _ptr(self.mean)
        a.alpha, a.frac_bits = self.alpha, frac_bits
        _check(lib.mpc_select(C.byref(a), None, 0, C.c_void_p(_stream())))

    def attn_args(self, q, k_new, v_new, advance=True, refs_list=None, out=None) -> AttnArgs:
        """The checked mpc_attn_args of one decode step for ``refs_list``
        (default: every processed layer); the struct keeps its refs array alive."""
        refs_list = self.refs_all if refs_list is None else refs_list
        out = self.out if out is None else out
        span = 1 + max((r[0] for r in refs_list), default=-1)
        _check_input(q, "q", self.dtype, (None, self.B, self.Hq, self.d), span)
        _check_input(k_new, "k_new", self.dtype, (None, self.B, self.Hkv, self.d), span)
        _check_input(v_new, "v_new", self.dtype, (None, self.B, self.Hkv, self.d), span)
        _check_input(out, "out", torch.float32, (None, self.B, self.Hq, self.d), span)
        if v_new.stride(0) != k_new.stride(0):
            raise ValueError("k_new and v_new must have the same layer stride")
        refs = _refs(refs_list)
        a = AttnArgs()
        a.struct_size = C.sizeof(AttnArgs)
        a.n_refs = len(refs_list)
        a.refs = C.cast(refs, C.POINTER(LayerRef))
        a.batch, a.n_q_heads, a.n_kv_heads, a.head_dim, a.dtype = self.B, self.Hq, self.Hkv, self.d, self.dcode
        a.q, a.k_new, a.v_new = _ptr(q), _ptr(k_new), _ptr(v_new)
        a.q_layer_stride, a.kv_new_layer_stride = q.stride(0), k_new.stride(0)
        a.kc, a.vc, a.cache_layer_stride, a.cap_tokens = _ptr(self.kc), _ptr(self.vc), self.kc.stride(0), self.cap_tokens
        a.sel, a.n_sel, a.sel_cap = _ptr(self.sel), _ptr(self.n_sel), self.sel_cap
        a.r_max, a.r_min, a.rep, a.summary_rows = _ptr(self.rmax), _ptr(self.rmin), _ptr(self.rep), self.rows
        a.mean = _ptr(self.mean)
        a.cluster_size, a.n_levels, a.fanout, a.alpha = self.s, self.n_levels, _fan(self.fanouts), self.alpha
        a.n_tok, a.advance, a.scale = _ptr(self.n_tok), int(bool(advance)), self.scale
        a.out, a.out_layer_stride = _ptr(out), out.stride(0)
        a._refs = refs  # keeps the host array alive as long as the args
        return a

    def attend(self, q, k_new, v_new, advance=True, out=None):
        """Append + sparse attention for every layer; writes ``out``
        ([L][B][Hq][d] float32, default ``self.out``)."""
        lib = load()
        a = self.attn_args(q, k_new, v_new, advance, out=out)
        n = C.c_size_t(0)
        _check(lib.mpc_sparse_decode_attn_workspace_size(C.byref(a), C.byref(n)))
        ws = _ws_zero(n.value, self._ws, "attn")
        _check(lib.mpc_sparse_decode_attn(C.byref(a), C.c_void_p(_ptr(ws)), n.value, C.c_void_p(_stream())))

    def step_args(self, q, k_new, v_new, advance=True, out=None, metric: int = MPC_SIM_EQ3,
                  frac_bits: int = FXP_FRAC_BITS, speculate: int = -1, static_ppm: int = 0,
                  slice_tiles: int = 0, fuse: int = -1) -> DecodeArgs:
        """The checked mpc_decode_args of one whole decode step of every
        processed layer (selection of the leaders, then attention)."""
        a = DecodeArgs()
        a.struct_size = C.sizeof(DecodeArgs)
        att = self.attn_args(q, k_new, v_new, advance, out=out)
        a.attn = att  # copied into the struct; its refs pointer still names att's array
        a._refs = att._refs  # which stays alive as long as the args
        a.level_keep_ppm = _fan(self.level_keep_ppm)
        a.metric, a.frac_bits, a.speculate = metric, frac_bits, speculate
        a.static_ppm, a.slice_tiles, a.fuse = static_ppm, slice_tiles, fuse
        return a

    def decode_step(self, q, k_new, v_new, out=None, metric: int = MPC_SIM_EQ3, speculate: int = -1,
                    static_ppm: int = 0, slice_tiles: int = 0, fuse: int = -1):
        """One decode step of every layer in one call (mpc_decode_step):
        q [L][B][Hq][d], k_new / v_new [L][B][Hkv][d] (layer index = position
        along dim 0).  Same selections and outputs as ``select`` followed by
        ``attend``; ``fuse`` = 1 runs the step as one fused kernel, 0 as the
        selection and attention launches, -1 lets the library choose."""
        lib = load()
        a = self.step_args(q, k_new, v_new, True, out, metric, speculate=speculate, static_ppm=static_ppm,
                           slice_tiles=slice_tiles, fuse=fuse)
        n = C.c_size_t(0)
        _check(lib.mpc_decode_step_workspace_size(C.byref(a), C.byref(n)))
        ws = _ws_zero(n.value, self._ws, "step")
        _check(lib.mpc_decode_step(C.byref(a), C.c_void_p(_ptr(ws)), n.value, C.c_void_p(_stream())))

    def commonality(self, m: int):
        """Commonality score of windows of m + 1 adjacent layers over this
        step's selections (the last select or decode step), compared as the
        token positions of the selected clusters.  Every processed layer
        must lead its own group (share_every = 1, consecutive layers).  The
        sets hold the first k clusters of each list, k the fewest selected by
        a sequence of the batch; returns (total, score), each [B][Hkv] on the
        device."""
        if self.n_groups != len(self.layers) or self.layers != list(range(self.layers[0], self.layers[-1] + 1)):
            raise ValueError("commonality needs consecutive layers, each its own leader (share_every = 1)")
        if self.prompt_lens is None:
            raise ValueError("commonality needs the prefill's prompt lengths (run static_evict first)")
        bound = self.t_max + self.cap_tokens  # every position: prompt rows and appended rows
        k = int(self.n_sel.min())
        if k < 1:
            raise ValueError("commonality needs a selection of at least one cluster per sequence")
        return commonality(self.sel, k, m, bound, kept=self.kept, cluster_size=self.s,
                           n_keep=self.n_keep, prompt_len=self.prompt_lens)

    def decode_step_launches(self, q, k_new, v_new, out=None, metric: int = MPC_SIM_EQ3, fuse: int = -1) -> int:
        """Kernel launches ``decode_step`` makes with these arguments
        (mpc_decode_step_plan: 1 for the fused kernel, 2 otherwise)."""
        a = self.step_args(q, k_new, v_new, True, out, metric, fuse=fuse)
        n = C.c_int32(0)
        _check(load().mpc_decode_step_plan(C.byref(a), C.byref(n)))
        return n.value

    def decode_step_two_calls(self, q, k_new, v_new, out=None):
        """The same decode step as two calls: ``select`` (leaders), then
        ``attend`` (every layer)."""
        self.select(q)
        self.attend(q, k_new, v_new, advance=True, out=out)
