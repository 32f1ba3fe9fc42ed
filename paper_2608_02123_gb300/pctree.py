"""Python binding of the PCTree C ABI (include/pctree.h).

Argument marshalling only: every step of a drafting round runs in the CUDA
library ``_build/libpctree_gb300.so``.  PyTorch supplies device memory and
streams; tensors are passed to the library as raw device pointers.  If the
library is missing, importing this module raises -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import math
import dataclasses
import os
from typing import Dict, Optional

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "_build",
                         "libpctree_gb300.so")

PCTREE_OK = 0
PCTREE_F32 = 0
PCTREE_BF16 = 1
MAX_K, MAX_N, MAX_POOL, MAX_ROWS = 32, 1024, 16384, 4096

STATUS_NAMES = {0: "ok", -1: "invalid argument", -2: "workspace",
                -3: "CUDA error", -4: "timeout", -5: "non-finite input",
                -6: "unsupported shape"}


class PctreeError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)} ({code})")
        self.code = code


class Config(ctypes.Structure):
    _fields_ = [("V", ctypes.c_int32), ("H", ctypes.c_int32),
                ("B", ctypes.c_int32), ("k", ctypes.c_int32),
                ("N", ctypes.c_int32), ("batch", ctypes.c_int32),
                ("pos_offset", ctypes.c_int32),
                ("weight_dtype", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("head_layout", ctypes.c_int32)]


class CompactLayout(ctypes.Structure):
    """pctree_compact_layout: shapes and byte strides of the cache planes."""
    _fields_ = [("batch", ctypes.c_int32), ("B", ctypes.c_int32),
                ("N", ctypes.c_int32), ("layers", ctypes.c_int32),
                ("planes", ctypes.c_int32), ("max_slots", ctypes.c_int32),
                ("row_bytes", ctypes.c_int64), ("slot_stride", ctypes.c_int64),
                ("request_stride", ctypes.c_int64),
                ("plane_stride", ctypes.c_int64),
                ("layer_stride", ctypes.c_int64),
                ("hidden_bytes", ctypes.c_int64)]


class AttnConfig(ctypes.Structure):
    """pctree_attn_config: one grouped-query attention layer."""
    _fields_ = [("batch", ctypes.c_int32), ("N", ctypes.c_int32),
                ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("D", ctypes.c_int32), ("max_slots", ctypes.c_int32),
                ("scale", ctypes.c_float)]


class _Tree(ctypes.Structure):
    _fields_ = [(name, ctypes.c_void_p) for name in (
        "n_nodes", "tokens", "parent", "depth", "logp", "position_ids",
        "mask", "retrieve", "n_leaves", "status", "pool_token",
        "pool_parent", "pool_logp")]


def _load() -> ctypes.CDLL:
    if not os.path.exists(_LIB_PATH):
        raise ImportError(
            f"PCTree CUDA library not built ({_LIB_PATH}); run "
            "`python -m paper_2608_02123_gb300.build`")
    lib = ctypes.CDLL(_LIB_PATH)
    vp, cfgp = ctypes.c_void_p, ctypes.POINTER(Config)
    lib.pctree_check_config.argtypes = [cfgp]
    lib.pctree_check_config.restype = ctypes.c_int
    lib.pctree_pool_capacity.argtypes = [cfgp]
    lib.pctree_pool_capacity.restype = ctypes.c_int32
    lib.pctree_workspace_bytes.argtypes = [cfgp]
    lib.pctree_workspace_bytes.restype = ctypes.c_size_t
    lib.pctree_draft.argtypes = [cfgp, vp, vp, vp, vp, ctypes.POINTER(_Tree),
                                 vp, ctypes.c_size_t, vp]
    lib.pctree_draft.restype = ctypes.c_int
    lib.pctree_draft_noalloc.argtypes = [cfgp, vp, vp, vp, vp,
                                         ctypes.POINTER(_Tree), vp]
    lib.pctree_draft_noalloc.restype = ctypes.c_int
    lib.pctree_packed_head_bytes.argtypes = [cfgp]
    lib.pctree_packed_head_bytes.restype = ctypes.c_size_t
    lib.pctree_pack_head.argtypes = [cfgp, vp, vp, vp]
    lib.pctree_pack_head.restype = ctypes.c_int
    lib.pctree_accept.argtypes = [cfgp, ctypes.POINTER(_Tree), vp, vp, vp, vp,
                                  vp]
    lib.pctree_accept.restype = ctypes.c_int
    lib.pctree_compact.argtypes = [ctypes.POINTER(CompactLayout), vp, vp, vp,
                                   vp, vp, vp, vp, vp]
    lib.pctree_compact.restype = ctypes.c_int
    ap = ctypes.POINTER(AttnConfig)
    lib.pctree_tree_attention_workspace_bytes.argtypes = [ap]
    lib.pctree_tree_attention_workspace_bytes.restype = ctypes.c_size_t
    lib.pctree_tree_attention.argtypes = [ap] + [vp] * 8 + [ctypes.c_size_t,
                                                           vp, vp]
    lib.pctree_tree_attention.restype = ctypes.c_int
    lib.pctree_status_string.argtypes = [ctypes.c_int32]
    lib.pctree_status_string.restype = ctypes.c_char_p
    lib.pctree_profile_enable.argtypes = [ctypes.c_int32]
    lib.pctree_profile_enable.restype = ctypes.c_int
    lib.pctree_profile_collect.argtypes = [ctypes.POINTER(ctypes.c_int64),
                                           ctypes.POINTER(ctypes.c_double)]
    lib.pctree_profile_collect.restype = ctypes.c_int
    lib.pctree_set_path.argtypes = [ctypes.c_int32]
    lib.pctree_set_path.restype = ctypes.c_int
    lib.pctree_debug_stall_stage.argtypes = [ctypes.c_int32, ctypes.c_int64]
    lib.pctree_debug_stall_stage.restype = ctypes.c_int
    lib.pctree_version.argtypes = []
    lib.pctree_version.restype = ctypes.c_int32
    return lib


LIB = _load()
LIB_PATH = _LIB_PATH


MODE_PARENT, MODE_SHARED = 0, 1
HEAD_ROWMAJOR, HEAD_TILED = 0, 1


def make_config(V: int, H: int, B: int, k: int, N: int, batch: int = 1,
                pos_offset: int = 0, weight_dtype: str = "bf16",
                mode: str = "parent", head_layout: str = "rowmajor") -> Config:
    """``mode``: "parent" (PCTree) or "shared" (the Shared-Markov control).
    ``head_layout``: "rowmajor" ([V][H]) or "tiled" (see pctree_pack_head)."""
    return Config(V, H, B, k, N, batch, pos_offset,
                  PCTREE_BF16 if weight_dtype == "bf16" else PCTREE_F32,
                  MODE_SHARED if mode == "shared" else MODE_PARENT,
                  HEAD_TILED if head_layout == "tiled" else HEAD_ROWMAJOR)


def pctree_packed_head_bytes(cfg: Config) -> int:
    return LIB.pctree_packed_head_bytes(ctypes.byref(cfg))


def pctree_pack_head(cfg: Config, head_out: torch.Tensor, packed: torch.Tensor,
                     stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue the repacking of a row-major bf16 W_out into the tiled layout
    (see pctree_pack_head in include/pctree.h)."""
    if not head_out.is_cuda or not head_out.is_contiguous() or not packed.is_cuda:
        raise ValueError("head_out and packed must be CUDA tensors (head_out contiguous)")
    if packed.numel() * packed.element_size() < pctree_packed_head_bytes(cfg):
        raise ValueError("packed is smaller than pctree_packed_head_bytes")
    rc = LIB.pctree_pack_head(ctypes.byref(cfg), head_out.data_ptr(),
                              packed.data_ptr(), _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_pack_head")


def pack_head(cfg: Config, head_out: torch.Tensor) -> torch.Tensor:
    """A new device tensor holding head_out in the tiled layout."""
    nbytes = pctree_packed_head_bytes(cfg)
    if nbytes == 0:
        raise PctreeError(-1, "pctree_packed_head_bytes")
    packed = torch.empty(nbytes // 2, dtype=torch.bfloat16, device=head_out.device)
    pctree_pack_head(cfg, head_out, packed)
    return packed


def pctree_check_config(cfg: Config) -> int:
    return LIB.pctree_check_config(ctypes.byref(cfg))


def pctree_pool_capacity(cfg: Config) -> int:
    return LIB.pctree_pool_capacity(ctypes.byref(cfg))


def pctree_workspace_bytes(cfg: Config) -> int:
    return LIB.pctree_workspace_bytes(ctypes.byref(cfg))


def pctree_status_string(code: int) -> str:
    return LIB.pctree_status_string(code).decode()


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


@dataclasses.dataclass
class Tree:
    """Device tensors of drafted trees (see pctree_tree in include/pctree.h)."""

    n_nodes: torch.Tensor
    tokens: torch.Tensor
    parent: torch.Tensor
    depth: torch.Tensor
    logp: torch.Tensor
    position_ids: torch.Tensor
    mask: torch.Tensor
    retrieve: torch.Tensor
    n_leaves: torch.Tensor
    status: torch.Tensor
    pool_token: Optional[torch.Tensor] = None
    pool_parent: Optional[torch.Tensor] = None
    pool_logp: Optional[torch.Tensor] = None

    def c_struct(self) -> _Tree:
        return _Tree(*[_ptr(getattr(self, f.name))
                       for f in dataclasses.fields(self)])

    def to_host(self) -> Dict[str, "object"]:
        return {f.name: (None if getattr(self, f.name) is None
                         else getattr(self, f.name).cpu().numpy())
                for f in dataclasses.fields(self)}


def _carve(device, specs):
    """Tensors of the given (name, shape, dtype) as views of one device
    buffer, each starting on a 256-byte boundary: a caller reads them all
    back with one copy.  Returns (buffer, {name: tensor})."""
    offs, off = [], 0
    for name, shape, dt in specs:
        n = math.prod(shape) * torch.empty(0, dtype=dt).element_size()
        offs.append((name, off, n, shape, dt))
        off = (off + n + 255) // 256 * 256
    blob = torch.empty(max(off, 256), dtype=torch.uint8, device=device)
    return blob, {name: blob[o:o + n].view(dt).view(*shape)
                  for name, o, n, shape, dt in offs}


def alloc_tree(cfg: Config, device, with_pool: bool = False, extra=()) -> Tree:
    """The output tensors of a round, carved from one device buffer
    (``tree.blob``) together with the ``extra`` (name, shape, dtype) tensors
    (``tree.extra``), so that all of them come back with one copy."""
    R, N, B = cfg.batch, cfg.N, cfg.B
    i32, f32, u8 = torch.int32, torch.float32, torch.uint8
    P = pctree_pool_capacity(cfg)
    specs = [("n_nodes", (R,), i32), ("tokens", (R, N), i32),
             ("parent", (R, N), i32), ("depth", (R, N), i32),
             ("logp", (R, N), f32), ("position_ids", (R, N), i32),
             ("mask", (R, N, N), u8), ("retrieve", (R, N, B + 1), i32),
             ("n_leaves", (R,), i32), ("status", (1,), i32)] + list(extra)
    blob, t = _carve(device, specs)
    tree = Tree(
        n_nodes=t["n_nodes"], tokens=t["tokens"], parent=t["parent"],
        depth=t["depth"], logp=t["logp"], position_ids=t["position_ids"],
        mask=t["mask"], retrieve=t["retrieve"], n_leaves=t["n_leaves"],
        status=t["status"],
        pool_token=torch.empty(R, P, dtype=i32, device=device) if with_pool else None,
        pool_parent=torch.empty(R, P, dtype=i32, device=device) if with_pool else None,
        pool_logp=(torch.empty(R, P, dtype=f32, device=device)
                   if with_pool else None))
    tree.blob = blob
    tree.extra = {name: t[name] for name, _, _ in extra}
    return tree


def alloc_workspace(cfg: Config, device) -> torch.Tensor:
    nbytes = pctree_workspace_bytes(cfg)
    if nbytes == 0:
        raise PctreeError(pctree_check_config(cfg), "pctree_workspace_bytes")
    # torch's caching allocator returns 512-byte aligned blocks
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def _stream_ptr(stream: Optional[torch.cuda.Stream]) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def _check_inputs(base_logits, head_emb, head_out, root_token) -> None:
    for name, t in (("base_logits", base_logits), ("head_emb", head_emb),
                    ("head_out", head_out), ("root_token", root_token)):
        host_ok = name in ("base_logits", "root_token")
        ok = t.is_cuda or (host_ok and t.is_pinned())
        if not ok or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous CUDA tensor"
                             + (" or a pinned CPU tensor" if host_ok else ""))


def pctree_draft(cfg: Config, base_logits: torch.Tensor, head_emb: torch.Tensor,
                 head_out: torch.Tensor, root_token: torch.Tensor, tree: Tree,
                 workspace: torch.Tensor,
                 stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue one drafting round (see pctree_draft in include/pctree.h).
    base_logits and root_token may also be pinned CPU tensors: the kernels
    read them over the host link."""
    _check_inputs(base_logits, head_emb, head_out, root_token)
    ts = tree.c_struct()
    rc = LIB.pctree_draft(ctypes.byref(cfg), base_logits.data_ptr(),
                          head_emb.data_ptr(), head_out.data_ptr(),
                          root_token.data_ptr(), ctypes.byref(ts),
                          workspace.data_ptr(), workspace.numel(),
                          _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_draft")


def pctree_draft_noalloc(cfg: Config, base_logits: torch.Tensor,
                         head_emb: torch.Tensor, head_out: torch.Tensor,
                         root_token: torch.Tensor, tree: Tree,
                         stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue one drafting round without a workspace: the library's fixed
    16 MiB device array serves as scratch, for callers that cannot allocate
    device memory when they draft (see pctree_draft_noalloc in
    include/pctree.h)."""
    _check_inputs(base_logits, head_emb, head_out, root_token)
    ts = tree.c_struct()
    rc = LIB.pctree_draft_noalloc(ctypes.byref(cfg), base_logits.data_ptr(),
                                  head_emb.data_ptr(), head_out.data_ptr(),
                                  root_token.data_ptr(), ctypes.byref(ts),
                                  _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_draft_noalloc")


def pctree_accept(cfg: Config, tree: Tree, target_tokens: torch.Tensor,
                  accepted_idx: torch.Tensor, accepted_len: torch.Tensor,
                  bonus_token: torch.Tensor,
                  stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue the greedy tree acceptance (see pctree_accept)."""
    ts = tree.c_struct()
    rc = LIB.pctree_accept(ctypes.byref(cfg), ctypes.byref(ts),
                           target_tokens.data_ptr(), accepted_idx.data_ptr(),
                           accepted_len.data_ptr(), bonus_token.data_ptr(),
                           _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_accept")


def compact_layout(batch: int, B: int, N: int, layers: int, planes: int,
                   max_slots: int, row_bytes: int, hidden_bytes: int = 0,
                   slot_stride: Optional[int] = None,
                   request_stride: Optional[int] = None,
                   plane_stride: Optional[int] = None,
                   layer_stride: Optional[int] = None) -> CompactLayout:
    """Layout of caches shaped ``[layers][planes][batch][max_slots][row]``
    unless strides (bytes) are given."""
    ss = row_bytes if slot_stride is None else slot_stride
    rs = ss * max_slots if request_stride is None else request_stride
    ps = rs * batch if plane_stride is None else plane_stride
    ls = ps * planes if layer_stride is None else layer_stride
    return CompactLayout(batch, B, N, layers, planes, max_slots, row_bytes,
                         ss, rs, ps, ls, hidden_bytes)


def pctree_compact(layout: CompactLayout, accepted_idx: torch.Tensor,
                   accepted_len: torch.Tensor, prefix_len: torch.Tensor,
                   cache: Optional[torch.Tensor],
                   hidden_in: Optional[torch.Tensor] = None,
                   hidden_out: Optional[torch.Tensor] = None,
                   status: Optional[torch.Tensor] = None,
                   stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue the accepted-row compaction (see pctree_compact)."""
    rc = LIB.pctree_compact(ctypes.byref(layout), accepted_idx.data_ptr(),
                            accepted_len.data_ptr(), prefix_len.data_ptr(),
                            _ptr(cache), _ptr(hidden_in), _ptr(hidden_out),
                            _ptr(status), _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_compact")


def attn_config(batch: int, N: int, Hq: int, Hkv: int, max_slots: int,
                D: int = 128, scale: Optional[float] = None) -> AttnConfig:
    """``scale`` defaults to 1/sqrt(D)."""
    return AttnConfig(batch, N, Hq, Hkv, D, max_slots,
                      D ** -0.5 if scale is None else scale)


def pctree_tree_attention_workspace_bytes(cfg: AttnConfig) -> int:
    return LIB.pctree_tree_attention_workspace_bytes(ctypes.byref(cfg))


def pctree_tree_attention(cfg: AttnConfig, q: torch.Tensor, k_cache: torch.Tensor,
                          v_cache: torch.Tensor, prefix_len: torch.Tensor,
                          n_nodes: torch.Tensor, parent: torch.Tensor,
                          out: torch.Tensor,
                          workspace: Optional[torch.Tensor] = None,
                          status: Optional[torch.Tensor] = None,
                          stream: Optional[torch.cuda.Stream] = None) -> None:
    """Enqueue one tree-verification attention layer (see
    pctree_tree_attention)."""
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    rc = LIB.pctree_tree_attention(ctypes.byref(cfg), q.data_ptr(),
                                   k_cache.data_ptr(), v_cache.data_ptr(),
                                   prefix_len.data_ptr(), n_nodes.data_ptr(),
                                   parent.data_ptr(), out.data_ptr(),
                                   _ptr(workspace), ws_bytes, _ptr(status),
                                   _stream_ptr(stream))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_tree_attention")


def pctree_profile_enable(on: bool) -> None:
    rc = LIB.pctree_profile_enable(1 if on else 0)
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_profile_enable")


def pctree_profile_collect():
    """Returns (launches, total milliseconds) of timed Markov projections."""
    n = ctypes.c_int64(0)
    ms = ctypes.c_double(0.0)
    rc = LIB.pctree_profile_collect(ctypes.byref(n), ctypes.byref(ms))
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_profile_collect")
    return int(n.value), float(ms.value)


PATH_AUTO, PATH_STAGEWISE = 0, 1


def pctree_set_path(path: int) -> None:
    """Select the kernel path (see pctree_set_path in include/pctree.h)."""
    rc = LIB.pctree_set_path(path)
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_set_path")


def uses_fused_round(cfg: Config, path: int = PATH_AUTO) -> bool:
    """Whether a round of `cfg` runs as one fused launch (mirrors the
    library's choice)."""
    return (path == PATH_AUTO and cfg.weight_dtype == PCTREE_BF16 and
            cfg.batch * cfg.k <= 16 and cfg.k <= 16)


def kernels_per_round(cfg: Config, path: int = PATH_AUTO) -> int:
    """Kernels of this library one pctree_draft launches."""
    if uses_fused_round(cfg, path):
        return 3                      # init, fused round, pack
    launches = 2                      # init, pack
    for d in range(cfg.B):
        rpq = 1 if (cfg.mode == MODE_SHARED or d == 0) else cfg.k
        rows = cfg.batch * rpq
        if cfg.weight_dtype == PCTREE_BF16:
            # projection passes (normaliser and top-k partials folded in), merge
            launches += (rows + 255) // 256 + 1
        else:
            launches += 3             # projection, partials, merge
    return launches


def pctree_version() -> int:
    return LIB.pctree_version()


class Drafter:
    """Owns the device workspace and output tensors for one configuration."""

    def __init__(self, cfg: Config, device="cuda", with_pool: bool = False):
        rc = pctree_check_config(cfg)
        if rc != PCTREE_OK:
            raise PctreeError(rc, "pctree_check_config")
        self.cfg = cfg
        self.device = torch.device(device)
        self.workspace = alloc_workspace(cfg, self.device)
        # the acceptance outputs share the tree's buffer (one copy back)
        self.tree = alloc_tree(cfg, self.device, with_pool, extra=(
            ("accepted_idx", (cfg.batch, cfg.B + 1), torch.int32),
            ("accepted_len", (cfg.batch,), torch.int32),
            ("bonus", (cfg.batch,), torch.int32)))
        self.accepted_idx = self.tree.extra["accepted_idx"]
        self.accepted_len = self.tree.extra["accepted_len"]
        self.bonus = self.tree.extra["bonus"]

    def draft(self, base_logits, head_emb, head_out, root_token, stream=None):
        pctree_draft(self.cfg, base_logits, head_emb, head_out, root_token,
                     self.tree, self.workspace, stream)
        return self.tree

    def accept(self, target_tokens, stream=None):
        pctree_accept(self.cfg, self.tree, target_tokens, self.accepted_idx,
                      self.accepted_len, self.bonus, stream)
        return self.accepted_idx, self.accepted_len, self.bonus

    def check_status(self) -> None:
        code = int(self.tree.status.item())
        if code != PCTREE_OK:
            raise PctreeError(code, "device status")

    def draft_from_host(self, base_logits_host: torch.Tensor,
                        root_host: torch.Tensor, head_emb, head_out,
                        stream=None):
        """End-to-end call a serving loop makes: pinned host inputs in, packed
        tree back on the host.  The kernels read the base logits and root
        tokens from the pinned host buffers as they need them (no copy); the
        outputs come back with one copy of the tree's buffer.  Returns the
        host tree arrays."""
        s = stream if stream is not None else torch.cuda.current_stream()
        blob = torch.empty(self.tree.blob.shape, dtype=torch.uint8, pin_memory=True)
        with torch.cuda.stream(s):
            self.draft(base_logits_host, head_emb, head_out, root_host, s)
            blob.copy_(self.tree.blob, non_blocking=True)
        s.synchronize()
        names = ("n_nodes", "tokens", "parent", "depth", "logp", "position_ids",
                 "mask", "retrieve", "n_leaves", "status")
        base = self.tree.blob.data_ptr()
        host = {}
        for name in names:
            t = getattr(self.tree, name)
            o = t.data_ptr() - base
            n = t.numel() * t.element_size()
            host[name] = blob[o:o + n].view(t.dtype).view(t.shape).numpy()
        return host


def pctree_debug_stall_stage(stage: int, wait_limit_ns: int = 1_000_000_000) -> None:
    """Failure-detection test hook (see include/pctree.h)."""
    rc = LIB.pctree_debug_stall_stage(stage, wait_limit_ns)
    if rc != PCTREE_OK:
        raise PctreeError(rc, "pctree_debug_stall_stage")
