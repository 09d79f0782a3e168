"""Thin Python binding of libchimera.so (argument marshalling only).

Every step of the Chimera draft-and-verify path runs in the library's sm_103a
kernels; this module only fills the C structs, passes device pointers (taken from
torch tensors) and host buffers, and maps status codes to exceptions.  It fails
loudly when the library is missing: there is no fallback implementation.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libchimera.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "chimera.h")

STATUS = {0: "OK", -1: "EINVAL", -2: "ENOMEM", -3: "ECAPACITY", -4: "ECUDA", -5: "ETIMEDOUT", -6: "ESTATE"}

DBG = dict(node_tokens=1, verify_logits=2, verify_hidden=3, argmax=4, path=5, accept_len=6,
           draft_logits=7, topk=8, hfull=9, n=10, tokens=11, prefill_logits=12, trigram_hits=13, htri=14)
KIND = {1: "linear", 2: "attention", 3: "norm", 4: "rope_kv", 5: "swiglu", 6: "embed", 7: "topk",
        8: "argmax", 9: "tree", 10: "accept", 11: "compact", 12: "other", 13: "chain"}
PHASE = {0: "draft", 1: "verify", 2: "commit"}


class ChimeraError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int), ("d_model", ctypes.c_int), ("n_heads", ctypes.c_int),
                ("head_dim", ctypes.c_int), ("ffn_dim", ctypes.c_int), ("vocab", ctypes.c_int),
                ("dtype", ctypes.c_int), ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("n_draft_heads", ctypes.c_int), ("tree_nodes", ctypes.c_int),
                ("topk", ctypes.c_int * 8), ("max_batch", ctypes.c_int), ("max_seq_len", ctypes.c_int),
                ("kv_block", ctypes.c_int), ("precision", ctypes.c_int), ("draft_mode", ctypes.c_int),
                ("accept_mode", ctypes.c_int), ("typical_eps", ctypes.c_float), ("typical_delta", ctypes.c_float),
                ("trigram_cache", ctypes.c_int), ("fused_chain", ctypes.c_int)]


class BlockWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate", "w_up", "w_down")]


class Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("layers", ctypes.POINTER(BlockWeights)),
                ("final_norm", ctypes.c_void_p), ("lm_head", ctypes.c_void_p),
                ("tri_w1", ctypes.c_void_p), ("tri_w2", ctypes.c_void_p), ("draft", BlockWeights),
                ("heads", ctypes.POINTER(ctypes.c_void_p))]


_lib = None

_SIGS = {
    "chimera_init": (ctypes.c_int, [ctypes.POINTER(Config), ctypes.POINTER(Weights), ctypes.c_void_p,
                                    ctypes.POINTER(ctypes.c_void_p)]),
    "chimera_prefill": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_step": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_generate": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_step_async": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int]),
    "chimera_sync": (ctypes.c_int, [ctypes.c_void_p]),
    "chimera_ar_generate": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_free": (None, [ctypes.c_void_p]),
    "chimera_last_error": (ctypes.c_char_p, [ctypes.c_void_p]),
    "chimera_tree": (ctypes.c_int, [ctypes.c_void_p] + [ctypes.c_void_p] * 4),
    "chimera_static_tree": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_int] + [ctypes.c_void_p] * 4),
    "chimera_profile_step": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int] + [ctypes.c_void_p] * 5),
    "chimera_profile_phases": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int] + [ctypes.c_void_p] * 3),
    "chimera_profile_kind": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_int] + [ctypes.c_void_p] * 3),
    "chimera_debug_override_tree": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_debug_set_root": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_debug_read": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t]),
    "chimera_debug_read_kv": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                                             ctypes.c_int, ctypes.c_void_p, ctypes.c_void_p]),
    "chimera_op_linear": (ctypes.c_int, [ctypes.c_int] * 6 + [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                                              ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                                              ctypes.c_void_p]),
    "chimera_op_linear_noalloc": (ctypes.c_int, [ctypes.c_int] * 5 + [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                                                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                                                      ctypes.c_void_p]),
    "chimera_op_sync": (ctypes.c_int, [ctypes.c_void_p]),
    "chimera_debug_set_wait_limit": (ctypes.c_int, [ctypes.c_uint64]),
    "chimera_op_attention": (ctypes.c_int, [ctypes.c_int] * 8 + [ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                                                 ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p,
                                                                 ctypes.c_int,
                                                                 ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                                                 ctypes.c_void_p, ctypes.c_int, ctypes.c_int,
                                                                 ctypes.c_void_p]),
}


def load(path: str = LIB_PATH):
    """Load the library (built by build.py / __graft_entry__.build); raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with paper_2402_15758_gb300.build.build() "
                           "(there is no CPU fallback)")
    lib = ctypes.CDLL(path)
    for name, (res, args) in _SIGS.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _ptr(t) -> int:
    return 0 if t is None else int(t.data_ptr())


def _stream_handle(stream) -> int:
    if stream is None:
        return 0
    return int(stream.cuda_stream)


def make_config(cfg: dict, max_batch: int | None = None, max_seq_len: int | None = None,
                precision: int | None = None) -> Config:
    c = Config()
    c.n_layers, c.d_model, c.n_heads = cfg["n_layers"], cfg["d_model"], cfg["n_heads"]
    c.head_dim, c.ffn_dim, c.vocab = cfg["head_dim"], cfg["ffn_dim"], cfg["vocab"]
    c.dtype = 0 if cfg["dtype"] == "fp32" else 1
    c.rms_eps, c.rope_theta = cfg["rms_eps"], cfg["rope_theta"]
    c.n_draft_heads, c.tree_nodes = cfg["n_draft_heads"], cfg["tree_nodes"]
    for i, k in enumerate(cfg["topk"]):
        c.topk[i] = k
    c.max_batch = max_batch or cfg["batch"]
    c.max_seq_len = max_seq_len or cfg.get("max_seq_len", 4096)
    c.kv_block = 16
    c.precision = cfg.get("precision", 1) if precision is None else precision
    c.draft_mode = cfg.get("draft_mode", 0)
    c.accept_mode = cfg.get("accept_mode", 0)
    c.typical_eps = cfg.get("typical_eps", 0.09)
    c.typical_delta = cfg.get("typical_delta", 0.3)
    c.trigram_cache = cfg.get("trigram_cache", 0)
    c.fused_chain = cfg.get("fused_chain", 0)
    return c


class Chimera:
    """One context: the weights (device tensors, kept alive here), KV caches and the
    captured step graph live in the library."""

    def __init__(self, cfg: dict, weights: dict, max_batch: int | None = None,
                 max_seq_len: int | None = None, stream=None, precision: int | None = None):
        self.lib = load()
        self.cfg = cfg
        self._w = weights
        self.c = make_config(cfg, max_batch, max_seq_len, precision)
        self.kv_f32 = cfg["dtype"] == "fp32" or self.c.precision == 1
        L, K = cfg["n_layers"], cfg["n_draft_heads"]

        def block(prefix):
            b = BlockWeights()
            for f in ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate", "w_up", "w_down"):
                setattr(b, f, _ptr(weights[f"{prefix}.{f}"]))
            return b

        self._layers = (BlockWeights * L)(*[block(f"layers.{i}") for i in range(L)])
        self._heads = (ctypes.c_void_p * K)(*[_ptr(weights[f"heads.{k}"]) for k in range(K)])
        w = Weights()
        w.embed = _ptr(weights["embed"])
        w.layers = self._layers
        w.final_norm, w.lm_head = _ptr(weights["final_norm"]), _ptr(weights["lm_head"])
        w.tri_w1, w.tri_w2 = _ptr(weights["tri_w1"]), _ptr(weights["tri_w2"])
        w.draft = block("draft")
        w.heads = self._heads
        self._wstruct = w
        h = ctypes.c_void_p()
        st = self.lib.chimera_init(ctypes.byref(self.c), ctypes.byref(w), _stream_handle(stream), ctypes.byref(h))
        if st != 0:
            raise ChimeraError(st, "chimera_init failed (check shapes / weights)")
        self.h = h
        self.batch = 0
        d = np.zeros(cfg["tree_nodes"], np.int32)
        p, r = np.zeros_like(d), np.zeros_like(d)
        a = np.zeros(cfg["tree_nodes"], np.uint64)
        self._check(self.lib.chimera_tree(self.h, d.ctypes.data, p.ctypes.data, r.ctypes.data, a.ctypes.data))
        self.tree = dict(depth=d.tolist(), parent=p.tolist(), rank=r.tolist(), anc=[int(x) for x in a])
        self.depth = max(self.tree["depth"])

    # ---- helpers ----
    def _check(self, st: int):
        if st != 0:
            raise ChimeraError(st, self.lib.chimera_last_error(self.h).decode())

    def close(self):
        if getattr(self, "h", None):
            self.lib.chimera_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # ---- the ABI ----
    def prefill(self, prompts: list[list[int]]):
        flat = np.ascontiguousarray(np.concatenate([np.asarray(p, np.int32) for p in prompts]))
        lens = np.asarray([len(p) for p in prompts], np.int32)
        self._check(self.lib.chimera_prefill(self.h, len(prompts), flat.ctypes.data, lens.ctypes.data))
        self.batch = len(prompts)

    def step(self):
        """One step; returns a list (per sequence) of emitted tokens."""
        D1 = self.depth + 1
        out = np.zeros((self.batch, D1), np.int32)
        cnt = np.zeros(self.batch, np.int32)
        self._check(self.lib.chimera_step(self.h, out.ctypes.data, cnt.ctypes.data))
        return [out[b, : cnt[b]].tolist() for b in range(self.batch)]

    def generate(self, n_steps: int):
        D1 = self.depth + 1
        out = np.zeros((self.batch, n_steps * D1), np.int32)
        cnt = np.zeros(self.batch, np.int32)
        self._check(self.lib.chimera_generate(self.h, n_steps, out.ctypes.data, cnt.ctypes.data))
        return [out[b, : cnt[b]].tolist() for b in range(self.batch)]

    def ar_generate(self, n_steps: int):
        """n_steps plain autoregressive steps; per sequence the n_steps emitted tokens."""
        out = np.zeros((self.batch, n_steps), np.int32)
        cnt = np.zeros(self.batch, np.int32)
        self._check(self.lib.chimera_ar_generate(self.h, n_steps, out.ctypes.data, cnt.ctypes.data))
        return [out[b, : cnt[b]].tolist() for b in range(self.batch)]

    def ar_step_async(self, n_steps: int = 1):
        self._check(self.lib.chimera_ar_generate(self.h, n_steps, None, None))

    def step_async(self, n_steps: int = 1):
        self._check(self.lib.chimera_step_async(self.h, n_steps))

    def sync(self):
        self._check(self.lib.chimera_sync(self.h))

    def profile_step(self, max_launches: int = 8192):
        kinds = np.zeros(max_launches, np.int32)
        phases = np.zeros(max_launches, np.int32)
        ms = np.zeros(max_launches, np.float32)
        by = np.zeros(max_launches, np.float64)
        cnt = ctypes.c_int32(0)
        self._check(self.lib.chimera_profile_step(self.h, max_launches, kinds.ctypes.data, phases.ctypes.data,
                                                  ms.ctypes.data, by.ctypes.data, ctypes.byref(cnt)))
        n = min(cnt.value, max_launches)
        return [dict(kind=KIND[int(kinds[i])], phase=PHASE[int(phases[i])], ms=float(ms[i]), bytes=float(by[i]))
                for i in range(n)]

    def profile_phases(self, n_steps: int):
        """Per-step (draft, verify, commit) ms of n_steps phase-timed graph replays."""
        d = np.zeros(n_steps, np.float32)
        v = np.zeros(n_steps, np.float32)
        c = np.zeros(n_steps, np.float32)
        self._check(self.lib.chimera_profile_phases(self.h, n_steps, d.ctypes.data, v.ctypes.data, c.ctypes.data))
        return d.tolist(), v.tolist(), c.tolist()

    def profile_kind(self, kind: str, n_reps: int):
        """Mean ms of one replay of a graph holding only one kernel class's launches of
        the step, with its launch count and algorithmic bytes."""
        code = {v: k for k, v in KIND.items()}[kind]
        ms = ctypes.c_float(0)
        n = ctypes.c_int32(0)
        by = ctypes.c_double(0)
        self._check(self.lib.chimera_profile_kind(self.h, code, n_reps, ctypes.byref(ms), ctypes.byref(n),
                                                  ctypes.byref(by)))
        return dict(ms=ms.value, launches=n.value, bytes=by.value)

    # ---- test hooks ----
    def override_tree(self, node_tokens):
        a = np.ascontiguousarray(np.asarray(node_tokens, np.int32).reshape(self.batch, -1))
        self._check(self.lib.chimera_debug_override_tree(self.h, a.ctypes.data))

    def set_root(self, roots):
        a = np.ascontiguousarray(np.asarray(roots, np.int32))
        self._check(self.lib.chimera_debug_set_root(self.h, a.ctypes.data))

    def read(self, what: str):
        """Copy a debug buffer to the host (numpy; bf16 buffers come back as float32)."""
        import torch
        cfg, B = self.cfg, max(self.batch, 1)
        N, V, d, K = cfg["tree_nodes"], cfg["vocab"], cfg["d_model"], cfg["n_draft_heads"]
        kmax = max(cfg["topk"])
        fdt = torch.float32 if cfg["dtype"] == "fp32" else torch.bfloat16
        shapes = dict(node_tokens=((B, N), torch.int32), verify_logits=((B, N, V), torch.float32),
                      verify_hidden=((B, N, d), torch.float32), argmax=((B, N), torch.int32),
                      path=((B, self.depth + 1), torch.int32), accept_len=((B,), torch.int32),
                      draft_logits=((K, B, V), torch.float32), topk=((B, K, kmax), torch.int32),
                      hfull=((K, B, d), torch.float32), n=((B,), torch.int32),
                      tokens=((B, self.c.max_seq_len + 1), torch.int32),
                      prefill_logits=((B, V), torch.float32), trigram_hits=((K, B), torch.int32),
                      htri=((K, B, d), torch.float32))
        shape, dt = shapes[what]
        t = torch.empty(shape, dtype=dt)
        self._check(self.lib.chimera_debug_read(self.h, DBG[what], t.data_ptr(), t.numel() * t.element_size()))
        return (t.float() if dt == torch.bfloat16 else t).numpy()

    def read_kv(self, layer: int, seq: int, pos0: int, count: int):
        import torch
        cfg = self.cfg
        dt = torch.float32 if self.kv_f32 else torch.bfloat16
        k = torch.empty((count, cfg["n_heads"], cfg["head_dim"]), dtype=dt)
        v = torch.empty_like(k)
        self._check(self.lib.chimera_debug_read_kv(self.h, layer, seq, pos0, count, k.data_ptr(), v.data_ptr()))
        return k.float().numpy(), v.float().numpy()


# ---- kernel-level entry points ----
def static_tree(topk, n_nodes: int) -> dict:
    """The static tree the library builds for these head limits and node count (host
    only, needs no GPU): depth, parent, rank and ancestor masks per node."""
    lib = load()
    tk = np.asarray(topk, np.int32)
    d = np.zeros(n_nodes, np.int32)
    p, r = np.zeros_like(d), np.zeros_like(d)
    a = np.zeros(n_nodes, np.uint64)
    st = lib.chimera_static_tree(tk.ctypes.data, len(tk), n_nodes, d.ctypes.data, p.ctypes.data,
                                 r.ctypes.data, a.ctypes.data)
    if st != 0:
        raise ChimeraError(st, "chimera_static_tree: limits or node count out of range")
    return dict(depth=d.tolist(), parent=p.tolist(), rank=r.tolist(), anc=[int(x) for x in a])


def op_linear(X, W, Y, epi: int = 0, out_f32: bool = False, X_lo=None, stream=None):
    """Y (epilogue)= (X + X_lo) W^T through chimera_op_linear (X, X_lo [M][K], W [N][K],
    Y [M][N] device tensors)."""
    lib = load()
    M, K = X.shape
    N = W.shape[0]
    dtype = 0 if X.element_size() == 4 else 1
    st = lib.chimera_op_linear(dtype, epi, int(out_f32), M, N, K, _ptr(X), _ptr(X_lo), X.stride(0), _ptr(W),
                               _ptr(Y), Y.stride(0), _stream_handle(stream))
    if st != 0:
        raise ChimeraError(st, "chimera_op_linear")


def op_linear_noalloc(X, W, Y, epi: int = 0, out_f32: bool = False, X_lo=None, stream=None):
    """Y (epilogue)= (X + X_lo) W^T through chimera_op_linear_noalloc (bf16 X, W; the
    library keeps the scratch in static device arrays, so the call allocates nothing)."""
    lib = load()
    M, K = X.shape
    N = W.shape[0]
    st = lib.chimera_op_linear_noalloc(epi, int(out_f32), M, N, K, _ptr(X), _ptr(X_lo), X.stride(0), _ptr(W),
                                       _ptr(Y), Y.stride(0), _stream_handle(stream))
    if st != 0:
        raise ChimeraError(st, "chimera_op_linear_noalloc")


def op_attention(q, pool, page_table, n_ctx, anc, out, nq, q_local0, n_local, q_rows, n_heads, head_dim,
                 splits=1, out_lo=None, stream=None):
    """Tree-masked paged attention through chimera_op_attention.  q fp32; pool
    [blocks][H][planes][16][hd]: fp32 K, V planes (fp32 model, out fp32) or bf16 planes
    (bf16 model, out bf16 + optional lo half): 2 planes K, V or 4 planes K_hi, K_lo,
    V_hi, V_lo."""
    lib = load()
    dtype = 0 if out.element_size() == 4 else 1
    kv_split = int(pool.shape[2] == 4)
    st = lib.chimera_op_attention(dtype, kv_split, n_ctx.shape[0], n_heads, head_dim, nq, q_local0, n_local,
                                  _ptr(q), q.stride(0), q_rows, _ptr(pool), pool.shape[0], _ptr(page_table),
                                  page_table.shape[1],
                                  _ptr(n_ctx), _ptr(anc), _ptr(out), _ptr(out_lo), out.stride(0), splits,
                                  _stream_handle(stream))
    if st != 0:
        raise ChimeraError(st, "chimera_op_attention")


def op_sync(stream=None):
    """Wait for the stateless entry points' work and raise what their kernels flagged
    on the device since the last call (ETIMEDOUT, EINVAL, ...)."""
    st = load().chimera_op_sync(_stream_handle(stream))
    if st != 0:
        raise ChimeraError(st, "chimera_op_sync: the device flagged an error")


def set_wait_limit(ns: int = 0):
    """Test hook: bounded-wait limit of the stateless linear entry points (0: default)."""
    load().chimera_debug_set_wait_limit(int(ns))


def declared_symbols(header: str = HEADER) -> list[str]:
    """Function names declared in include/chimera.h."""
    import re
    src = open(header).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(chimera_[a-z_]+)\s*\(", src)))
