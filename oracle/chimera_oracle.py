"""fp64 CPU oracle of one Chimera draft-and-verify step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or link
this package; only tests/, the smoke check and the benchmark's CPU baseline use it.
It shares no code with the CUDA path: it gets the same stored weights (bf16 or
fp32, up-cast exactly to float64) and the same token ids, nothing else.

What it computes (paper = Chimera, arXiv 2402.15758):
  * base LLM: a Llama-style decoder (Table 1 shapes), greedy next token (eq. 1);
  * trigram encoder (eq. "trigram_calculations"): h_tri = W2 SiLU(W1 [x_{i-2};x_{i-1};x_i]);
  * full-context encoder (eq. "fullcontext_calculations"): one Transformer block over
    [H_LLM ; H_tri], keeping the trigram rows;
  * residual decoding heads (eq. "residual decoding head"): head k scores
    Theta_k [h_LLM_n ; h_full_{n+1+k}] and predicts word n+2+k;
  * tree-structured verification (Section "Verification", Medusa-style) and
    greedy acceptance of the longest matching path;
  * the state update that commits the accepted tokens (their KV entries).

Readings where the paper is silent (each one value):
  R1 RMSNorm eps 1e-6, no biases;  R2 Llama rotate-half RoPE, theta 1e4, 0-based
  positions;  R3 missing leading embeddings of the first trigrams are zeros;
  R4 each "MLP" of the trigram encoder is one bias-free linear;  R5 the draft runs
  K sequential sub-steps, sub-step k adding the trigram that ends at the (k)th
  drafted token, head k reading the newest full-context row;  R6 the full-context
  block is one Llama block, keys = all H_LLM rows plus trigram rows up to the
  query (causal over the concatenation), no final norm;  R7 Theta_k has shape
  2d x |V| (the concatenated input), softmax skipped (monotone);  R8 K = 4;
  R9 static tree (oracle/tree.py);  R10 node at depth j sits at position n+j and
  attends the committed prefix plus its ancestors-or-self;  R11 h_LLM is the
  post-final-norm hidden state;  R12 ties: larger value first, then smaller
  token id;  R13 the root is the base model's own next token, a step emits the
  root plus the accepted drafted tokens, and the bonus token becomes the next root.

Positions are 0-based: the paper's word i sits at position i-1.  State after a
step: tokens x[0..n] where x[n] is the root (not yet in the KV cache), base KV and
H_LLM rows for positions 0..n-1, draft-layer KV for positions 0..n-1.
"""
from __future__ import annotations

import numpy as np

try:  # weights may arrive as torch tensors (bf16 has no numpy dtype)
    import torch
except Exception:  # pragma: no cover
    torch = None


# ----------------------------------------------------------------------------
# weights
# ----------------------------------------------------------------------------
class OracleWeights:
    """Exact float64 view of the stored weights.

    `cache=True` keeps every up-cast matrix (small configs); otherwise each access
    up-casts again, so a 7B model never needs all its weights in float64 at once.
    """

    def __init__(self, weights: dict, cache: bool = True):
        self._src = weights
        self._cache = {} if cache else None

    def __call__(self, name: str) -> np.ndarray:
        if self._cache is not None and name in self._cache:
            return self._cache[name]
        t = self._src[name]
        if torch is not None and isinstance(t, torch.Tensor):
            a = t.detach().to("cpu").to(torch.float64).numpy()
        else:
            a = np.asarray(t, dtype=np.float64)
        if self._cache is not None:
            self._cache[name] = a
        return a

    def subset(self, prefix: str) -> "OracleWeights":
        """A caching view of the matrices whose names start with `prefix` (one layer):
        each is up-cast once while the view lives (the prompt chunks of a layer)."""
        return OracleWeights({k: v for k, v in self._src.items() if k.startswith(prefix)}, cache=True)

    def rows(self, name: str, idx) -> np.ndarray:
        """Selected rows of a matrix (the embedding gather), up-cast exactly."""
        t = self._src[name]
        if torch is not None and isinstance(t, torch.Tensor):
            sel = t[torch.as_tensor(np.asarray(idx, dtype=np.int64), device=t.device)]
            return sel.detach().to("cpu").to(torch.float64).numpy()
        return np.asarray(t, dtype=np.float64)[np.asarray(idx)]


# ----------------------------------------------------------------------------
# layer math
# ----------------------------------------------------------------------------
def rmsnorm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm (Llama; reading R1): x / sqrt(mean(x^2) + eps) * g, row-wise."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * g


def silu(x: np.ndarray) -> np.ndarray:
    """SiLU(x) = x * sigmoid(x) (eq. trigram_calculations, SwiGLU)."""
    return x / (1.0 + np.exp(-x))


def rope_angles(pos: np.ndarray, head_dim: int, theta: float) -> np.ndarray:
    """Angles pos * theta^(-2i/hd), i < hd/2 (reading R2)."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    inv = theta ** (-2.0 * i / head_dim)
    return np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate-half RoPE on x[R][H][hd]: pairs (i, i + hd/2) rotated by angle(pos, i)."""
    hd = x.shape[-1]
    half = hd // 2
    a = rope_angles(pos, hd, theta)[:, None, :]  # [R][1][half]
    c, s = np.cos(a), np.sin(a)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def attend(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """Softmax attention of one query row: q[H][hd], k/v[m][H][hd] -> [H][hd]."""
    hd = q.shape[-1]
    s = np.einsum("hd,mhd->hm", q, k) / np.sqrt(hd)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    return np.einsum("hm,mhd->hd", p, v)


def topk_desc(z: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k largest entries, larger value first, then smaller id (R12)."""
    order = np.lexsort((np.arange(z.shape[0]), -z))
    return order[:k]


def argmax_desc(z: np.ndarray) -> int:
    return int(topk_desc(z, 1)[0])


def top2_margin(z: np.ndarray) -> float:
    """(v1 - v2) / max|z| of a score row (near-tie measure)."""
    o = topk_desc(z, 2)
    return float((z[o[0]] - z[o[1]]) / np.max(np.abs(z)))


# ----------------------------------------------------------------------------
# one Llama block over a set of rows with explicit visibility
# ----------------------------------------------------------------------------
def block_rows(W: OracleWeights, prefix: str, cfg: dict, x: np.ndarray, pos: np.ndarray,
               ctx_k: np.ndarray, ctx_v: np.ndarray, local_mask: np.ndarray):
    """Llama block on rows x[R][d] at positions pos[R].

    Every row sees all context keys ctx_k/ctx_v[m][H][hd] (already rotated) and the
    local rows j with local_mask[i][j].  Returns (out[R][d], k_local, v_local) where
    k_local is rotated.

    The attention of row i is the softmax over its visible keys (all m context keys,
    then the visible local rows), written as one score row per (head, query) over the
    union [context ; local] with the invisible local keys at -inf.  The key rows are
    never copied, so a context of many thousand rows costs one score matrix per call.
    """
    H, hd, eps, th = cfg["n_heads"], cfg["head_dim"], cfg["rms_eps"], cfg["rope_theta"]
    R, d = x.shape
    h = rmsnorm(x, W(f"{prefix}.attn_norm"), eps)
    qkv = h @ W(f"{prefix}.wqkv").T
    q = rope(qkv[:, :d].reshape(R, H, hd), pos, th)
    k = rope(qkv[:, d:2 * d].reshape(R, H, hd), pos, th)
    v = qkv[:, 2 * d:].reshape(R, H, hd)
    qh = q.transpose(1, 0, 2)                                   # [H][R][hd]
    s_ctx = qh @ ctx_k.transpose(1, 2, 0)                      # [H][R][m]
    s_loc = qh @ k.transpose(1, 2, 0)                          # [H][R][R]
    s_loc = np.where(np.asarray(local_mask, dtype=bool)[None], s_loc, -np.inf)
    s = np.concatenate([s_ctx, s_loc], axis=-1) / np.sqrt(hd)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p = p / p.sum(axis=-1, keepdims=True)
    m = ctx_k.shape[0]
    att = p[..., :m] @ ctx_v.transpose(1, 0, 2) + p[..., m:] @ v.transpose(1, 0, 2)  # [H][R][hd]
    att = att.transpose(1, 0, 2)
    x = x + att.reshape(R, d) @ W(f"{prefix}.wo").T
    h2 = rmsnorm(x, W(f"{prefix}.ffn_norm"), eps)
    ffn = silu(h2 @ W(f"{prefix}.w_gate").T) * (h2 @ W(f"{prefix}.w_up").T)
    x = x + ffn @ W(f"{prefix}.w_down").T
    return x, k, v


def causal_block_dense(W: OracleWeights, prefix: str, cfg: dict, x: np.ndarray) -> np.ndarray:
    """The same Llama block over a whole sequence (positions 0..R-1), written with a
    dense causal score matrix instead of per-row key lists.  Used as brute force."""
    H, hd, eps, th = cfg["n_heads"], cfg["head_dim"], cfg["rms_eps"], cfg["rope_theta"]
    R, d = x.shape
    pos = np.arange(R)
    h = rmsnorm(x, W(f"{prefix}.attn_norm"), eps)
    qkv = h @ W(f"{prefix}.wqkv").T
    q = rope(qkv[:, :d].reshape(R, H, hd), pos, th)
    k = rope(qkv[:, d:2 * d].reshape(R, H, hd), pos, th)
    v = qkv[:, 2 * d:].reshape(R, H, hd)
    s = np.einsum("ihd,jhd->hij", q, k) / np.sqrt(hd)
    s = np.where(np.tril(np.ones((R, R), dtype=bool))[None], s, -np.inf)
    s = s - s.max(axis=-1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(axis=-1, keepdims=True)
    att = np.einsum("hij,jhd->ihd", p, v).reshape(R, d)
    x = x + att @ W(f"{prefix}.wo").T
    h2 = rmsnorm(x, W(f"{prefix}.ffn_norm"), eps)
    x = x + (silu(h2 @ W(f"{prefix}.w_gate").T) * (h2 @ W(f"{prefix}.w_up").T)) @ W(f"{prefix}.w_down").T
    return x


# ----------------------------------------------------------------------------
# base model
# ----------------------------------------------------------------------------
def causal_forward(W: OracleWeights, cfg: dict, tokens: list[int]):
    """From-scratch causal forward over a whole token sequence (eq. 1 context).

    Returns (H_LLM[R][d] post final norm, logits[R][V])."""
    x = W.rows("embed", tokens)
    for l in range(cfg["n_layers"]):
        x = causal_block_dense(W, f"layers.{l}", cfg, x)
    hs = rmsnorm(x, W("final_norm"), cfg["rms_eps"])
    return hs, hs @ W("lm_head").T


def ar_generate(W: OracleWeights, cfg: dict, prompt: list[int], n_new: int) -> list[int]:
    """Plain greedy autoregressive decoding (eq. 1 with argmax): the stream that
    lossless speculative decoding must reproduce.  Recomputes from scratch."""
    toks = list(prompt)
    out = []
    for _ in range(n_new):
        _, logits = causal_forward(W, cfg, toks)
        t = argmax_desc(logits[-1])
        out.append(t)
        toks.append(t)
    return out


class SeqState:
    """Committed state of one sequence (see module docstring)."""

    def __init__(self, cfg: dict, cap: int):
        L, H, hd, d = cfg["n_layers"], cfg["n_heads"], cfg["head_dim"], cfg["d_model"]
        self.tokens: list[int] = []
        self.n = 0
        self.K = np.zeros((L, cap, H, hd))
        self.V = np.zeros((L, cap, H, hd))
        self.Hs = np.zeros((cap, d))
        self.dK = np.zeros((cap, H, hd))
        self.dV = np.zeros((cap, H, hd))


def draft_kv_rows(W: OracleWeights, cfg: dict, hs: np.ndarray, pos: np.ndarray):
    """Draft-layer keys/values of H_LLM rows (the H_LLM part of the full-context
    encoder input, eq. fullcontext_calculations): RoPE(Wk n1(h)), Wv n1(h)."""
    H, hd, d = cfg["n_heads"], cfg["head_dim"], cfg["d_model"]
    h = rmsnorm(hs, W("draft.attn_norm"), cfg["rms_eps"])
    wqkv = W("draft.wqkv")
    k = (h @ wqkv[d:2 * d].T).reshape(-1, H, hd)
    v = (h @ wqkv[2 * d:].T).reshape(-1, H, hd)
    return rope(k, pos, cfg["rope_theta"]), v


def prefill(W: OracleWeights, cfg: dict, prompt: list[int], cap: int, chunk: int | None = None) -> SeqState:
    """Causal forward over the prompt; fills base KV, H_LLM and draft KV; the root is
    the greedy next token (eq. 1).

    With `chunk`, each layer takes the prompt `chunk` rows at a time: the rows of a
    chunk attend the keys of all earlier rows of that layer (already computed) plus
    the causal part of their own chunk, which is the same causal attention as one
    pass over the whole prompt (every row's softmax still runs over positions
    0..itself); only the score matrices get smaller, so long prompts fit in memory."""
    R = len(prompt)
    st = SeqState(cfg, cap)
    x = W.rows("embed", prompt)
    pos = np.arange(R)
    C = R if not chunk else int(chunk)
    for l in range(cfg["n_layers"]):
        Wl = W.subset(f"layers.{l}.") if C < R else W
        xs = []
        for a in range(0, R, C):
            b = min(R, a + C)
            causal = np.tril(np.ones((b - a, b - a), dtype=bool))
            xo, k, v = block_rows(Wl, f"layers.{l}", cfg, x[a:b], pos[a:b], st.K[l, :a], st.V[l, :a], causal)
            st.K[l, a:b], st.V[l, a:b] = k, v
            xs.append(xo)
        x = np.concatenate(xs, axis=0)
    hs = rmsnorm(x, W("final_norm"), cfg["rms_eps"])
    st.Hs[:R] = hs
    st.dK[:R], st.dV[:R] = draft_kv_rows(W, cfg, hs, pos)
    logits = hs[-1] @ W("lm_head").T
    st.n = R
    st.tokens = list(prompt) + [argmax_desc(logits)]
    st.prefill_logits = logits
    return st


# ----------------------------------------------------------------------------
# draft model (lightweight draft: trigram encoder, full-context encoder, heads)
# ----------------------------------------------------------------------------
def trigram_input(W: OracleWeights, cfg: dict, ids: list[int]) -> np.ndarray:
    """t = [x_{i-2}; x_{i-1}; x_i]; a missing leading token (id < 0) is a zero
    block (reading R3 of the collapsed uni/bigram)."""
    d = cfg["d_model"]
    parts = []
    for t in ids:
        parts.append(np.zeros(d) if t < 0 else W.rows("embed", [t])[0])
    return np.concatenate(parts)


def trigram_encoder(W: OracleWeights, t: np.ndarray) -> np.ndarray:
    """eq. trigram_calculations with reading R4: W2 SiLU(W1 t)."""
    return W("tri_w2") @ silu(W("tri_w1") @ t)


def draft(W: OracleWeights, cfg: dict, st: SeqState, kmax: int) -> dict:
    """K sequential sub-steps (reading R5).  Sub-step k encodes the trigram ending at
    x[n+k] (x[n] = root, x[n+1+j] = head j's top-1), runs the full-context block on
    it at position n+k against the committed draft KV (0..n-1) plus the trigram rows
    of sub-steps 0..k, and scores head k on [H_LLM[n-1]; h_full].

    cfg["draft_mode"] selects the ablation variants of the draft (Section "Residual
    decoding heads" and its ablation):
      bit 0 (one pass): only sub-step 0 runs; every head k scores h_full_{n+1}
        (the alternative reading of eq. "residual decoding head" with one trigram row);
      bit 1 (no residual): head k scores h_full alone, Theta_k in R^{|V| x d}
        (the "w/o residual" variant of the ablation figure)."""
    n, K = st.n, cfg["n_draft_heads"]
    mode = cfg.get("draft_mode", 0)
    one_pass, no_resid = bool(mode & 1), bool(mode & 2)
    chain = [st.tokens[n]]
    tk, tv, top, logits, hfull, htri = [], [], [], [], [], []

    def tok(i):  # x[i] for i <= n+k
        if i < 0:
            return -1
        return st.tokens[i] if i <= n else chain[i - n]

    for k in range(K):
        if k == 0 or not one_pass:
            t = trigram_input(W, cfg, [tok(n - 2 + k), tok(n - 1 + k), tok(n + k)])
            g = trigram_encoder(W, t)
            htri.append(g)
            # incremental full-context block: new row at position n+k
            # the new row sees the committed draft KV, the earlier trigram rows (given
            # as context) and itself (its only local row).
            ctx_k = np.concatenate([st.dK[:n]] + [kk[None] for kk in tk], axis=0)
            ctx_v = np.concatenate([st.dV[:n]] + [vv[None] for vv in tv], axis=0)
            out, k_new, v_new = block_rows(W, "draft", cfg, g[None, :], np.array([n + k]),
                                           ctx_k, ctx_v, np.ones((1, 1), dtype=bool))
            tk.append(k_new[0])
            tv.append(v_new[0])
            h = out[0]
        hfull.append(h)
        head_in = h if no_resid else np.concatenate([st.Hs[n - 1], h])
        z = W(f"heads.{k}") @ head_in
        logits.append(z)
        idx = topk_desc(z, kmax)
        top.append(idx)
        chain.append(int(idx[0]))
    return dict(topk=np.array(top), logits=np.array(logits), hfull=np.array(hfull),
                htri=np.array(htri), chain=chain)


def draft_bruteforce(W: OracleWeights, cfg: dict, st: SeqState, chain: list[int]) -> np.ndarray:
    """From-scratch full-context encoder over the explicit [H_LLM ; H_tri] sequence
    (eq. fullcontext_calculations, causal over the concatenation, reading R6);
    returns the trigram-row outputs h_full for sub-steps 0..len(chain)-1."""
    n = st.n
    toks = st.tokens[: n] + list(chain)

    def tok(i):
        return toks[i] if i >= 0 else -1

    rows = [trigram_encoder(W, trigram_input(W, cfg, [tok(n - 2 + k), tok(n - 1 + k), tok(n + k)]))
            for k in range(len(chain))]
    seq = np.concatenate([st.Hs[:n], np.array(rows)], axis=0)
    out = causal_block_dense(W, "draft", cfg, seq)
    return out[n:]


# ----------------------------------------------------------------------------
# tree, verification, acceptance, commit
# ----------------------------------------------------------------------------
def tree_tokens(tree: dict, root: int, topk: np.ndarray) -> list[int]:
    """Node token = top-k[depth-1][rank]; the root is x[n] (Section "Inference")."""
    return [root] + [int(topk[tree["depth"][i] - 1][tree["rank"][i]]) for i in range(1, tree["n"])]


def verify(W: OracleWeights, cfg: dict, st: SeqState, tree: dict, node_tokens: list[int]) -> dict:
    """One base forward over every tree node (Section "Verification"): node i at
    position n+depth_i attends the committed prefix and its ancestors-or-self
    (reading R10).  Returns post-norm hidden rows, logits and the node K/V."""
    n, N = st.n, tree["n"]
    pos = n + np.array(tree["depth"])
    mask = np.array([[(tree["anc"][i] >> j) & 1 == 1 for j in range(N)] for i in range(N)])
    x = W.rows("embed", node_tokens)
    ks, vs = [], []
    for l in range(cfg["n_layers"]):
        x, k, v = block_rows(W, f"layers.{l}", cfg, x, pos, st.K[l, :n], st.V[l, :n], mask)
        ks.append(k)
        vs.append(v)
    hv = rmsnorm(x, W("final_norm"), cfg["rms_eps"])
    return dict(hidden=hv, logits=hv @ W("lm_head").T, k=np.array(ks), v=np.array(vs))


def accept(tree: dict, node_tokens: list[int], logits: np.ndarray):
    """Greedy acceptance (Section "Verification"): from the root, step to the child
    whose token equals the base argmax of the current node; stop when none does.
    Returns (path of node indices, bonus token = argmax of the last path node)."""
    cur, path = 0, [0]
    while True:
        p = argmax_desc(logits[cur])
        nxt = [c for c in tree["children"][cur] if node_tokens[c] == p]
        if not nxt:
            return path, p
        cur = nxt[0]
        path.append(cur)


def typical_threshold(z: np.ndarray, eps: float, delta: float) -> tuple[np.ndarray, float]:
    """Probabilities at temperature 1 of a score row and the typical-acceptance
    threshold min(eps, delta * exp(-H(p))), H the entropy in nats (the typical decoding
    of the verification step, Section "Verification"; criterion of the cited work)."""
    z = np.asarray(z, dtype=np.float64)
    e = np.exp(z - z.max())
    p = e / e.sum()
    nz = p > 0
    H = -float(np.sum(p[nz] * np.log(p[nz])))
    return p, min(eps, delta * np.exp(-H))


def accept_typical(tree: dict, node_tokens: list[int], logits: np.ndarray, eps: float, delta: float):
    """Typical acceptance (T = 1): a node is acceptable when its parent is and its token
    has probability above the parent's typical threshold under the base model's
    distribution at the parent.  The accepted path ends at the deepest acceptable node
    (ties: the smallest node index, i.e. the lexicographically first rank tuple); the
    bonus token is the base argmax there.  Returns (path, bonus)."""
    N = tree["n"]
    ok = [False] * N
    ok[0] = True
    probs = [typical_threshold(logits[i], eps, delta) for i in range(N)]
    for c in range(1, N):
        par = tree["parent"][c]
        p, thr = probs[par]
        ok[c] = ok[par] and p[node_tokens[c]] > thr
    best = 0
    for c in range(1, N):
        if ok[c] and tree["depth"][c] > tree["depth"][best]:
            best = c
    path, j = [], best
    while j >= 0:
        path.append(j)
        j = tree["parent"][j]
    return path[::-1], argmax_desc(logits[best])


def commit(W: OracleWeights, cfg: dict, st: SeqState, node_tokens: list[int], ver: dict,
           path: list[int], bonus: int) -> list[int]:
    """State update (reading R13): the path's tokens, base KV and H_LLM rows become
    positions n..n+L; their draft-layer K/V are appended; the bonus is the new root.
    Returns the emitted tokens (root + accepted drafted tokens)."""
    n, L = st.n, len(path) - 1
    for j, node in enumerate(path):
        st.K[:, n + j] = ver["k"][:, node]
        st.V[:, n + j] = ver["v"][:, node]
        st.Hs[n + j] = ver["hidden"][node]
    dk, dv = draft_kv_rows(W, cfg, st.Hs[n:n + L + 1], np.arange(n, n + L + 1))
    st.dK[n:n + L + 1], st.dV[n:n + L + 1] = dk, dv
    emitted = [node_tokens[node] for node in path]
    st.tokens = st.tokens[: n] + emitted + [bonus]
    st.n = n + L + 1
    return emitted


def step(W: OracleWeights, cfg: dict, st: SeqState, tree: dict, override=None) -> dict:
    """One draft-and-verify step.  `override` replaces the drafted node tokens
    (nodes 1..N-1) to force acceptance lengths in tests.  cfg["accept_mode"] = 1 takes
    the typical acceptance (thresholds cfg["typical_eps"], cfg["typical_delta"])
    instead of the greedy one."""
    kmax = max(cfg["topk"])
    dr = draft(W, cfg, st, kmax)
    toks = tree_tokens(tree, st.tokens[st.n], dr["topk"])
    if override is not None:
        toks = [toks[0]] + [int(t) for t in override[1:]]
    n_before = st.n
    ver = verify(W, cfg, st, tree, toks)
    if cfg.get("accept_mode", 0) == 1:
        path, bonus = accept_typical(tree, toks, ver["logits"], cfg["typical_eps"], cfg["typical_delta"])
    else:
        path, bonus = accept(tree, toks, ver["logits"])
    emitted = commit(W, cfg, st, toks, ver, path, bonus)
    return dict(draft=dr, node_tokens=toks, verify=ver, path=path, bonus=bonus,
                emitted=emitted, n_before=n_before)


def generate(W: OracleWeights, cfg: dict, prompt: list[int], n_new: int, tree: dict,
             override_fn=None) -> tuple[list[int], list[dict]]:
    """Speculative greedy generation: prefill, then steps until n_new tokens."""
    cap = len(prompt) + n_new + tree["n"] + 8
    st = prefill(W, cfg, prompt, cap)
    out, recs = [], []
    while len(out) < n_new:
        ov = override_fn(st) if override_fn else None
        rec = step(W, cfg, st, tree, ov)
        out += rec["emitted"]
        recs.append(rec)
    return out[:n_new], recs
