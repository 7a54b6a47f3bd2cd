"""Oracle transformer: a plain fp64 pre-norm decoder, the M_p / M_q of the paper.

TEST INFRASTRUCTURE. Only tests/, ``__graft_entry__.smoke()`` and bench.py's ``cpu_baseline``
and ``--impl reference`` legs may import this package. The product path never does.

The paper treats the target M_p and draft M_q as black-box next-token distributions
(Sec. 2.2, Sec. 3.2.1) and runs OPT/Bloomz/Qwen models (Sec. 4.2). The synthetic workloads use
Llama-style decoders instead; this file is the definition of those models:

    h_0 = E[token]
    per layer:  a = RMSNorm(h) * g_attn
                q, k, v = a Wq^T, a Wk^T, a Wv^T          (GQA: query head h -> kv head h // G)
                q, k = RoPE(q, pos), RoPE(k, pos)         (rotate-half pairing (i, i + hd/2))
                h += softmax(q k^T / sqrt(hd) + causal) v Wo^T
                a = RMSNorm(h) * g_ffn
                h += (silu(a Wg^T) * (a Wu^T)) Wd^T
    final:      h_f = RMSNorm(h) * g_final ; logits = h_f W_lm^T

Everything is float64. bf16 weights are widened from the same bf16 bits the GPU reads.
Multiple independent sequences can be pushed through one call (their rows share each matmul;
the attention of every sequence only sees its own cache), which is how Alg. 1's "run M_p in
parallel" and the k-beam batching are expressed.
"""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

import numpy as np


def widen(w: np.ndarray) -> np.ndarray:
    """float32, or uint16 bf16 bit patterns -> float64."""
    if w.dtype == np.uint16:
        return (w.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return np.asarray(w, dtype=np.float64)


def rms_norm(x: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """x / sqrt(mean(x^2) + eps) * g over the last axis."""
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * g


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary position embedding, rotate-half form.

    x: [n, heads, hd]; pos: [n]. Dimension i < hd/2 is paired with i + hd/2 and the pair is
    rotated by the angle pos * theta^(-2i/hd)."""
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = theta ** (-np.arange(half, dtype=np.float64) * 2.0 / hd)
    ang = pos.astype(np.float64)[:, None] * inv_freq[None, :]
    cos = np.cos(ang)[:, None, :]
    sin = np.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * cos - x2 * sin, x2 * cos + x1 * sin], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def softmax(s: np.ndarray, axis: int = -1) -> np.ndarray:
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def log_softmax(v: np.ndarray) -> np.ndarray:
    m = np.max(v, axis=-1, keepdims=True)
    return v - (m + np.log(np.sum(np.exp(v - m), axis=-1, keepdims=True)))


class KVCache:
    """Keys/values of one sequence, per layer, [T, n_kv_heads, head_dim] float64.

    ``fork()`` gives a child that sees the parent's first ``len(parent)`` positions (shared,
    not copied) and then its own rows: the k beams of a step all fork the prompt's prefix."""

    def __init__(self, n_layers: int, parent: "KVCache | None" = None):
        self.n_layers = n_layers
        self.parent = parent
        self.parent_len = len(parent) if parent is not None else 0
        self._k: List[List[np.ndarray]] = [[] for _ in range(n_layers)]
        self._v: List[List[np.ndarray]] = [[] for _ in range(n_layers)]
        self._own = [0] * n_layers

    def __len__(self) -> int:
        return self.parent_len + self._own[self.n_layers - 1]

    def own_len(self, layer: int) -> int:
        return self._own[layer]

    def append(self, layer: int, k: np.ndarray, v: np.ndarray) -> None:
        self._k[layer].append(k)
        self._v[layer].append(v)
        self._own[layer] += k.shape[0]

    def keys(self, layer: int) -> Tuple[np.ndarray, np.ndarray]:
        """(K, V) of all visible positions of ``layer``."""
        ks, vs = [], []
        if self.parent is not None:
            pk, pv = self.parent.keys(layer)
            ks.append(pk[: self.parent_len])
            vs.append(pv[: self.parent_len])
        ks += self._k[layer]
        vs += self._v[layer]
        return np.concatenate(ks, axis=0), np.concatenate(vs, axis=0)

    def fork(self) -> "KVCache":
        return KVCache(self.n_layers, parent=self)

    def truncated(self, length: int) -> "KVCache":
        """A standalone cache holding the first ``length`` positions."""
        out = KVCache(self.n_layers)
        for l in range(self.n_layers):
            k, v = self.keys(l)
            assert length <= k.shape[0]
            out.append(l, k[:length].copy(), v[:length].copy())
        return out


class Transformer:
    """One model (target or draft) with fp64 arithmetic.

    weights: name -> array (float32 or bf16 bits), names as in ``synth.ModelShape``.
    keep_widened: cache the float64 copies (fast, 4x the bf16 memory); otherwise each matrix
    is widened when used (for 7B-sized models)."""

    def __init__(self, shape, weights: Dict[str, np.ndarray], keep_widened: bool = True):
        self.shape = shape
        self.raw = weights
        self.keep = keep_widened
        self._wide: Dict[str, np.ndarray] = {}
        self.n_calls = 0  # forward calls, for the paper's calls-per-token counters (Sec. 4.3)

    def w(self, name: str) -> np.ndarray:
        if name in self._wide:
            return self._wide[name]
        x = widen(self.raw[name])
        if self.keep:
            self._wide[name] = x
        return x

    def new_cache(self) -> KVCache:
        return KVCache(self.shape.n_layers)

    def forward(self, seqs: Sequence[Tuple[KVCache, Sequence[int]]], last_only: bool = False):
        """Append each sequence's new tokens after its cache and run them through the model.

        seqs: list of (cache, tokens). Token i of a sequence sits at position len(cache) + i and
        attends to every cached position and to its own sequence's new tokens up to itself.
        Caches are extended in place. Returns (logits, hidden) lists, one [n_i, V] / [n_i, D]
        pair per sequence; ``hidden`` is the final-normed state that feeds the LM head. With
        ``last_only`` the LM head runs on each sequence's last row only ([1, V] / [1, D])."""
        S = self.shape
        H, KVH, hd = S.n_heads, S.n_kv_heads, S.head_dim
        G = H // KVH
        self.n_calls += 1
        counts = [len(t) for _, t in seqs]
        starts = [len(c) for c, _ in seqs]
        tokens = np.concatenate([np.asarray(t, dtype=np.int64) for _, t in seqs])
        pos = np.concatenate([np.arange(s, s + n) for s, n in zip(starts, counts)])
        offs = np.concatenate([[0], np.cumsum(counts)])
        N = tokens.shape[0]

        h = self.w("embed")[tokens]
        for l in range(S.n_layers):
            a = rms_norm(h, self.w(f"l{l}.attn_norm"), S.norm_eps)
            q = (a @ self.w(f"l{l}.wq").T).reshape(N, H, hd)
            k = (a @ self.w(f"l{l}.wk").T).reshape(N, KVH, hd)
            v = (a @ self.w(f"l{l}.wv").T).reshape(N, KVH, hd)
            q = rope(q, pos, S.rope_theta)
            k = rope(k, pos, S.rope_theta)
            att = np.empty((N, H, hd))
            for s, (cache, _) in enumerate(seqs):
                r0, r1 = offs[s], offs[s + 1]
                cache.append(l, k[r0:r1], v[r0:r1])
                K, Vv = cache.keys(l)
                K = np.repeat(K, G, axis=1)      # [T, H, hd]: query head h reads kv head h // G
                Vv = np.repeat(Vv, G, axis=1)
                T = K.shape[0]
                n = r1 - r0
                visible = starts[s] + np.arange(n)[:, None] + 1   # row i sees positions < visible
                mask = np.arange(T)[None, :] >= visible           # [n, T]
                qh = q[r0:r1].transpose(1, 0, 2)                  # [H, n, hd]
                for h0 in range(0, H, G):                         # one KV head's query heads
                    sc = (qh[h0:h0 + G] @ K[:, h0:h0 + G].transpose(1, 2, 0)) / np.sqrt(hd)
                    sc = np.where(mask[None, :, :], -np.inf, sc)  # [G, n, T]
                    p = softmax(sc, axis=-1)
                    att[r0:r1, h0:h0 + G] = (p @ Vv[:, h0:h0 + G].transpose(1, 0, 2)).transpose(1, 0, 2)
            h = h + att.reshape(N, H * hd) @ self.w(f"l{l}.wo").T
            a = rms_norm(h, self.w(f"l{l}.ffn_norm"), S.norm_eps)
            g = a @ self.w(f"l{l}.w_gate").T
            u = a @ self.w(f"l{l}.w_up").T
            h = h + (silu(g) * u) @ self.w(f"l{l}.w_down").T
        if last_only:
            h = h[offs[1:] - 1]
            offs = np.arange(len(seqs) + 1)
        hf = rms_norm(h, self.w("final_norm"), S.norm_eps)
        logits = hf @ self.w("lm_head").T
        return ([logits[offs[s]:offs[s + 1]] for s in range(len(seqs))],
                [hf[offs[s]:offs[s + 1]] for s in range(len(seqs))])

    def forward_full(self, tokens: Sequence[int]):
        """All-position logits and final hidden of one sequence, no cache reuse."""
        lg, hf = self.forward([(self.new_cache(), tokens)])
        return lg[0], hf[0]
