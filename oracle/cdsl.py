"""Oracle of the CDSL lookahead step (fp64), plus the paper's Algorithm 1 and Algorithm 2.

TEST INFRASTRUCTURE. Only tests/, ``__graft_entry__.smoke()`` and bench.py's ``cpu_baseline``
and ``--impl reference`` legs may import this package. The product path never does.

What is computed, in the paper's notation (M_p target, M_q draft, R reward, d lookahead
length, k beams, a_t / r_t thresholds, T the generated sequence, pfx the prefix):

CDSL-k step (the batched reading of Algorithm 1 that the GPU path implements, one step per
prompt):
  1. c_1..c_k   = top-k of M_p(pfx)              (Alg. 2 "argmax topk"; descending logit,
                                                  equal logits -> lower token id first)
  2. x_{b,1..d} = greedy rollout of M_q from pfx + c_b                 (Sec. 3.2.1, Alg. 1)
  3. p_{b,1..d+1} = M_p(pfx + c_b + x_{b,<j}), j = 1..d+1, one pass   (Sec. 3.2.2, Alg. 1)
  4. n_b = number of leading j with argmax p_{b,j} = x_{b,j}           (hard rejection)
     or with u_{b,j} <= min(1, p_{b,j}(x_{b,j}) / q_{b,j}(x_{b,j}))     (speculative sampling,
                                                                         Sec. 3.2.2)
     a_b = n_b / d                                                      (acceptance score)
  5. r_b^full = R(T + c_b + x_{b,1..d})  (the CDLH-appx score, Alg. 2)
     r_b^acc  = R(T + c_b + x_{b,1..n_b}) (the S1 score, Alg. 1)
  6. b* = first beam with the largest r^full                           (Alg. 2 keeps the
                                                                        first of equal rewards)
  7. S1 (a_{b*} >= a_t and r_{b*}^acc >= r_t): emit c_{b*}, x_{b*,1..n}; else (S2/S3/S4
     with b = 0) emit c_{b*} only -- the single CDLH-appx token of Alg. 1's fallback.
  The emission is cut to l_m - len(T) tokens (Alg. 1 only tests the length at its loop head).

Reward (Sec. 4.1): coverage = |keywords covered by T + span| / |keywords| (the lexical
concept-counting reward; 2 of 5 covered -> 0.4). The composite reward of the 7B/13B workloads
is 0.5 * coverage + 0.5 * sigmoid(w . h_last), h_last = M_p's final-normed hidden state at
the span's last token, standing in for the trained reward model of the HTG task.

Readings taken where the paper is silent or garbled are listed in the project's design notes
and repeated at the point of use below.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Sequence

import numpy as np

from .model import KVCache, Transformer, log_softmax

S1, S2_S3, S2_S3_STEP1, S4 = 1, 2, 3, 4


# ------------------------------------------------------------------------------------------
# Decisions (argmax, top-k, beam choice, S1 test) with optional near-tie resolution
# ------------------------------------------------------------------------------------------

class Decider:
    """Takes every discrete decision of a step.

    Alone it applies the tie rules (equal values -> lower index). For parity runs it can be
    given the other implementation's choices (``other``: name -> array) and tolerances: where
    the oracle's own values put that choice within ``tol`` (logits) or ``tol_r`` (rewards) of
    the best, but not exactly equal to it, the choice is adopted and logged in ``adopted``, so
    a run continues along the same path after a near tie. Exact ties always follow the rule."""

    def __init__(self, other: Optional[Dict[str, np.ndarray]] = None,
                 tol: float = 0.0, tol_r: float = 0.0):
        self.other = other
        self.tol = tol
        self.tol_r = tol_r
        self.adopted: List[tuple] = []
        # the oracle's own margin against each adopted choice, in the units of its tolerance
        # (logit / log-probability / reward differences), in the order of ``adopted``
        self.margins: List[float] = []

    def _theirs(self, kind, idx):
        if self.other is None or kind not in self.other:
            return None
        return self.other[kind][idx]

    def argmax(self, v: np.ndarray, kind: str, idx) -> int:
        a = int(np.argmax(v))  # numpy returns the first (lowest) index among equal maxima
        g = self._theirs(kind, idx)
        if g is not None:
            g = int(g)
            if g != a and 0 <= g < v.shape[0] and v[g] != v[a] and v[g] >= v[a] - self.tol:
                self.adopted.append((kind, idx, a, g))
                self.margins.append(float(v[a] - v[g]))
                return g
        return a

    def topk(self, v: np.ndarray, k: int, kind: str, idx) -> np.ndarray:
        order = np.lexsort((np.arange(v.shape[0]), -v))[:k]  # by -value, then by id
        g = self._theirs(kind, idx)
        if g is not None:
            g = np.asarray(g, dtype=np.int64)
            if (not np.array_equal(g, order) and len(set(g.tolist())) == k
                    and np.all((g >= 0) & (g < v.shape[0]))
                    and np.all(np.abs(v[g] - v[order]) <= self.tol)
                    and not np.all(v[g] == v[order])):
                self.adopted.append((kind, idx, order.tolist(), g.tolist()))
                self.margins.append(float(np.max(np.abs(v[g] - v[order]))))
                return g
        return order

    def first_max(self, r: np.ndarray, kind: str, idx) -> int:
        best, best_r = 0, r[0]
        for i in range(1, r.shape[0]):
            if r[i] > best_r:           # strict '>' keeps the first of equal rewards (Alg. 2)
                best, best_r = i, r[i]
        g = self._theirs(kind, idx)
        if g is not None and 0 <= int(g) < r.shape[0]:
            g = int(g)
            if g != best and r[g] != best_r and r[g] >= best_r - self.tol_r:
                self.adopted.append((kind, idx, best, g))
                self.margins.append(float(best_r - r[g]))
                return g
        return best

    def accept(self, log_u: float, log_ratio: float, j: int, kind: str, idx) -> bool:
        """Speculative-sampling test u <= min(1, p/q), as log u <= log p - log q (u < 1).

        ``other[kind][idx]`` is the other side's accepted count n; its decision for position
        j is ``j < n``, adopted when this side's margin is within ``tol``."""
        ok = bool(log_u <= log_ratio)
        g = self._theirs(kind, idx)
        if g is not None:
            theirs = j < int(g)
            if theirs != ok and abs(log_u - log_ratio) <= self.tol:
                self.adopted.append((kind, idx, j, ok, theirs))
                self.margins.append(float(abs(log_u - log_ratio)))
                return theirs
        return ok

    def reward_ok(self, r: float, r_t: float, kind: str, idx) -> bool:
        """r >= r_t, compared in float32 (the precision the CUDA path decides in)."""
        ok = bool(np.float32(r) >= np.float32(r_t))
        g = self._theirs(kind, idx)
        if g is not None and abs(r - r_t) <= self.tol_r and bool(g) != ok:
            self.adopted.append((kind, idx, ok, bool(g)))
            self.margins.append(float(abs(r - r_t)))
            return bool(g)
        return ok


# ------------------------------------------------------------------------------------------
# Parameters, reward, thresholds
# ------------------------------------------------------------------------------------------

@dataclasses.dataclass
class RunParams:
    k: int
    d: int
    a_t: float
    r_t: float
    max_new: int                  # l_m of Alg. 1
    composite_reward: bool        # 0.5 coverage + 0.5 sigmoid(w.h) instead of coverage alone
    b: int = 0                    # Step-1 budget of Alg. 1 (0 = Step-2 only)
    acceptance: int = 0           # 0 hard rejection, 1 speculative sampling (Sec. 3.2.2)
    seed: int = 0                 # seed of the speculative-sampling uniforms


HARD, SPECULATIVE = 0, 1
_MASK64 = (1 << 64) - 1


def splitmix64(seed: int, c: int) -> int:
    """Output number c (from 0) of the SplitMix64 generator seeded with ``seed``.

    SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number generators", OOPSLA
    2014): the state advances by the golden-ratio gamma 0x9E3779B97F4A7C15 and each output is
    the state after that step run through the variant-13 mixer (xor-shift 30, multiply,
    xor-shift 27, multiply, xor-shift 31)."""
    z = (seed + (c + 1) * 0x9E3779B97F4A7C15) & _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def uniform24(seed: int, c: int) -> float:
    """u in [0, 1) with 24 random bits (exact in float32): the top 24 bits of output c."""
    return (splitmix64(seed, c) >> 40) / float(1 << 24)


def draw_index(step: int, B: int, b: int, k: int, beam: int, d: int, j: int) -> int:
    """Counter of the uniform of prompt b, beam, lookahead position j (0-based) at ``step``."""
    return ((step * B + b) * k + beam) * d + j


def n_min(a_t: float, d: int) -> int:
    """Smallest n in [0, d] with n / d >= a_t, both in float32; d + 1 when none is.

    a = n/d >= a_t is then tested as n >= n_min on both sides, so the float division is
    taken once, in one precision."""
    for n in range(d + 1):
        if np.float32(n) / np.float32(d) >= np.float32(a_t):
            return n
    return d + 1


def coverage(keywords: Sequence[int], tokens: Sequence[int]) -> float:
    """Fraction of the keyword ids that occur in ``tokens`` (Sec. 4.1: 2 of 5 -> 0.4)."""
    kw = [int(x) for x in keywords]
    present = set(int(t) for t in tokens)
    return sum(1 for x in kw if x in present) / len(kw)


def reward(keywords, generated: Sequence[int], h_last: np.ndarray, w_head: np.ndarray,
           composite: bool) -> float:
    """R of Sec. 3.2.2 for the synthetic tasks.

    ``generated`` is T followed by the span being scored (the prompt is left out: in the
    CommonGen setting the concept list is part of the prompt itself)."""
    cov = coverage(keywords, generated)
    if not composite:
        return cov
    z = float(np.dot(w_head.astype(np.float64), h_last))
    return 0.5 * cov + 0.5 / (1.0 + np.exp(-z))


def runtime_per_token(c: float, draft_calls: float, target_calls: float) -> float:
    """Sec. 4.3 runtime model: P = c * (M_q calls per token) + (M_p calls per token), where c is
    the cost of one M_q call in units of one M_p call (the ratio of their greedy tokens/s)."""
    return c * draft_calls + target_calls


def speedup(p_base: float, p_method: float) -> float:
    """Sec. 4.3: the speedup of a method over a baseline is the ratio of their runtimes P."""
    return p_base / p_method


# ------------------------------------------------------------------------------------------
# Per-prompt decoding state
# ------------------------------------------------------------------------------------------

@dataclasses.dataclass
class PromptState:
    prompt: List[int]
    T: List[int]                 # generated sequence
    keywords: np.ndarray
    tcache: KVCache              # M_p keys/values of pfx = prompt + T
    dcache: KVCache              # M_q keys/values of pfx
    p_root: np.ndarray           # M_p(pfx): logits of the token after pfx
    h_root: np.ndarray           # M_p final hidden at the last pfx position
    q_root: Optional[np.ndarray]  # M_q(pfx) logits (kept only for the literal Alg. 1)

    @property
    def pfx(self) -> List[int]:
        return self.prompt + self.T


def prefill(target: Transformer, draft: Transformer, prompts: np.ndarray,
            keywords: np.ndarray, keep_draft_logits: bool = False) -> List[PromptState]:
    """Run both models over every prompt; the target's last row gives M_p(pfx)."""
    B = prompts.shape[0]
    tcs = [target.new_cache() for _ in range(B)]
    dcs = [draft.new_cache() for _ in range(B)]
    tl, th = target.forward([(tcs[b], prompts[b].tolist()) for b in range(B)], last_only=True)
    dl, _ = draft.forward([(dcs[b], prompts[b].tolist()) for b in range(B)], last_only=True)
    return [PromptState(prompt=prompts[b].tolist(), T=[], keywords=keywords[b], tcache=tcs[b],
                        dcache=dcs[b], p_root=tl[b][-1], h_root=th[b][-1],
                        q_root=dl[b][-1] if keep_draft_logits else None) for b in range(B)]


# ------------------------------------------------------------------------------------------
# CDSL-k step
# ------------------------------------------------------------------------------------------

@dataclasses.dataclass
class StepRecord:
    """Everything one CDSL-k step decides, per prompt (arrays over beams / positions)."""
    active: bool
    roots: np.ndarray            # [k]       c_1..c_k
    x: np.ndarray                # [k, d]    drafted tokens
    logq: np.ndarray             # [k, d]    log q_j(x_j)
    vlogits: np.ndarray          # [k, d+1, V]  M_p logits of rows [c, x_1..x_d]
    argmax: np.ndarray           # [k, d+1]  argmax of each verify row
    logp: np.ndarray             # [k, d]    log p_j(x_j)
    n: np.ndarray                # [k]       accepted count
    r_full: np.ndarray           # [k]
    r_acc: np.ndarray            # [k]
    head: np.ndarray             # [k, d+1]  sigmoid(w . h) per verify row (0 without a head)
    beam: int
    state: int
    emitted: List[int]
    # Step-1 rounds after the first (budget b >= 2), in order: the round's M_p greedy token and
    # its d-token M_q lookahead [tok, lh_1..lh_d], and the reward R(T + X + tok + lh)
    step1_rounds: List[tuple] = dataclasses.field(default_factory=list)


def _step1(target: Transformer, draft: Transformer, st: PromptState, run: RunParams, w_head,
           dec: "Decider", b: int, L: int, roots, r_full, vlog, am, tc, dc, X: List[tuple],
           rounds: List[tuple]) -> bool:
    """Step-1 of Alg. 1's S2/S3 branch (Sec. 3.2.3) in the CDSL-k step, budget run.b.

    Round 1: M_p's greedy token after pfx is the root c_1 and its d-token M_q lookahead is beam
    1's draft, so its reward is r_1^full (data the step already has). Round i > 1: the next
    token is M_p's argmax after pfx + X (round 2: verify row (1, 0)), its lookahead is d greedy
    M_q tokens after pfx + X + token, and the reward is R(T + X + token + lh) with M_p's hidden
    state at lh_d. The first round whose reward reaches r_t ends Step-1 with X emitted.

    Appends (token, M_p cache through it, M_q cache through it, M_p logits after it) to X for
    every round taken and (token + lh, reward) to ``rounds`` for rounds > 1. True on success."""
    d = run.d
    c1 = int(roots[0])
    X.append((c1, tc[(b, 0)].truncated(L + 1), dc[(b, 0)].truncated(L + 1), vlog[0, 0]))
    if dec.reward_ok(r_full[0], run.r_t, "step1", b):
        return True
    for i in range(1, run.b):
        _, tcx, dcx, p_after = X[-1]
        tok = int(am[0, 0]) if i == 1 else dec.argmax(p_after, "step1_tok", (b, i))
        dce = dcx.fork()
        lg, _ = draft.forward([(dce, [tok])])
        lh = []
        for j in range(d):
            t = dec.argmax(lg[0][-1], "step1_x", (b, i, j))
            lh.append(t)
            if j + 1 < d:
                lg, _ = draft.forward([(dce, [t])])
        tce = tcx.fork()
        vl2, vh2 = target.forward([(tce, [tok] + lh)])
        span = [t for t, _, _, _ in X] + [tok] + lh
        r = reward(st.keywords, st.T + span, vh2[0][d], w_head, run.composite_reward)
        n_x = len(X) + 1
        X.append((tok, tce.truncated(L + n_x), dce.truncated(L + n_x), vl2[0][0]))
        rounds.append((np.asarray([tok] + lh, dtype=np.int64), r))
        if dec.reward_ok(r, run.r_t, f"step1_{i + 1}", b):
            return True
    return False


def cdsl_k_step(target: Transformer, draft: Transformer, states: List[PromptState],
                run: RunParams, w_head: np.ndarray,
                decider: Optional[Decider] = None, step: int = 0) -> List[StepRecord]:
    """One CDSL-k step for every prompt that has not reached l_m; updates ``states``.

    ``step`` is the number of steps taken before this one (it indexes the speculative-sampling
    uniforms)."""
    dec = decider or Decider()
    k, d = run.k, run.d
    nmin = n_min(run.a_t, d)
    V = target.shape.vocab
    live = [b for b, st in enumerate(states) if len(st.T) < run.max_new]
    recs: List[Optional[StepRecord]] = [None] * len(states)
    for b, st in enumerate(states):
        if b not in live:
            z = np.zeros
            recs[b] = StepRecord(False, z(k, np.int64), z((k, d), np.int64), z((k, d)),
                                 z((k, d + 1, V)), z((k, d + 1), np.int64), z((k, d)),
                                 z(k, np.int64), z(k), z(k), z((k, d + 1)), -1, 0, [])
    if not live:
        return recs

    # 1. roots
    roots = {b: dec.topk(states[b].p_root, k, "roots", b) for b in live}

    # 2. greedy draft rollout of every beam: d calls of M_q, each over all (prompt, beam) rows
    dc = {(b, i): states[b].dcache.fork() for b in live for i in range(k)}
    x = {b: np.zeros((k, d), np.int64) for b in live}
    logq = {b: np.zeros((k, d)) for b in live}
    feed = {(b, i): int(roots[b][i]) for b in live for i in range(k)}
    keys = [(b, i) for b in live for i in range(k)]
    for j in range(d):
        lg, _ = draft.forward([(dc[key], [feed[key]]) for key in keys])
        for key, row in zip(keys, lg):
            b, i = key
            xj = dec.argmax(row[0], "x", (b, i, j))
            x[b][i, j] = xj
            logq[b][i, j] = log_softmax(row[0])[xj]
            feed[key] = xj

    # 3. one M_p pass over [c_b, x_b1..x_bd] for every beam
    tc = {(b, i): states[b].tcache.fork() for b in live for i in range(k)}
    vl, vh = target.forward([(tc[(b, i)], [int(roots[b][i])] + x[b][i].tolist())
                             for (b, i) in keys])
    for b in live:
        st = states[b]
        vlog = np.stack([vl[keys.index((b, i))] for i in range(k)])   # [k, d+1, V]
        vhid = np.stack([vh[keys.index((b, i))] for i in range(k)])   # [k, d+1, D]
        am = np.zeros((k, d + 1), np.int64)
        logp = np.zeros((k, d))
        n = np.zeros(k, np.int64)
        head = np.zeros((k, d + 1))
        for i in range(k):
            for j in range(d + 1):
                am[i, j] = dec.argmax(vlog[i, j], "argmax", (b, i, j))
                if run.composite_reward:
                    head[i, j] = 1.0 / (1.0 + np.exp(-float(np.dot(w_head.astype(np.float64),
                                                                   vhid[i, j]))))
            for j in range(d):
                logp[i, j] = log_softmax(vlog[i, j])[x[b][i, j]]
            # 4. validation by M_p (Sec. 3.2.2): row j-1 gives p_j for x_j
            for j in range(d):
                if run.acceptance == HARD:        # hard rejection: argmax p_j == x_j
                    ok = am[i, j] == x[b][i, j]
                else:                             # speculative sampling: u <= min(1, p/q)
                    u = uniform24(run.seed, draw_index(step, len(states), b, k, i, d, j))
                    log_u = np.log(u) if u > 0.0 else -np.inf
                    ok = dec.accept(log_u, logp[i, j] - logq[b][i, j], j, "spec", (b, i))
                if not ok:
                    break
                n[i] += 1
        # 5. rewards
        r_full = np.zeros(k)
        r_acc = np.zeros(k)
        for i in range(k):
            span_full = [int(roots[b][i])] + x[b][i].tolist()
            span_acc = [int(roots[b][i])] + x[b][i, :n[i]].tolist()
            r_full[i] = reward(st.keywords, st.T + span_full, vhid[i, d], w_head,
                               run.composite_reward)
            r_acc[i] = reward(st.keywords, st.T + span_acc, vhid[i, n[i]], w_head,
                              run.composite_reward)
        # 6. beam
        bs = dec.first_max(r_full, "beam", b)
        # 7. state and emission
        L = len(st.prompt) + len(st.T)
        rounds: List[tuple] = []
        X: List[int] = []
        if n[bs] >= nmin and dec.reward_ok(r_acc[bs], run.r_t, "s1", b):
            state = S1
            out = [int(roots[b][bs])] + x[b][bs, :n[bs]].tolist()
        elif n[bs] < nmin and run.b >= 1 and _step1(target, draft, st, run, w_head, dec, b, L,
                                                    roots[b], r_full, vlog, am, tc, dc, X,
                                                    rounds):
            # S2/S3, Step-1 (Alg. 1, Sec. 3.2.3): X = M_p's greedy tokens, the last of which
            # had a lookahead reward >= r_t
            state = S2_S3_STEP1
            bs = 0
            out = [t for t, _, _, _ in X]
        else:
            state = S2_S3 if n[bs] < nmin else S4
            out = [int(roots[b][bs])]
        n_emit = min(len(out), run.max_new - len(st.T))
        out = out[:n_emit]

        # commit: pfx <- pfx + O. The winner's caches hold exactly these positions.
        if state == S2_S3_STEP1 and n_emit >= 2:
            _, tcx, dcx, p_after = X[n_emit - 1]
            st.tcache = tcx.truncated(L + n_emit)
            st.p_root = p_after
            st.h_root = None
            st.dcache = dcx.truncated(L + n_emit)
        else:
            st.tcache = tc[(b, bs)].truncated(L + n_emit)
            st.p_root = vlog[bs, n_emit - 1]
            st.h_root = vhid[bs, n_emit - 1]
            # the winner's draft cache holds [c, x_1..x_{d-1}]; x_d (full accept) is run now
            st.dcache = dc[(b, bs)].truncated(L + min(n_emit, d))
            if n_emit == d + 1:
                draft.forward([(st.dcache, [out[d]])])
        st.T = st.T + out
        recs[b] = StepRecord(True, np.asarray(roots[b]), x[b], logq[b], vlog, am, logp, n,
                             r_full, r_acc, head, bs, state, out, rounds)
    return recs


def cdsl_k_generate(target, draft, prompts, keywords, run: RunParams, w_head,
                    max_steps: int = 10_000):
    """Run CDSL-k steps until every prompt has l_m tokens. Returns (states, records)."""
    states = prefill(target, draft, prompts, keywords)
    records = []
    for step in range(max_steps):
        if all(len(st.T) >= run.max_new for st in states):
            break
        records.append(cdsl_k_step(target, draft, states, run, w_head, step=step))
    return states, records


# ------------------------------------------------------------------------------------------
# Literal Algorithm 1 (single draft, Step-1 budget b) and Algorithm 2 (CDLH / CDLH-appx)
# ------------------------------------------------------------------------------------------

def _extend(model: Transformer, cache: KVCache, tokens: Sequence[int]):
    c = cache.fork()
    lg, hf = model.forward([(c, list(tokens))])
    return c, lg[0], hf[0]


def _greedy(model: Transformer, cache: KVCache, first_logits: np.ndarray, first_token,
            d: int) -> List[int]:
    """d greedy tokens of ``model`` after pfx (+ first_token when given).

    first_logits: the model's logits at the end of pfx (used when first_token is None)."""
    c = cache.fork()
    if first_token is None:
        logits = first_logits
    else:
        lg, _ = model.forward([(c, [int(first_token)])])
        logits = lg[0][-1]
    out = []
    for j in range(d):
        t = int(np.argmax(logits))
        out.append(t)
        if j + 1 < d:
            lg, _ = model.forward([(c, [t])])
            logits = lg[0][-1]
    return out


def _score(target: Transformer, st: PromptState, base: List[int], span: List[int],
           run: RunParams, w_head) -> float:
    """R(pfx + base + span): coverage over T + base + span, head on M_p's last hidden."""
    h_last = None
    if run.composite_reward:
        _, _, hf = _extend(target, st.tcache, base + span)
        h_last = hf[-1]
    return reward(st.keywords, st.T + base + span, h_last, w_head, run.composite_reward)


def cdlh_token(target: Transformer, lookahead: Transformer, st: PromptState,
               base: List[int], run: RunParams, w_head) -> int:
    """One token of Algorithm 2 at pfx + base: top-k of M_p, a d-token greedy lookahead of
    ``lookahead`` (M_p for CDLH, M_q for CDLH-appx) after each candidate, the candidate with
    the largest R(pfx + x_i + lh) wins (strict '>', so the first of equal rewards).

    Reading: the candidate x_i is part of the scored text and the prefix update happens once,
    after the candidate loop (Algorithm 2's loop nesting and its R(pfx + lh) are read as typos)."""
    if base:
        tcache, p, _ = _extend(target, st.tcache, base)
        p = p[-1]
        lcache = (tcache if lookahead is target else _extend(lookahead, st.dcache, base)[0])
    else:
        p, tcache = st.p_root, st.tcache
        lcache = st.tcache if lookahead is target else st.dcache
    cands = np.lexsort((np.arange(p.shape[0]), -p))[:run.k]
    best, best_r = None, -np.inf
    for c in cands:
        lh = _greedy(lookahead, lcache, None, int(c), run.d)
        r = _score(target, st, base, [int(c)] + lh, run, w_head)
        if r > best_r:
            best, best_r = int(c), r
    return best


def _commit(target, draft, st: PromptState, out: List[int], keep_draft_logits=True):
    """pfx <- pfx + O by running both models over O (plain recomputation)."""
    if not out:
        return
    lg, hf = target.forward([(st.tcache, out)])
    st.p_root, st.h_root = lg[0][-1], hf[0][-1]
    dl, _ = draft.forward([(st.dcache, out)])
    if keep_draft_logits:
        st.q_root = dl[0][-1]
    st.T = st.T + out


def alg1_step(target: Transformer, draft: Transformer, st: PromptState, run: RunParams,
              w_head) -> dict:
    """One decision of literal Algorithm 1 (Sec. 3.2.3; hard rejection, Step-1 budget b), from the
    method's description: d greedy M_q tokens, one M_p pass over them, the count n of accepted
    tokens, the reward of the accepted span, then S1, S2/S3 (Step-1 rounds, else the Step-2
    CDLH-appx token) or S4.

    Readings: the verify pass yields p_i = M_p(pfx + x_<i) for i = 1..d (its last row, the
    (d+1)-th distribution, is not used); Step-1 tokens are new tokens appended to X, the
    drafted x_1..x_n stay; with n = 0 the S1 reward is R(T) on the prefix alone."""
    d = run.d
    nmin = n_min(run.a_t, d)
    x = _greedy(draft, st.dcache, st.q_root, None, d)
    tc, vl, vh = _extend(target, st.tcache, x)
    p = [st.p_root] + [vl[j] for j in range(d)]
    hrow = [st.h_root] + [vh[j] for j in range(d)]
    n = 0
    for i in range(d):
        if int(np.argmax(p[i])) != x[i]:
            break
        n += 1
    r = reward(st.keywords, st.T + x[:n], hrow[n], w_head, run.composite_reward)
    acc = x[:n]
    if n >= nmin and np.float32(r) >= np.float32(run.r_t):
        state, out = S1, acc
    elif n < nmin:
        state, out = S2_S3, None
        X: List[int] = []
        for _ in range(run.b):                       # Step-1
            p_next = _extend(target, st.tcache, acc + X)[1][-1] if acc + X else st.p_root
            X.append(int(np.argmax(p_next)))
            dcache_x, ql, _ = _extend(draft, st.dcache, acc + X)
            lh = _greedy(draft, dcache_x, ql[-1], None, d)
            if np.float32(_score(target, st, acc + X, lh, run, w_head)) >= np.float32(run.r_t):
                out = acc + X
                break
        if out is None:                              # Step-2 = CDLH-appx
            out = acc + [cdlh_token(target, draft, st, acc, run, w_head)]
    else:
        state = S4
        out = acc + [cdlh_token(target, draft, st, acc, run, w_head)]
    out = out[:run.max_new - len(st.T)]
    _commit(target, draft, st, out)
    return dict(x=x, n=n, a=n / d, r=r, state=state, emitted=out)


def alg1_generate(target, draft, prompt, kw, run: RunParams, w_head, max_steps=10_000):
    st = prefill(target, draft, np.asarray([prompt]), np.asarray([kw]), keep_draft_logits=True)[0]
    recs = []
    for _ in range(max_steps):
        if len(st.T) >= run.max_new:
            break
        recs.append(alg1_step(target, draft, st, run, w_head))
    return st, recs


def cdlh_generate(target, lookahead, draft_for_state, prompt, kw, run: RunParams, w_head,
                  max_steps=10_000):
    """Algorithm 2: CDLH (lookahead = target) or CDLH-appx (lookahead = draft)."""
    st = prefill(target, draft_for_state, np.asarray([prompt]), np.asarray([kw]))[0]
    for _ in range(max_steps):
        if len(st.T) >= run.max_new:
            break
        t = cdlh_token(target, lookahead, st, [], run, w_head)
        _commit(target, draft_for_state, st, [t], keep_draft_logits=False)
    return st
