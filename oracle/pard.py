"""PARD decode step on the CPU -- oracle (test infrastructure only).

Follows the paper's statement of the method:

* Parallel draft (Section 3.1, Eq. 6): the draft model reads the accepted
  prefix followed by mask tokens m_0..m_{K-2} (one shared id by default,
  Section 4.3 "Shared Mask Token ID"; one id per offset when mask_ids is set,
  the alternative that section compares) and predicts x_n..x_{n+K-1} in one
  forward pass;
  the prediction for x_{n+k} is read at the row holding m_{k-1} (k >= 1) or at
  the last real token (k = 0), so it conditions on x_0..x_{n-1}, m_0..m_{k-1}.
* Verification (Section 2.2): one target forward over the last accepted
  token and the K candidates, at positions n-1..n+K-1.
* Acceptance: the paper defers to speculative sampling (Chen et al. 2023;
  Leviathan et al. 2023, cited in Section 1 and 2.2).  Greedy: keep the
  longest prefix of candidates equal to the target's argmax, then emit the
  target's argmax at the first mismatch.  Sampling: accept d_i when
  u_i * q_i(d_i) < p_i(d_i); at the first rejection emit a token drawn from
  norm(max(0, p_i - q_i)); when all K are accepted emit one drawn from p_K.
* Commit / rollback: the target cache keeps the verified prefix; rejected
  slots are dropped by length.  Draft KV of accepted candidates was computed
  from mask tokens, so those tokens are re-fed to the draft next step.
* Autoregressive greedy decoding (Eq. 2) is the lossless reference.
* Vanilla speculative decoding (Section 2.2, drafting stage; the
  autoregressive factorization of Section 3.1): the same draft model
  produces the K candidates one forward pass at a time, pass i feeding
  candidate i-1 at the next position; verification, acceptance and commit are
  unchanged.  Its per-iteration time is K * T_D + T_T against T_D + T_T for
  PARD (Section 2.2).

Readings where the paper is silent are listed in the repository's design
notes; the ones that change numbers are: argmax takes the lowest index on
ties; acceptance uses a strict '<'; categorical draws use the Gumbel-max
trick with Philox uniforms (stream layout in ``philox.py``).
"""
from __future__ import annotations

import ctypes
from typing import List, Optional, Sequence, Tuple

import numpy as np

from . import OCfg, OWeights, LAYER_ORDER, T_PER_LAYER, lib
from .philox import (STREAM_ACCEPT, STREAM_BONUS, STREAM_DRAFT, gumbel, raw_words, uniform01)


class OracleModel:
    """One decoder (target or draft) with a per-sequence KV cache.  The cache
    holds bf16 values (the paper's model precision, Table 3) unless
    ``kv_bf16=False``, which keeps fp32 keys and values."""

    def __init__(self, shape, weights: dict, batch: int, max_pos: int, kv_bf16: bool = True):
        self.shape = shape
        self.max_pos = max_pos
        self.kv_bf16 = bool(kv_bf16)
        self.cfg = OCfg(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads,
                        shape.head_dim, shape.ffn, shape.vocab, shape.rope_theta, shape.rms_eps)
        self._keep = []
        ptrs = (ctypes.c_void_p * (shape.n_layers * T_PER_LAYER))()
        for l in range(shape.n_layers):
            for j, name in enumerate(LAYER_ORDER):
                a = np.ascontiguousarray(weights["layers"][l][name], dtype=np.uint16)
                self._keep.append(a)
                ptrs[l * T_PER_LAYER + j] = a.ctypes.data
        glob = [np.ascontiguousarray(weights[n], dtype=np.uint16) for n in ("embed", "final_norm", "lm_head")]
        self._keep += glob
        self._ptrs = ptrs
        self.w = OWeights(glob[0].ctypes.data, glob[1].ctypes.data, glob[2].ctypes.data,
                          ctypes.cast(ptrs, ctypes.POINTER(ctypes.c_void_p)))
        kv_shape = (shape.n_layers, max_pos, shape.n_kv_heads, shape.head_dim)
        self.kc = [np.zeros(kv_shape, dtype=np.float32) for _ in range(batch)]
        self.vc = [np.zeros(kv_shape, dtype=np.float32) for _ in range(batch)]

    def forward(self, b: int, tokens: Sequence[int], positions: Sequence[int],
                out_rows: Sequence[int], want_hidden: bool = False):
        """New rows ``tokens`` at ``positions`` for sequence b; their K/V are
        written to the cache.  Returns logits [len(out_rows), V] (and the
        final-norm input when ``want_hidden``)."""
        tok = np.ascontiguousarray(tokens, dtype=np.int32)
        pos = np.ascontiguousarray(positions, dtype=np.int32)
        rows = np.ascontiguousarray(out_rows, dtype=np.int32)
        m = len(tok)
        logits = np.empty((max(len(rows), 1), self.shape.vocab), dtype=np.float32)
        hidden = np.empty((m, self.shape.d_model), dtype=np.float32) if want_hidden else None
        rc = lib().oracle_forward(ctypes.byref(self.cfg), ctypes.byref(self.w),
                                  self.kc[b].ctypes.data, self.vc[b].ctypes.data, self.max_pos,
                                  tok.ctypes.data, m, pos.ctypes.data, rows.ctypes.data, len(rows),
                                  logits.ctypes.data, hidden.ctypes.data if want_hidden else None,
                                  int(self.kv_bf16))
        if rc != 0:
            raise ValueError(f"oracle_forward rejected its arguments (code {rc})")
        logits = logits[:len(rows)]
        return (logits, hidden) if want_hidden else logits


# --------------------------------------------------------------------------
# Acceptance rules
# --------------------------------------------------------------------------
def argmax_lowest(x: np.ndarray) -> int:
    """Argmax, lowest index on ties (np.argmax's rule)."""
    return int(np.argmax(x))


def softmax_t(logits: np.ndarray, temperature: float) -> np.ndarray:
    """softmax(logits / T) in fp32."""
    z = (np.asarray(logits, dtype=np.float32) / np.float32(temperature)).astype(np.float32)
    e = np.exp((z - z.max()).astype(np.float32)).astype(np.float32)
    return (e / e.sum(dtype=np.float32)).astype(np.float32)


def gumbel_noise(seed: int, stream: int, step: int, b: int, i: int, V: int) -> np.ndarray:
    return gumbel(raw_words(seed, stream, step, b, i, np.arange(V, dtype=np.uint64)))


def sample_gumbel_max(scores: np.ndarray, seed: int, stream: int, step: int, b: int, i: int) -> int:
    """One categorical draw from softmax(scores): argmax(scores + Gumbel)."""
    g = gumbel_noise(seed, stream, step, b, i, scores.shape[-1])
    return argmax_lowest((np.asarray(scores, dtype=np.float32) + g).astype(np.float32))


def accept_greedy(d: Sequence[int], y: np.ndarray) -> Tuple[int, List[int]]:
    """Greedy verification: a = longest prefix with d_i == argmax y_i,
    emitted = d_0..d_{a-1} followed by argmax y_a."""
    K = len(d)
    t = [argmax_lowest(y[i]) for i in range(K + 1)]
    a = 0
    while a < K and int(d[a]) == t[a]:
        a += 1
    return a, [int(x) for x in d[:a]] + [t[a]]


def accept_sampling(d: Sequence[int], z: np.ndarray, y: np.ndarray, temperature: float,
                    seed: int, step: int, b: int) -> Tuple[int, List[int]]:
    """Speculative sampling: accept d_i while u_i * q_i(d_i) < p_i(d_i);
    at the first rejection j draw the bonus from norm(max(0, p_j - q_j));
    if all K are accepted draw it from p_K.  p = softmax(y/T), q = softmax(z/T)."""
    K = len(d)
    for i in range(K):
        p = softmax_t(y[i], temperature)
        q = softmax_t(z[i], temperature)
        u = uniform01(raw_words(seed, STREAM_ACCEPT, step, b, i, np.zeros(1, dtype=np.uint64)))[0]
        di = int(d[i])
        if np.float32(u * q[di]) < p[di]:
            continue
        w = np.maximum(p - q, np.float32(0.0)).astype(np.float32)
        g = gumbel_noise(seed, STREAM_BONUS, step, b, 0, len(w))
        with np.errstate(divide="ignore"):
            score = np.where(w > 0, np.log(w).astype(np.float32) + g, -np.inf).astype(np.float32)
        if not np.isfinite(score).any():          # p == q everywhere: cannot reject
            score = (np.log(p).astype(np.float32) + g).astype(np.float32)
        return i, [int(x) for x in d[:i]] + [argmax_lowest(score)]
    zK = (np.asarray(y[K], dtype=np.float32) / np.float32(temperature)).astype(np.float32)
    return K, [int(x) for x in d] + [sample_gumbel_max(zK, seed, STREAM_BONUS, step, b, 0)]


def draft_token(zi: np.ndarray, i: int, sample: bool, temperature: float, seed: int, step: int, b: int) -> int:
    """Candidate i: argmax z_i (greedy) or a draw from softmax(z_i / T) by
    Gumbel-max with the draft stream's uniforms of row i."""
    if not sample:
        return argmax_lowest(zi)
    zt = (np.asarray(zi, dtype=np.float32) / np.float32(temperature)).astype(np.float32)
    return sample_gumbel_max(zt, seed, STREAM_DRAFT, step, b, i)


def draft_tokens(z: np.ndarray, sample: bool, temperature: float, seed: int, step: int, b: int) -> List[int]:
    """d_i = argmax z_i (greedy) or a draw from softmax(z_i / T) by Gumbel-max."""
    return [draft_token(z[i], i, sample, temperature, seed, step, b) for i in range(z.shape[0])]


# --------------------------------------------------------------------------
# Decode loop
# --------------------------------------------------------------------------
class OracleDecoder:
    """Step-by-step PARD decoding of a batch, mirroring the library's calls:
    prefill -> (draft -> verify -> accept -> commit)*."""

    def __init__(self, wl, target_w: dict, draft_w: dict,
                 page_order_t: Optional[np.ndarray] = None, page_order_d: Optional[np.ndarray] = None,
                 prompt_lens: Optional[Sequence[int]] = None):
        self.wl = wl
        self.K = wl.K
        lens = list(prompt_lens) if prompt_lens is not None else wl.prompt_lens()
        self.reserve = [wl.pages_per_seq(L) for L in lens]
        max_pos = max(self.reserve) * wl.page_size
        self.T = OracleModel(wl.target, target_w, wl.batch, max_pos)
        self.D = OracleModel(wl.draft, draft_w, wl.batch, max_pos)
        self.mask_id = wl.draft.mask_id
        self.mask_ids: Optional[List[int]] = None  # one id per mask offset (Section 4.3); None: shared
        n_pages = sum(self.reserve)
        po_t = page_order_t if page_order_t is not None else np.arange(n_pages, dtype=np.int32)
        po_d = page_order_d if page_order_d is not None else np.arange(n_pages, dtype=np.int32)
        self.table_t = self._reserve(po_t)
        self.table_d = self._reserve(po_d)

    def _reserve(self, order: np.ndarray) -> List[np.ndarray]:
        """Sequences take their pages in order b = 0..B-1 from the front of
        the pool's page order."""
        out, at = [], 0
        for r in self.reserve:
            out.append(np.asarray(order[at:at + r], dtype=np.int64))
            at += r
        return out

    def slot(self, table: np.ndarray, pos: int) -> int:
        ps = self.wl.page_size
        return int(table[pos // ps]) * ps + pos % ps

    # -- prefill ----------------------------------------------------------
    def prefill(self, prompts: Sequence[np.ndarray], seed: int = 0) -> List[int]:
        """Both models process the prompt; the target's last-row logits give
        the first new token.  After it: n = P + 1, target cache P entries,
        draft pending = [x_P]."""
        wl = self.wl
        self.n, self.pending, self.generated, self.done = [], [], [], []
        self.prefill_logits = []
        first = []
        for b, pr in enumerate(prompts):
            P = len(pr)
            pos = np.arange(P, dtype=np.int32)
            lg = self.T.forward(b, pr, pos, [P - 1])[0]
            self.prefill_logits.append(lg)
            self.D.forward(b, pr, pos, [])
            if wl.sample:
                zT = (lg / np.float32(wl.temperature)).astype(np.float32)
                x = sample_gumbel_max(zT, seed, STREAM_BONUS, 0, b, 0)
            else:
                x = argmax_lowest(lg)
            first.append(x)
            self.n.append(P + 1)
            self.pending.append([x])
            self.generated.append([x])
            self.done.append(wl.n_new <= 1)
        return first

    def force_first(self, b: int, tok: int) -> None:
        """Teacher forcing: replace sequence b's first generated token."""
        self.pending[b] = [int(tok)]
        self.generated[b] = [int(tok)]

    # -- one step -----------------------------------------------------------
    def draft(self, step: int, seed: int = 0) -> Tuple[np.ndarray, np.ndarray]:
        """Eq. 6: pending real tokens then K-1 mask tokens; logits read at the
        last real row and at every mask row.  Returns d [B,K], z [B,K,V]."""
        wl, K = self.wl, self.K
        V = wl.draft.vocab
        d = np.zeros((wl.batch, K), dtype=np.int32)
        z = np.zeros((wl.batch, K, V), dtype=np.float32)
        for b in range(wl.batch):
            if self.done[b]:
                continue
            pend = self.pending[b]
            p, n = len(pend), self.n[b]
            masks = [self.mask_id] * (K - 1) if self.mask_ids is None else [int(x) for x in self.mask_ids[:K - 1]]
            rows = list(pend) + masks
            pos = list(range(n - p, n + K - 1))
            zb = self.D.forward(b, rows, pos, [p - 1 + i for i in range(K)])
            z[b] = zb
            d[b] = draft_tokens(zb, wl.sample, wl.temperature, seed, step, b)
        return d, z

    def draft_sequential(self, step: int, seed: int = 0,
                         feed: Optional[np.ndarray] = None) -> Tuple[np.ndarray, np.ndarray]:
        """Vanilla speculative decoding's drafting stage: K forward passes of
        the draft model; pass 0 feeds the pending real tokens and reads its
        last row, pass i >= 1 feeds candidate i-1 at position n-1+i.  The
        draft cache keeps what the passes wrote; commit rolls it back by
        length exactly as for the parallel draft (the pending tokens are fed
        again next step).  feed [B,K] (teacher forcing): pass i >= 1 feeds
        feed[b, i-1] instead of the oracle's own candidate.  Returns d [B,K],
        z [B,K,V]."""
        wl, K = self.wl, self.K
        V = wl.draft.vocab
        d = np.zeros((wl.batch, K), dtype=np.int32)
        z = np.zeros((wl.batch, K, V), dtype=np.float32)
        for b in range(wl.batch):
            if self.done[b]:
                continue
            pend = self.pending[b]
            p, n = len(pend), self.n[b]
            zi = self.D.forward(b, pend, list(range(n - p, n)), [p - 1])[0]
            for i in range(K):
                if i > 0:
                    prev = int(d[b, i - 1]) if feed is None else int(feed[b, i - 1])
                    zi = self.D.forward(b, [prev], [n - 1 + i], [0])[0]
                z[b, i] = zi
                d[b, i] = draft_token(zi, i, wl.sample, wl.temperature, seed, step, b)
        return d, z

    def verify(self, d: np.ndarray) -> np.ndarray:
        """Target forward over [x_{n-1}, d_0..d_{K-1}] at positions n-1..n+K-1."""
        wl, K = self.wl, self.K
        y = np.zeros((wl.batch, K + 1, wl.target.vocab), dtype=np.float32)
        for b in range(wl.batch):
            if self.done[b]:
                continue
            n = self.n[b]
            rows = [self.pending[b][-1]] + [int(x) for x in d[b]]
            y[b] = self.T.forward(b, rows, list(range(n - 1, n + K)), list(range(K + 1)))
        return y

    def accept(self, d: np.ndarray, z: np.ndarray, y: np.ndarray, step: int, seed: int = 0):
        """Returns accept lengths [B] and emitted lists (a+1 tokens each)."""
        wl = self.wl
        acc, emitted = [], []
        for b in range(wl.batch):
            if self.done[b]:
                acc.append(0)
                emitted.append([])
                continue
            if wl.sample:
                a, e = accept_sampling(d[b], z[b], y[b], wl.temperature, seed, step, b)
            else:
                a, e = accept_greedy(d[b], y[b])
            acc.append(a)
            emitted.append(e)
        return acc, emitted

    def commit(self, acc: Sequence[int], emitted: Sequence[Sequence[int]]):
        """Target keeps positions n-1..n-1+a (x_{n-1} and the accepted
        candidates); rejected slots are dropped by length.  Draft pending
        becomes the emitted tokens.  Returns (kv_slots [B, K+1] with -1 past
        a, number of tokens counted toward n_new per sequence)."""
        wl, K = self.wl, self.K
        slots = np.full((wl.batch, K + 1), -1, dtype=np.int64)
        n_out = []
        for b in range(wl.batch):
            if self.done[b]:
                n_out.append(0)
                continue
            a, n = int(acc[b]), self.n[b]
            for j in range(a + 1):
                slots[b, j] = self.slot(self.table_t[b], n - 1 + j)
            self.n[b] = n + a + 1
            self.pending[b] = [int(x) for x in emitted[b]]
            room = wl.n_new - len(self.generated[b])
            take = min(room, a + 1)
            self.generated[b] += [int(x) for x in emitted[b][:take]]
            n_out.append(take)
            if len(self.generated[b]) >= wl.n_new:
                self.done[b] = True
        return slots, n_out

    def all_done(self) -> bool:
        return all(self.done)

    def run(self, prompts, seed: int = 0, max_steps: int = 10 ** 6, sequential: bool = False):
        """Full generation; returns (generated tokens per sequence, trace).
        sequential: vanilla speculative decoding's K-pass draft instead of
        the parallel one."""
        self.prefill(prompts, seed)
        trace = []
        step = 1
        while not self.all_done() and step <= max_steps:
            d, z = self.draft_sequential(step, seed) if sequential else self.draft(step, seed)
            y = self.verify(d)
            acc, em = self.accept(d, z, y, step, seed)
            slots, n_out = self.commit(acc, em)
            trace.append(dict(d=d, acc=acc, emitted=em, slots=slots))
            step += 1
        return self.generated, trace


def ar_greedy(shape, weights: dict, prompt: Sequence[int], n_new: int, kv_bf16: bool = True) -> List[int]:
    """Eq. 2: x_t = argmax P(x | x_0..x_{t-1}), one target forward per token."""
    P = len(prompt)
    m = OracleModel(shape, weights, 1, P + n_new + 1, kv_bf16)
    lg = m.forward(0, prompt, np.arange(P, dtype=np.int32), [P - 1])[0]
    out = [argmax_lowest(lg)]
    while len(out) < n_new:
        pos = P + len(out) - 1
        lg = m.forward(0, [out[-1]], [pos], [0])[0]
        out.append(argmax_lowest(lg))
    return out
