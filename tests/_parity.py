"""Shared harness of the GPU parity tests: the same seeded inputs go to the
CUDA path (through the C ABI) and to the CPU oracle; results are compared
step by step.

Tolerances (the decode step's floating-point contract): logits within
max-abs 3e-2 of the fp32 oracle; token ids, accept lengths and KV slot
indices bit-exact wherever the oracle's top-1 / top-2 logit margin exceeds
5e-2.  Where a margin is below that, the GPU's choice must still be a valid
one (within 2 x 3e-2 of the oracle's maximum) and the oracle is forced onto
the GPU's tokens (teacher forcing), so later steps compare like with like."""
from __future__ import annotations

import numpy as np

import oracle
import synthetic as S
from oracle import pard as OP
from oracle.philox import STREAM_ACCEPT, STREAM_BONUS, STREAM_DRAFT, raw_words, uniform01

LOGIT_TOL = 3e-2
MARGIN = 5e-2
# Gumbel noise is -log(-log u) on both sides, with different log routines:
# allow a few fp32 ulps of the largest noise values (|G| < 20)
GUMBEL_EPS = 1e-5


def margin(row: np.ndarray) -> float:
    top2 = np.partition(row, -2)[-2:]
    return float(top2[1] - top2[0])


def gumbel_scores(logits_row: np.ndarray, T: float, seed: int, stream: int, step: int, b: int, i: int) -> np.ndarray:
    """The oracle's Gumbel-max scores z / T + G (the categorical draw is their argmax)."""
    z = (np.asarray(logits_row, dtype=np.float32) / np.float32(T)).astype(np.float32)
    return (z + OP.gumbel_noise(seed, stream, step, b, i, z.shape[0])).astype(np.float32)


def check_sampled(gpu_tok: int, scores: np.ndarray, bound: float, stats: dict, what: str) -> None:
    """A Gumbel-max draw: each score of the GPU differs from the oracle's by at
    most bound / 2, so where the oracle's winner leads the runner-up by more
    than bound the GPU must draw the same token; elsewhere its token must
    score within bound of the oracle's winner."""
    o_tok = int(np.argmax(scores))
    stats["sampled_checked"] = stats.get("sampled_checked", 0) + 1
    if margin(scores) > bound:
        assert gpu_tok == o_tok, f"{what}: gpu {gpu_tok} oracle {o_tok} margin {margin(scores):.3g} > {bound:.3g}"
        stats["sampled_exact"] = stats.get("sampled_exact", 0) + 1
    else:
        assert scores[gpu_tok] >= scores[o_tok] - bound, what
        if gpu_tok != o_tok:
            stats["excused_tokens"] += 1


def check_residual_draw(gpu_tok: int, y: np.ndarray, z: np.ndarray, T: float, err_y: float, err_z: float,
                        seed: int, step: int, b: int, stats: dict, what: str) -> None:
    """The bonus token after a rejection: a Gumbel-max draw over
    log max(0, p - q) with Philox stream 2.  With the GPU's logits within
    err_y / err_z of the oracle's, log p_v and log q_v move by at most
    2 err / T, which bounds every GPU weight w_v = max(0, p_v - q_v) to
    [w_v - s_v, w_v + s_v]; the GPU must draw the oracle's winner whenever the
    winner's lowest possible score beats every other entry's highest."""
    p = OP.softmax_t(y, T).astype(np.float64)
    q = OP.softmax_t(z, T).astype(np.float64)
    w = np.maximum(p - q, 0.0)
    if not (w > 0).any():
        return
    slack = p * np.expm1(2 * err_y / T) + q * np.expm1(2 * err_z / T) + 1e-12
    g = OP.gumbel_noise(seed, STREAM_BONUS, step, b, 0, y.shape[0]).astype(np.float64)
    with np.errstate(divide="ignore"):
        score = np.where(w > 0, np.log(w) + g, -np.inf)
        hi = np.log(w + slack) + g
        lo = np.where(w - slack > 0, np.log(np.maximum(w - slack, 1e-300)) + g, -np.inf)
    o_tok = int(np.argmax(score))
    others = hi.copy()
    others[o_tok] = -np.inf
    stats["sampled_checked"] = stats.get("sampled_checked", 0) + 1
    if lo[o_tok] > others.max() + GUMBEL_EPS:
        assert gpu_tok == o_tok, f"{what}: gpu {gpu_tok} oracle {o_tok}"
        stats["sampled_exact"] = stats.get("sampled_exact", 0) + 1
    else:
        assert hi[gpu_tok] + GUMBEL_EPS >= lo[o_tok], what
        if gpu_tok != o_tok:
            stats["excused_tokens"] += 1


class Pair:
    """GPU engine and oracle decoder on identical weights and page orders."""

    def __init__(self, wl, draft_is_target: bool = False, prefill_chunk: int = 64):
        import torch
        from paper_2504_18583_gb300 import pard
        self.wl = wl
        tw = S.model_weights(wl.target, wl.seed, S.TARGET, wl.norm_jitter)
        dw = tw if draft_is_target else S.model_weights(wl.draft, wl.seed, S.DRAFT, wl.norm_jitter)
        dshape = wl.target if draft_is_target else wl.draft
        self.wl = wl = wl.replace(draft=dshape)
        self.tw_host, self.dw_host = tw, dw
        self.prompts = wl.prompts()
        lens = [len(p) for p in self.prompts]
        n_pages = wl.n_pages()
        self.order_t, self.order_d = wl.page_order(S.TARGET), wl.page_order(S.DRAFT)
        self.oracle = oracle.OracleDecoder(wl, tw, dw, self.order_t, self.order_d)
        self.tw_dev = S.device_weights(wl.target, 0, 0, host=tw)
        self.dw_dev = self.tw_dev if draft_is_target else S.device_weights(dshape, 0, 0, host=dw)
        max_ctx = max(lens) + wl.n_new + 2 * wl.K + 16
        self.eng = pard.PardEngine(wl.target, self.tw_dev, dshape, self.dw_dev, max_batch=wl.batch, max_k=wl.K,
                                   max_ctx=max_ctx, n_pages=n_pages, prefill_chunk=prefill_chunk,
                                   page_order_target=self.order_t, page_order_draft=self.order_d)
        self.torch = torch
        self.stats = dict(excused_tokens=0, checked_tokens=0, max_logit_err=0.0, max_draft_logit_err=0.0)

    def prefill(self, seed=0):
        first_g = self.eng.prefill(self.prompts, self.wl.n_new, self.wl.K, self.wl.sample, self.wl.temperature,
                                   seed).cpu().numpy()
        first_o = self.oracle.prefill(self.prompts, seed)
        for b in range(self.wl.batch):
            if not self.wl.sample:
                check_token(int(first_g[b]), self.oracle.prefill_logits[b], self.stats, f"first token seq {b}")
            else:
                # drawn from the target's last prompt row (stream 2, step 0); the
                # GPU's prefill logits are within LOGIT_TOL of the oracle's
                T = self.wl.temperature
                sc = gumbel_scores(self.oracle.prefill_logits[b], T, seed, STREAM_BONUS, 0, b, 0)
                check_sampled(int(first_g[b]), sc, 2 * LOGIT_TOL / T + GUMBEL_EPS, self.stats,
                              f"sampled first token seq {b}")
            if int(first_g[b]) != int(first_o[b]):
                self.stats["excused_tokens"] += 1
                self.oracle.force_first(b, int(first_g[b]))
        return first_g, first_o

    def active(self):
        return [b for b in range(self.wl.batch) if not self.oracle.done[b]]


def check_token(gpu_tok: int, oracle_logits: np.ndarray, stats: dict, what: str) -> None:
    """Bit-exact where the margin is clear; otherwise the GPU's token must be
    within 2 x LOGIT_TOL of the oracle's maximum."""
    o_tok = int(np.argmax(oracle_logits))
    stats["checked_tokens"] += 1
    if margin(oracle_logits) > MARGIN:
        assert gpu_tok == o_tok, f"{what}: gpu {gpu_tok} oracle {o_tok} margin {margin(oracle_logits):.3g}"
    else:
        assert oracle_logits[gpu_tok] >= oracle_logits[o_tok] - 2 * LOGIT_TOL, what
        if gpu_tok != o_tok:
            stats["excused_tokens"] += 1


def greedy_step(P: Pair, step: int, inject=None, sequential: bool = False):
    """One teacher-forced greedy step; returns the GPU outputs.  sequential:
    vanilla speculative decoding's K-pass draft on both sides."""
    torch = P.torch
    wl, K = P.wl, P.wl.K
    out = P.eng.alloc_step_outputs(want_logits=True)
    if sequential:
        P.eng.draft_sequential(out, False, 1.0, 0, step)
    else:
        P.eng.draft(out, False, 1.0, 0, step)
    d_gpu = out["draft"].cpu().numpy()
    z_gpu = out["draft_logits"].cpu().numpy()
    # the sequential draft feeds each candidate to the next pass: the oracle
    # is fed the GPU's (teacher forcing), so near-tie choices do not diverge
    d_or, z_or = P.oracle.draft_sequential(step, feed=d_gpu) if sequential else P.oracle.draft(step)
    for b in P.active():
        err = float(np.abs(z_gpu[b] - z_or[b]).max())
        P.stats["max_draft_logit_err"] = max(P.stats["max_draft_logit_err"], err)
        assert err <= LOGIT_TOL, f"draft logits step {step} seq {b}: {err}"
        for i in range(K):
            check_token(int(d_gpu[b, i]), z_or[b, i], P.stats, f"draft step {step} seq {b} i {i}")
    cand = d_gpu if inject is None else inject
    cand_t = None if inject is None else torch.as_tensor(inject, dtype=torch.int32, device="cuda")
    P.eng.verify(out, cand_t, 1.0)
    y_gpu = out["logits"].cpu().numpy()
    y_or = P.oracle.verify(cand)
    for b in P.active():
        err = float(np.abs(y_gpu[b] - y_or[b]).max())
        P.stats["max_logit_err"] = max(P.stats["max_logit_err"], err)
        assert err <= LOGIT_TOL, f"verify logits step {step} seq {b}: {err}"
    P.eng.accept_commit(out, False, 1.0, 0, step)
    a_gpu = out["accept_len"].cpu().numpy()
    em_gpu = out["emitted"].cpu().numpy()
    slots_gpu = out["kv_slots"].cpu().numpy()
    n_emit = out["n_emit"].cpu().numpy()
    acc, emitted = [], []
    for b in range(wl.batch):
        if P.oracle.done[b]:
            assert a_gpu[b] == 0 and n_emit[b] == 0 and (em_gpu[b] == -1).all()
            acc.append(0)
            emitted.append([])
            continue
        a = int(a_gpu[b])
        t_gpu = [int(np.argmax(y_gpu[b, i])) for i in range(K + 1)]
        for i in range(K + 1):
            check_token(t_gpu[i], y_or[b, i], P.stats, f"verify step {step} seq {b} row {i}")
        # the accept kernel applies the prefix rule exactly to the GPU's own argmax
        a_rule = 0
        while a_rule < K and int(cand[b, a_rule]) == t_gpu[a_rule]:
            a_rule += 1
        assert a == a_rule, f"accept length {a} != prefix rule {a_rule}"
        a_or, em_or = OP.accept_greedy(cand[b], y_or[b])
        if a_or != a:
            # only allowed when the deciding row's margin is within tolerance
            i = min(a, a_or)
            assert margin(y_or[b, i]) <= MARGIN, f"accept length step {step} seq {b}: gpu {a} oracle {a_or}"
            P.stats["excused_tokens"] += 1
        gpu_em = [int(x) for x in cand[b, :a]] + [int(np.argmax(y_gpu[b, a]))]
        take = int(n_emit[b])
        assert [int(x) for x in em_gpu[b, :take]] == gpu_em[:take]
        assert (em_gpu[b, take:] == -1).all()
        acc.append(a)
        emitted.append(gpu_em)
    slots_or, nout = P.oracle.commit(acc, emitted)
    for b in range(wl.batch):
        if b < len(nout) and nout[b] == 0 and a_gpu[b] == 0 and n_emit[b] == 0:
            continue
        assert np.array_equal(slots_gpu[b], slots_or[b]), f"kv slots step {step} seq {b}"
        assert n_emit[b] == nout[b]
    return dict(a=a_gpu, emitted=em_gpu, slots=slots_gpu, d=d_gpu, y=y_gpu, z=z_gpu)


def sampling_step(P: Pair, step: int, seed: int, sequential: bool = False) -> dict:
    """One teacher-forced speculative-sampling step (Section 2.2 with the
    draft of Eq. 6 at temperature T; sequential: vanilla speculative
    decoding's K-pass draft, the oracle fed the GPU's candidates between
    passes): draft logits, verify logits within LOGIT_TOL; the draft's
    Gumbel-max candidates, the accept / reject decisions and the bonus draw
    against the oracle's on the same Philox streams wherever the margins are
    clear; KV slots bit-exact.  The oracle is then committed with the GPU's
    tokens."""
    wl, K, T = P.wl, P.wl.K, P.wl.temperature
    out = P.eng.alloc_step_outputs(want_logits=True)
    if sequential:
        P.eng.draft_sequential(out, True, T, seed, step)
    else:
        P.eng.draft(out, True, T, seed, step)
    d_g = out["draft"].cpu().numpy()
    z_g = out["draft_logits"].cpu().numpy()
    d_o, z_o = P.oracle.draft_sequential(step, seed, feed=d_g) if sequential else P.oracle.draft(step, seed)
    for b in P.active():
        for i in range(K):
            err = float(np.abs(z_g[b, i] - z_o[b, i]).max())
            P.stats["max_draft_logit_err"] = max(P.stats["max_draft_logit_err"], err)
            assert err <= LOGIT_TOL, f"draft logits step {step} seq {b} row {i}: {err}"
            sc = gumbel_scores(z_o[b, i], T, seed, STREAM_DRAFT, step, b, i)
            assert int(d_o[b, i]) == int(np.argmax(sc))
            check_sampled(int(d_g[b, i]), sc, 2 * err / T + GUMBEL_EPS, P.stats,
                          f"sampled draft step {step} seq {b} row {i}")
    P.eng.verify(out, None, T)
    y_g = out["logits"].cpu().numpy()
    y_o = P.oracle.verify(d_g)
    for b in P.active():
        err = float(np.abs(y_g[b] - y_o[b]).max())
        P.stats["max_logit_err"] = max(P.stats["max_logit_err"], err)
        assert err <= LOGIT_TOL, f"verify logits step {step} seq {b}: {err}"
    P.eng.accept_commit(out, True, T, seed, step)
    a_g = out["accept_len"].cpu().numpy()
    em_g = out["emitted"].cpu().numpy()
    n_emit = out["n_emit"].cpu().numpy()
    slots_g = out["kv_slots"].cpu().numpy()
    acc, emitted = [], []
    for b in range(wl.batch):
        if P.oracle.done[b]:
            assert a_g[b] == 0 and n_emit[b] == 0
            acc.append(0)
            emitted.append([])
            continue
        a = int(a_g[b])
        for i in range(min(a + 1, K)):
            p = OP.softmax_t(y_o[b, i], T)[d_g[b, i]]
            q = OP.softmax_t(z_o[b, i], T)[d_g[b, i]]
            u = uniform01(raw_words(seed, STREAM_ACCEPT, step, b, i, np.zeros(1, np.uint64)))[0]
            if abs(u - p / q) > 1e-3:
                assert (u * q < p) == (i < a), (step, b, i)
                P.stats["decisions_checked"] = P.stats.get("decisions_checked", 0) + 1
        take = int(n_emit[b])
        em = [int(x) for x in em_g[b, :take]]
        assert em[:min(a, take)] == [int(x) for x in d_g[b, :min(a, take)]]
        a_o, _ = OP.accept_sampling(d_g[b], z_o[b], y_o[b], T, seed, step, b)
        if a_o == a and take == a + 1:
            err_y = float(np.abs(y_g[b, a] - y_o[b, a]).max())
            if a == K:
                sc = gumbel_scores(y_o[b, K], T, seed, STREAM_BONUS, step, b, 0)
                check_sampled(em[a], sc, 2 * err_y / T + GUMBEL_EPS, P.stats, f"bonus p_K step {step} seq {b}")
            else:
                err_z = float(np.abs(z_g[b, a] - z_o[b, a]).max())
                check_residual_draw(em[a], y_o[b, a], z_o[b, a], T, err_y, err_z, seed, step, b, P.stats,
                                    f"residual draw step {step} seq {b} row {a}")
        full = em if len(em) == a + 1 else em + [0] * (a + 1 - len(em))
        acc.append(a)
        emitted.append(full)
    slots_o, nout = P.oracle.commit(acc, emitted)
    for b in range(wl.batch):
        if nout[b] == 0 and a_g[b] == 0 and n_emit[b] == 0:
            continue
        assert np.array_equal(slots_g[b], slots_o[b]), f"kv slots step {step} seq {b}"
        assert n_emit[b] == nout[b]
    return dict(a=a_g, emitted=em_g, d=d_g)
