"""Pins for the CPU oracle: checks against closed forms, library routines,
published known-answer vectors and invariants the paper's method fixes.
None of these re-types the oracle's own formulas."""
import os

import numpy as np
import pytest

import oracle
import synthetic as S
from oracle import pard as P
from oracle.philox import philox4x32_10, raw_words, uniform01, uniform_open01

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# Philox: published known-answer vectors
# --------------------------------------------------------------------------
def test_philox_known_answer_vectors():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = philox4x32_10(v[0:4], v[4:6])
        assert [int(o) for o in out] == v[6:10]


def test_uniform_maps_are_exact_and_in_range():
    x = np.array([0, 0xFF, 0x100, 0xFFFFFFFF], dtype=np.uint32)
    u = uniform01(x)
    assert u[0] == 0.0 and u[1] == 0.0 and u[2] == np.float32(2.0 ** -24)
    assert u[3] == np.float32(1.0 - 2.0 ** -24)
    uo = uniform_open01(x)
    assert uo[0] == np.float32(0.5 * 2.0 ** -23) and uo[3] == np.float32(1.0 - 2.0 ** -24)


def test_philox_streams_are_distinct():
    a = raw_words(7, 0, 1, 0, 0, np.arange(64, dtype=np.uint64))
    b = raw_words(7, 1, 1, 0, 0, np.arange(64, dtype=np.uint64))
    c = raw_words(7, 0, 2, 0, 0, np.arange(64, dtype=np.uint64))
    assert len(set(a.tolist())) == 64
    assert not np.array_equal(a, b) and not np.array_equal(a, c)


# --------------------------------------------------------------------------
# Primitives: closed forms and library routines
# --------------------------------------------------------------------------
def test_rope_closed_forms():
    v = np.arange(1, 9, dtype=np.float32)
    assert np.array_equal(oracle.rope(v, 0, 10000.0), v)           # position 0: identity
    # hd = 2: one pair, inverse frequency 1, so the pair rotates by `pos` radians
    r = oracle.rope(np.array([1.0, 0.0], np.float32), 1, 10000.0)
    assert np.allclose(r, [np.cos(1.0), np.sin(1.0)], atol=1e-7)
    r = oracle.rope(np.array([0.0, 2.0], np.float32), 3, 500000.0)
    assert np.allclose(r, [-2 * np.sin(3.0), 2 * np.cos(3.0)], atol=1e-6)
    # rotation preserves the norm; scores depend on the position difference only
    rng = np.random.default_rng(0)
    q, k = rng.standard_normal(128).astype(np.float32), rng.standard_normal(128).astype(np.float32)
    assert np.isclose(np.linalg.norm(oracle.rope(q, 777, 5e5)), np.linalg.norm(q), rtol=1e-5)
    s1 = oracle.rope(q, 5, 1e4) @ oracle.rope(k, 2, 1e4)
    s2 = oracle.rope(q, 1003, 1e4) @ oracle.rope(k, 1000, 1e4)
    assert np.isclose(s1, s2, rtol=2e-4, atol=2e-4)
    # the rotate-half pairing matches a complex rotation of (x_j, x_{j+hd/2})
    hd, pos, theta = 64, 41, 10000.0
    x = rng.standard_normal(hd).astype(np.float32)
    j = np.arange(hd // 2)
    c = (x[: hd // 2] + 1j * x[hd // 2:]) * np.exp(1j * pos * theta ** (-2.0 * j / hd))
    assert np.allclose(oracle.rope(x, pos, theta), np.concatenate([c.real, c.imag]), atol=2e-5)


def test_rmsnorm_closed_form():
    g = S.f32_to_bf16(np.array([1.0, 2.0], np.float32))
    out = oracle.rmsnorm(np.array([[3.0, 4.0]], np.float32), g, 1e-5)
    r = 1.0 / np.sqrt(12.5 + 1e-5)
    assert np.allclose(out, [[3 * r, 8 * r]], rtol=1e-6)


def test_matmul_matches_float64_library_product():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, 200)).astype(np.float32)
    wb = S.f32_to_bf16(rng.standard_normal((37, 200)).astype(np.float32) * 0.02)
    ref = x.astype(np.float64) @ S.bf16_to_f32(wb).astype(np.float64).T
    got = oracle.matmul(x, wb)
    assert np.allclose(got, ref, rtol=1e-5, atol=1e-5)
    cols = np.array([36, 0, 17], np.int32)
    assert np.array_equal(oracle.matmul_cols(x, wb, cols), got[:, cols])


def test_attention_closed_forms_and_library():
    import torch
    import torch.nn.functional as F
    rng = np.random.default_rng(2)
    hkv, hd, L = 2, 16, 9
    kc = rng.standard_normal((L, hkv, hd)).astype(np.float32)
    vc = rng.standard_normal((L, hkv, hd)).astype(np.float32)
    q = rng.standard_normal(hd).astype(np.float32)
    # a single visible key: the output is that key's value row
    assert np.array_equal(oracle.attend(q, kc, vc, 1, 0), vc[0, 1])
    # identical keys: uniform weights, the output is the mean value row
    kc2 = np.repeat(kc[:1], L, axis=0)
    assert np.allclose(oracle.attend(q, kc2, vc, 0, L - 1), vc[:, 0].mean(0), atol=1e-6)
    # library routine (float64 scaled-dot-product attention)
    ref = F.scaled_dot_product_attention(torch.from_numpy(q).double()[None, None],
                                         torch.from_numpy(kc[:7, 1]).double()[None],
                                         torch.from_numpy(vc[:7, 1]).double()[None])[0, 0].numpy()
    assert np.allclose(oracle.attend(q, kc, vc, 1, 6), ref, atol=2e-6)


# --------------------------------------------------------------------------
# Whole model against an independent float64 build from torch library routines
# --------------------------------------------------------------------------
def torch_llama_logits(shape, w, tokens):
    """Full-sequence causal forward from library routines: F.rms_norm,
    complex-number RoPE, F.scaled_dot_product_attention with GQA expansion
    by repeat_interleave, F.silu.  Returns float64 logits for every row."""
    import torch
    import torch.nn.functional as F
    f = lambda bits: torch.from_numpy(S.bf16_to_f32(bits)).double()
    d, hq, hkv, hd = shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim
    T = len(tokens)
    h = f(w["embed"])[torch.as_tensor(np.asarray(tokens, np.int64))]
    j = torch.arange(hd // 2, dtype=torch.float64)
    ang = torch.arange(T, dtype=torch.float64)[:, None] * shape.rope_theta ** (-2.0 * j / hd)
    rot = torch.polar(torch.ones_like(ang), ang)

    def rope(t):
        c = torch.complex(t[..., : hd // 2], t[..., hd // 2:]) * rot[:, None, :]
        return torch.cat([c.real, c.imag], dim=-1)

    for L in w["layers"]:
        x = F.rms_norm(h, (d,), weight=f(L["attn_norm"]), eps=shape.rms_eps)
        q = rope((x @ f(L["wq"]).T).view(T, hq, hd))
        k = rope((x @ f(L["wk"]).T).view(T, hkv, hd))
        v = (x @ f(L["wv"]).T).view(T, hkv, hd)
        k = k.repeat_interleave(hq // hkv, dim=1)
        v = v.repeat_interleave(hq // hkv, dim=1)
        o = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                           is_causal=True).transpose(0, 1).reshape(T, hq * hd)
        h = h + o @ f(L["wo"]).T
        x = F.rms_norm(h, (d,), weight=f(L["mlp_norm"]), eps=shape.rms_eps)
        h = h + (F.silu(x @ f(L["wg"]).T) * (x @ f(L["wu"]).T)) @ f(L["wd"]).T
    x = F.rms_norm(h, (d,), weight=f(w["final_norm"]), eps=shape.rms_eps)
    return (x @ f(w["lm_head"]).T).numpy()


@pytest.fixture(scope="module")
def tiny():
    wl = S.WORKLOADS["tiny"].replace(norm_jitter=0.1)
    tw, dw = S.workload_weights(wl)
    return wl, tw, dw


def test_forward_matches_library_model_prefill_and_incremental(tiny):
    wl, tw, _ = tiny
    toks = wl.prompts()[0].tolist() + [5, 77, 2047, 1000]
    ref = torch_llama_logits(wl.target, tw, toks)
    m = P.OracleModel(wl.target, tw, 1, 64, kv_bf16=False)
    P0 = 32
    pre = m.forward(0, toks[:P0], list(range(P0)), list(range(P0)))
    assert np.abs(pre - ref[:P0]).max() < 2e-4
    # one row at a time on top of the cache, then a 2-row chunk
    r1 = m.forward(0, toks[P0:P0 + 1], [P0], [0])
    r2 = m.forward(0, toks[P0 + 1:P0 + 2], [P0 + 1], [0])
    r3 = m.forward(0, toks[P0 + 2:], [P0 + 2, P0 + 3], [0, 1])
    inc = np.concatenate([r1, r2, r3])
    assert np.abs(inc - ref[P0:]).max() < 2e-4
    assert np.abs(ref).max() > 0.5                # not a degenerate all-zero model


def test_bf16_cache_stores_rounded_fp32_values(tiny):
    """With the bf16 cache, every stored key/value is the round-to-nearest-even
    bf16 value of the fp32 one, and logits stay within bf16-storage error."""
    wl, tw, _ = tiny
    toks = wl.prompts()[0].tolist()
    a = P.OracleModel(wl.target, tw, 1, 40, kv_bf16=False)
    b = P.OracleModel(wl.target, tw, 1, 40, kv_bf16=True)
    la = a.forward(0, toks[:1], [0], [0])
    lb = b.forward(0, toks[:1], [0], [0])
    # one row: attention reads only its own key/value, so layer 0's cache entry is comparable exactly
    k32 = a.kc[0][0, 0].astype(np.float32)
    u = k32.view(np.uint32).astype(np.uint64)
    rne = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16 << 16).astype(np.uint32).view(np.float32)
    assert np.array_equal(b.kc[0][0, 0], rne)
    assert np.abs(la - lb).max() < 0.05 * np.abs(la).max()
    la = a.forward(0, toks[1:], range(1, len(toks)), range(len(toks) - 1))
    lb = b.forward(0, toks[1:], range(1, len(toks)), range(len(toks) - 1))
    assert 0 < np.abs(la - lb).max() < 0.05 * np.abs(la).max()


def test_forward_rejects_bad_arguments(tiny):
    wl, tw, _ = tiny
    m = P.OracleModel(wl.target, tw, 1, 8)
    with pytest.raises(ValueError):
        m.forward(0, [1], [8], [0])
    with pytest.raises(ValueError):
        m.forward(0, [wl.target.vocab], [0], [0])


# --------------------------------------------------------------------------
# Invariants of the method
# --------------------------------------------------------------------------
def test_rows_are_batch_invariant(tiny):
    wl, tw, _ = tiny
    pr = wl.prompts()[0]
    a = P.OracleModel(wl.target, tw, 1, 64)
    b = P.OracleModel(wl.target, tw, 1, 64)
    a.forward(0, pr, range(32), [])
    b.forward(0, pr, range(32), [])
    new = [11, 22, 33, 44, 55]
    together = a.forward(0, new, range(32, 37), range(5))
    alone = np.concatenate([b.forward(0, [t], [32 + i], [0]) for i, t in enumerate(new)])
    assert np.array_equal(together, alone)


def test_extra_mask_changes_no_earlier_row(tiny):
    """Eq. 6 with K-1 masks == the same pass with K masks, first K rows."""
    wl, _, dw = tiny
    pr = wl.prompts()[0]
    K, mask = wl.K, wl.draft.mask_id
    outs = []
    for extra in (0, 1):
        m = P.OracleModel(wl.draft, dw, 1, 64)
        m.forward(0, pr[:-1], range(31), [])
        rows = [int(pr[-1])] + [mask] * (K - 1 + extra)
        outs.append(m.forward(0, rows, range(31, 31 + len(rows)), range(K)))
    assert np.array_equal(outs[0], outs[1])


def _greedy_equivalence(wl, tw, dw, sequential=False):
    pr = wl.prompts()
    dec = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    gen, trace = dec.run(pr, sequential=sequential)
    for b in range(wl.batch):
        assert gen[b] == oracle.ar_greedy(wl.target, tw, pr[b], wl.n_new)
    return trace


def test_pard_greedy_equals_autoregressive_greedy(tiny):
    wl, tw, dw = tiny
    _greedy_equivalence(wl, tw, dw)


def test_pard_greedy_equals_ar_with_accepting_draft(tiny):
    """Draft = the target's weights: d_0 is always the target's argmax, so
    every step accepts >= 1 token and exercises commit/rollback with a > 0."""
    wl, tw, _ = tiny
    wl = wl.replace(draft=wl.target, n_new=24, batch=2)
    trace = _greedy_equivalence(wl, tw, tw)
    accs = [a for t in trace for a in t["acc"]]
    assert min(accs[:len(trace)]) >= 1 and max(accs) >= 1


def test_vanilla_sd_greedy_equals_autoregressive_greedy(tiny):
    """Vanilla speculative decoding (K sequential draft passes) is lossless
    too: greedy output equals the target's autoregressive greedy decode."""
    wl, tw, dw = tiny
    _greedy_equivalence(wl, tw, dw, sequential=True)


def test_vanilla_sd_candidates_are_the_drafts_own_greedy_continuation(tiny):
    """Greedy vanilla SD's candidates are the draft model's autoregressive
    greedy continuation of the accepted prefix (Section 3.1's factorization),
    here checked against Eq. 2 run on the draft model alone; and with the
    target as its own draft every candidate is accepted."""
    wl, tw, dw = tiny
    pr = wl.prompts()
    dec = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    first = dec.prefill(pr)
    d, _ = dec.draft_sequential(1)
    for b in range(wl.batch):
        cont = oracle.ar_greedy(wl.draft, dw, list(pr[b]) + [first[b]], wl.K)
        assert [int(x) for x in d[b]] == cont
    wl2 = wl.replace(draft=wl.target, n_new=20, batch=1)
    trace = _greedy_equivalence(wl2, tw, tw, sequential=True)
    assert all(a == wl2.K for t in trace[:-1] for a in t["acc"])


def test_distinct_mask_ids_keep_pard_lossless_and_reach_the_draft(tiny):
    """One mask id per offset (Section 4.3's alternative to the shared id):
    greedy PARD still equals autoregressive greedy decoding, K = 12 (verify
    13 rows, draft up to 24); and the mask rows' logits are the draft model's
    forward over exactly those ids (they differ from the shared-id ones)."""
    wl, tw, dw = tiny
    wl = wl.replace(K=12, n_new=20, batch=2)
    V = wl.draft.vocab
    ids = [V - 2 - k for k in range(wl.K - 1)]
    pr = wl.prompts()
    dec = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    dec.mask_ids = ids
    gen, _ = dec.run(pr)
    for b in range(wl.batch):
        assert gen[b] == oracle.ar_greedy(wl.target, tw, pr[b], wl.n_new)
    dec2 = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    first = dec2.prefill(pr)
    dec2.mask_ids = ids
    _, z = dec2.draft(1)
    m = P.OracleModel(wl.draft, dw, 1, 128)
    P0 = len(pr[0])
    m.forward(0, pr[0], range(P0), [])
    ref = m.forward(0, [first[0]] + ids, range(P0, P0 + wl.K), range(wl.K))
    assert np.array_equal(z[0], ref)
    dec3 = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    dec3.prefill(pr)
    _, z_shared = dec3.draft(1)
    assert np.array_equal(z_shared[0, 0], z[0, 0]) and not np.array_equal(z_shared[0, 1:], z[0, 1:])


# --------------------------------------------------------------------------
# COD data construction (Section 3.2, appendix algorithm and worked example)
# --------------------------------------------------------------------------
def test_cod_worked_example_from_the_paper():
    """The appendix example (tests/golden/cod_worked_example.txt): with the
    example's choice at +2, the +3 candidates, the number kept and the
    contexts and labels of m_{1,2} and m_{1,3} are the ones the paper states."""
    from oracle import cod
    g = {}
    for line in open(os.path.join(GOLDEN, "cod_worked_example.txt")):
        if line.strip() and not line.startswith("#"):
            key, *vals = line.split()
            g[key] = vals
    words = g["tokens"]
    ids = {w: 10 + i for i, w in enumerate(words)}
    toks = [ids[w] for w in words]
    N, K, r = len(toks) - 1, int(g["K"][0]), float(g["r"][0])
    masks = [900, 901]
    mask_name = {900: "m0", 901: "m1"}
    kept_2 = [int(x) for x in g["kept_2"]]
    assert cod.retained_count(N, 2, r, 0.0) == len(kept_2)
    assert cod.retained_count(N, 3, r, 0.0) == int(g["n_kept_3"][0])
    keep, counts = cod.cod_select(N, K, r, 0.0, seed=1, sample_id=0, forced=[kept_2])
    assert cod.candidates(keep, 3, N) == [int(x) for x in g["candidates_3"]]
    assert counts == [N, len(kept_2), int(g["n_kept_3"][0])]
    for j in (int(x) for x in g["candidates_3"]):
        keep, _ = cod.cod_select(N, K, r, 0.0, seed=1, sample_id=0, forced=[kept_2, [j]])
        rows = cod.packed_rows(toks, keep, masks)
        k3 = [row for row in rows if row[0] == 3][0]
        real_words = [words[toks.index(rows[i][1])] for i in range(k3[5])]
        chain, at = [], k3[4]
        while at >= 0:
            chain.append("%s%d" % (mask_name[rows[at][1]], rows[at][2]))
            at = rows[at][4]
        ctx = " ".join(real_words) + " | " + " ".join(reversed(chain))
        assert ctx == " ".join(g["context_m1%d" % j]), (ctx, j)
        assert words[toks.index(k3[3])] == g["label_m1%d" % j][0]


def test_cod_counts_follow_the_geometric_retention():
    """N_k = N max(r^(k-1), r_min) per subtask (Section 3.2); with r_min = 0
    the total is N (1 - r^K) / (1 - r) up to the per-subtask rounding."""
    from oracle import cod
    N, K = 1000, 6
    for r, r_min in ((0.5, 0.0), (0.7, 0.0), (0.5, 0.2)):
        _, counts = cod.cod_select(N, K, r, r_min, seed=5, sample_id=3)
        for k in range(1, K + 1):
            assert counts[k - 1] == int(np.floor(N * max(r ** (k - 1), r_min) + 0.5)), (r, r_min, k)
        if r_min == 0.0:
            assert abs(sum(counts) - N * (1 - r ** K) / (1 - r)) <= K


def test_cod_every_kept_row_has_its_whole_context():
    """Integrity of prefix key-value states: every kept row of subtask k >= 3
    has its predecessor chain down to subtask 2 kept; r = 1 keeps every row
    (plain mask-token training)."""
    from oracle import cod
    rng = np.random.default_rng(7)
    for t in range(30):
        N, K = int(rng.integers(1, 60)), int(rng.integers(2, 9))
        r, r_min = float(rng.uniform(0.2, 1.0)), float(rng.uniform(0.0, 0.3))
        keep, counts = cod.cod_select(N, K, r, r_min, seed=t, sample_id=t)
        for k in range(3, K + 1):
            for j in range(N):
                if keep[k - 2, j]:
                    assert j >= k - 2 and all(keep[kk - 2, j - (k - kk)] for kk in range(2, k))
        assert counts == [N] + [int(keep[k - 2].sum()) for k in range(2, K + 1)]
    keep, _ = cod.cod_select(20, 5, 1.0, 0.0, seed=1, sample_id=1)
    for k in range(2, 6):
        assert keep[k - 2].tolist() == [0] * (k - 2) + [1] * (20 - k + 2)


def test_cod_choice_is_uniform_over_candidates():
    """The random choice of subtask 2 keeps each position with probability
    n / N: chi-square over 400 samples, N = 10, n = 5."""
    from oracle import cod
    hits = np.zeros(10)
    S_ = 400
    for sid in range(S_):
        keep, _ = cod.cod_select(10, 2, 0.5, 0.0, seed=11, sample_id=sid)
        hits += keep[0]
    exp = S_ * 0.5
    chi2 = float((((hits - exp) ** 2) / exp).sum())
    assert chi2 < 27.9  # 9 degrees of freedom, p = 0.001


def test_rollback_then_recompute_gives_identical_cache_values(tiny):
    """Rollback is by length only: after rows at positions p..p+2 are written
    and the last is rejected, feeding another token at p+2 and then the
    original one again rewrites exactly the first values (rows do not depend
    on what was written past them)."""
    wl, tw, _ = tiny
    pr = wl.prompts()[0].tolist()
    P0 = len(pr)
    m = P.OracleModel(wl.target, tw, 1, 64)
    m.forward(0, pr, range(P0), [])
    m.forward(0, [5, 77, 300], [P0, P0 + 1, P0 + 2], [])
    k1, v1 = m.kc[0][:, :P0 + 3].copy(), m.vc[0][:, :P0 + 3].copy()
    m.forward(0, [1999], [P0 + 2], [])
    assert not np.array_equal(m.kc[0][:, P0 + 2], k1[:, P0 + 2])
    m.forward(0, [300], [P0 + 2], [])
    assert np.array_equal(m.kc[0][:, :P0 + 3], k1) and np.array_equal(m.vc[0][:, :P0 + 3], v1)


def test_greedy_accept_rule_every_length():
    rng = np.random.default_rng(3)
    K, V = 5, 11
    y = rng.standard_normal((K + 1, V)).astype(np.float32)
    t = y.argmax(1)
    for j in range(K + 1):
        d = t[:K].copy()
        if j < K:
            d[j] = (d[j] + 1) % V
        a, em = P.accept_greedy(d, y)
        assert a == j and em == list(t[:j]) + [int(t[j])]


def test_commit_slots_follow_page_table(tiny):
    wl, tw, dw = tiny
    dec = oracle.OracleDecoder(wl, tw, dw, wl.page_order(0), wl.page_order(1))
    dec.prefill(wl.prompts())
    n = dec.n[0]
    slots, _ = dec.commit([2], [[1, 2, 3]])
    tbl = dec.table_t[0]
    for j in range(3):
        pos = n - 1 + j
        assert slots[0, j] == tbl[pos // 16] * 16 + pos % 16
    assert (slots[0, 3:] == -1).all() and dec.n[0] == n + 3 and dec.pending[0] == [1, 2, 3]


# --------------------------------------------------------------------------
# Speculative sampling reproduces the target distribution
# --------------------------------------------------------------------------
def _chi2_p(counts, probs):
    from scipy.stats import chisquare
    exp = probs / probs.sum() * counts.sum()
    keep = exp > 0
    assert counts[~keep].sum() == 0
    return chisquare(counts[keep], exp[keep]).pvalue


def test_gumbel_max_sampler_matches_softmax():
    scores = np.array([0.3, -1.0, 2.0, 0.0, 0.5, -0.2, 1.1, -3.0], np.float32)
    n = 20000
    counts = np.zeros(8)
    for s in range(n):
        counts[P.sample_gumbel_max(scores, 1234 + s, 2, 0, 0, 0)] += 1
    assert _chi2_p(counts, P.softmax_t(scores, 1.0).astype(np.float64)) > 1e-3


def test_speculative_sampling_is_lossless():
    """V=8, K=3, fixed per-position target/draft logits: the token emitted at
    position i (accepted draft, residual draw or bonus) is distributed as
    p_i = softmax(y_i / T), whatever q is."""
    rng = np.random.default_rng(4)
    V, K, T = 8, 3, 1.0
    y = rng.standard_normal((K + 1, V)).astype(np.float32) * 1.5
    z = (y[:K] + rng.standard_normal((K, V)).astype(np.float32) * 0.8).astype(np.float32)
    n = 30000
    counts = np.zeros((K + 1, V))
    acc_hist = np.zeros(K + 1)
    for s in range(n):
        seed = 99991 * s + 7
        d = P.draft_tokens(z, True, T, seed, 1, 0)
        a, em = P.accept_sampling(d, z, y, T, seed, 1, 0)
        acc_hist[a] += 1
        for i, tok in enumerate(em):
            counts[i, tok] += 1
    for i in range(K + 1):
        assert counts[i].sum() > 300
        assert _chi2_p(counts[i], P.softmax_t(y[i], T).astype(np.float64)) > 1e-3, i
    # the acceptance rate of position 0 is sum_v min(p, q)
    p0, q0 = P.softmax_t(y[0], T), P.softmax_t(z[0], T)
    rate = 1 - acc_hist[0] / n
    assert abs(rate - np.minimum(p0, q0).sum()) < 0.02


def test_sampling_with_identical_draft_accepts_everything():
    rng = np.random.default_rng(5)
    y = rng.standard_normal((4, 16)).astype(np.float32)
    for s in range(50):
        d = P.draft_tokens(y[:3], True, 1.0, s, 3, 0)
        a, em = P.accept_sampling(d, y[:3], y, 1.0, s, 3, 0)
        assert a == 3 and em[:3] == d


# --------------------------------------------------------------------------
# Byte model against the paper's printed draft traffic
# --------------------------------------------------------------------------
def test_draft_bytes_match_paper_table():
    vals = {l.split()[0]: l.split()[1:] for l in open(os.path.join(GOLDEN, "paper_numbers.txt"))
            if l.strip() and not l.startswith("#")}
    gb, tol = float(vals["draft_bytes_gb_1b"][0]), float(vals["draft_bytes_gb_1b"][1])
    assert abs(S.DRAFT_1B.streamed_weight_bytes() / 1e9 - gb) <= tol
