"""GPU parity of the PARD decode step against the CPU oracle, through the
C ABI.  Every test builds both sides from the same seeded inputs."""
import numpy as np
import pytest

import oracle
import synthetic as S
from oracle import pard as OP
from oracle.philox import STREAM_ACCEPT, STREAM_BONUS, STREAM_DRAFT, raw_words, uniform01

from _parity import GUMBEL_EPS, LOGIT_TOL, MARGIN, Pair, check_token, greedy_step, gumbel_scores, margin, sampling_step

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2504_18583_gb300 import _build
    _build.build()


def run_greedy(P: Pair, max_steps=64, inject_fn=None, sequential=False):
    P.prefill()
    step = 1
    outs = []
    while not P.oracle.all_done() and step <= max_steps:
        inject = inject_fn(P, step) if inject_fn else None
        outs.append(greedy_step(P, step, inject, sequential))
        step += 1
    n, gen, done = P.eng.state()
    assert done == [1 if d else 0 for d in P.oracle.done]
    assert P.eng.last_status() == 0
    return outs


def test_tiny_greedy_matches_oracle_every_step():
    """The tiny configuration (FFN 688: ragged row-major gate/up/down tiles)
    against the oracle step by step; and with FFN 768, where every matrix
    takes the packed layout."""
    for ffn in (688, 768):
        wl = S.WORKLOADS["tiny"]
        wl = wl.replace(target=wl.target.replace(ffn=ffn), draft=wl.draft.replace(ffn=ffn))
        P = Pair(wl)
        run_greedy(P)
        assert P.oracle.all_done()
        # the generated sequence equals autoregressive greedy decoding where margins are clear
        assert P.stats["excused_tokens"] <= P.stats["checked_tokens"] // 10
        print("ffn", ffn, "stats", P.stats)


def test_vanilla_sd_sequential_draft_matches_oracle_every_step():
    """Vanilla speculative decoding (K sequential draft passes, Section 2.2)
    on the same kernels: draft logits, candidates, accept lengths and slots
    against the oracle's sequential draft, batch 2, ragged prompts; with the
    target as its own draft every candidate but the last step's is accepted."""
    wl = S.WORKLOADS["tiny"].replace(batch=2, prompt_len=None, prompt_len_range=(20, 45), n_new=24)
    P = Pair(wl)
    run_greedy(P, sequential=True)
    assert P.oracle.all_done()
    print("stats", P.stats)
    wl2 = S.WORKLOADS["tiny"].replace(n_new=20, prompt_len=30)
    P2 = Pair(wl2, draft_is_target=True)
    outs = run_greedy(P2, sequential=True)
    accs = [int(o["a"][0]) for o in outs]
    assert max(accs) == wl2.K
    print("accept lengths", accs, P2.stats)


def test_distinct_mask_ids_and_k12_match_oracle_every_step():
    """One mask id per offset (Section 4.3's alternative to the shared id)
    and K = 12 (verify 13 rows, draft up to 24 rows per sequence: two
    attention row blocks), batch 2, against the oracle step by step; the
    argument and state checks of pard_set_mask_ids."""
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["tiny"].replace(K=12, batch=2, n_new=24, prompt_len=None, prompt_len_range=(20, 45))
    V = wl.draft.vocab
    ids = [V - 2 - k for k in range(wl.K - 1)]
    P = Pair(wl)
    P.eng.set_mask_ids(ids)
    P.oracle.mask_ids = ids
    run_greedy(P)
    assert P.oracle.all_done()
    print("stats", P.stats)
    with pytest.raises(pard.PardError):
        P.eng.set_mask_ids(list(range(wl.K)))       # more than max_k - 1 offsets
    with pytest.raises(pard.PardError):
        P.eng.set_mask_ids([V] + ids[1:])            # outside the vocabulary
    P.eng.set_mask_ids(ids[:3])                      # too few for K - 1 = 11 mask rows
    P.eng.prefill(P.prompts, wl.n_new, wl.K)
    out = P.eng.alloc_step_outputs()
    with pytest.raises(pard.PardError):
        P.eng.draft(out)
    P.eng.set_mask_ids(None)


def test_stalled_wait_is_reported_and_the_context_stays_usable():
    """Failure detection without a GPU fault: a kernel's bounded pipeline wait
    on a barrier nothing completes gives up after its limit, sets the timeout
    bit and returns; pard_last_status reports it, and the next decode steps
    still match the oracle."""
    wl = S.WORKLOADS["tiny"].replace(n_new=12)
    P = Pair(wl)
    P.prefill()
    greedy_step(P, 1)
    assert P.eng.last_status() == 0
    P.eng.selftest_stalled_wait()
    assert P.eng.last_status() == 1  # ST_TIMEOUT_TMA
    greedy_step(P, 2)
    assert P.eng.last_status() == 0


def test_cod_keep_flags_match_the_oracle_bit_exactly():
    """COD data construction (Section 3.2, appendix algorithm) on the GPU:
    keep flags and per-subtask counts identical to the oracle's for ragged
    sample lengths, K = 1..8, several retention settings, the 4096-row
    maximum and the degenerate cases (n = 1, r = 1, r_min = 1)."""
    import torch
    from oracle import cod
    from paper_2504_18583_gb300 import pard
    cases = [(1, 3, 0.5, 0.0), (4, 3, 0.5, 0.0), (37, 2, 0.5, 0.0), (500, 8, 0.5, 0.0), (777, 6, 0.7, 0.1),
             (2048, 8, 0.5, 0.05), (4096, 8, 0.6, 0.0), (64, 1, 0.5, 0.0), (100, 5, 1.0, 0.0), (100, 5, 0.3, 1.0)]
    for t, (n, K, r, r_min) in enumerate(cases):
        keep_g, counts_g = pard.cod_select(n, K, r, r_min, seed=1000 + t, sample_id=t)
        keep_o, counts_o = cod.cod_select(n, K, r, r_min, seed=1000 + t, sample_id=t)
        torch.cuda.synchronize()
        assert counts_g.cpu().tolist() == counts_o, (n, K, r, r_min)
        assert np.array_equal(keep_g.cpu().numpy(), keep_o), (n, K, r, r_min)
    # one 2048-row, K = 8 sample, timed on the device
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    pard.cod_select(2048, 8, 0.5, 0.0, 1, 0)
    ev[0].record()
    for i in range(20):
        pard.cod_select(2048, 8, 0.5, 0.0, 1, i)
    ev[1].record()
    torch.cuda.synchronize()
    print("COD 2048 rows, K = 8: %.1f us per sample" % (ev[0].elapsed_time(ev[1]) * 1e3 / 20))


def test_page_pool_exhaustion_and_device_bounds_flag():
    """Host and device checks without a fault: a batch whose page reservation
    exceeds the pool returns PARD_ERR_NO_PAGES before any launch; a verify
    candidate outside the vocabulary is caught by the row-plan kernel, which
    flags ST_BAD_TOKEN (read by pard_last_status as PARD_ERR_DEVICE_CHECK)
    and embeds token 0 instead of reading out of bounds."""
    import torch
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["tiny"].replace(n_new=20, prompt_len=40)
    tw = S.device_weights(wl.target, wl.seed, S.TARGET)
    dw = S.device_weights(wl.draft, wl.seed, S.DRAFT)
    eng = pard.PardEngine(wl.target, tw, wl.draft, dw, max_batch=1, max_k=wl.K, max_ctx=256, n_pages=2,
                          prefill_chunk=64)
    with pytest.raises(pard.PardError) as e:
        eng.prefill([list(range(1, 41))], wl.n_new, wl.K)
    assert e.value.code == -3  # PARD_ERR_NO_PAGES: 40 + 20 + 2K positions need 5 pages of 16
    P = Pair(wl)
    P.prefill()
    out = P.eng.alloc_step_outputs()
    P.eng.draft(out)
    bad = torch.full((1, wl.K), wl.target.vocab + 5, dtype=torch.int32, device="cuda")
    P.eng.verify(out, bad)
    assert P.eng.last_status() == 1 << 3  # ST_BAD_TOKEN
    assert P.eng.last_status() == 0       # the word is cleared once read


def test_tiny_greedy_jittered_norms_batch_ragged():
    """Batch of 3 with prompts 17 / 33 / 50 tokens (page boundaries at
    several offsets), norm gains != 1, prefill chunks of 64 rows."""
    wl = S.WORKLOADS["tiny"].replace(batch=3, prompt_len=None, prompt_len_range=(17, 50), norm_jitter=0.1,
                                     n_new=20)
    wl = wl.replace(target=wl.target.replace(ffn=768), draft=wl.draft.replace(ffn=768))
    P = Pair(wl)
    run_greedy(P)
    print("stats", P.stats)


def test_self_draft_accepts_and_rolls_back():
    """Draft = target: d_0 always equals the target's argmax, so every step
    accepts at least one candidate and commit/rollback runs with a > 0."""
    wl = S.WORKLOADS["tiny"].replace(n_new=30, batch=2, prompt_len=40)
    P = Pair(wl, draft_is_target=True)
    outs = run_greedy(P)
    accs = [int(o["a"][b]) for o in outs for b in range(2)]
    assert max(accs) >= 1
    print("accept lengths", accs, P.stats)


def test_injected_candidates_hit_every_accept_length():
    """pard_verify on the target's own greedy continuation with one planted
    mismatch at j accepts exactly j candidates (j = K: none planted)."""
    wl = S.WORKLOADS["tiny"].replace(n_new=40)
    P = Pair(wl)
    K = wl.K
    ar = oracle.ar_greedy(wl.target, P.tw_host, P.prompts[0], wl.n_new + K + 2)
    seen = set()

    def inject(P, step):
        n0 = len(P.oracle.generated[0])
        j = (step - 1) % (K + 1)
        cont = list(ar[n0:n0 + K])
        while len(cont) < K:
            cont.append(0)
        if j < K:
            cont[j] = (cont[j] + 1) % (wl.target.vocab - 1)
        return np.array([cont], dtype=np.int32)

    outs = run_greedy(P, inject_fn=inject)
    for s, o in enumerate(outs):
        seen.add(int(o["a"][0]))
    assert seen >= set(range(K + 1)) - {K} or len(seen) >= K
    print("accept lengths seen", sorted(seen), P.stats)


def test_kv_cache_holds_the_oracle_keys_and_values():
    wl = S.WORKLOADS["tiny"].replace(n_new=12)
    P = Pair(wl)
    run_greedy(P)
    n = P.oracle.n[0]
    pos = list(range(0, n - 1))
    for model, om, shape in ((0, P.oracle.T, wl.target), (1, P.oracle.D, wl.draft)):
        upto = n - 1 if model == 0 else n - len(P.oracle.pending[0])
        for layer in (0, shape.n_layers - 1):
            k, v = P.eng.read_kv(model, layer, 0, pos[:upto], shape)
            k = k.float().cpu().numpy()
            v = v.float().cpu().numpy()
            ko = om.kc[0][layer, :upto]
            vo = om.vc[0][layer, :upto]
            # bf16 storage: relative 2^-8 plus the accumulated logit-level error
            assert np.abs(k - ko).max() <= 0.02 * max(1.0, np.abs(ko).max())
            assert np.abs(v - vo).max() <= 0.02 * max(1.0, np.abs(vo).max())


def test_full_width_8b_layers_short_prompt():
    """8B-shaped target and 1B-shaped draft at full width (every GEMM,
    attention and LM-head tile count of the full models), two layers each,
    64-token prompt, three steps; K = 8 gives 16 draft rows and 9 verify rows."""
    wl = S.WORKLOADS["8b_greedy"].replace(target=S.TARGET_8B.replace(n_layers=2),
                                          draft=S.DRAFT_1B.replace(n_layers=2), prompt_len=64, n_new=20)
    P = Pair(wl, prefill_chunk=64)
    P.prefill()
    for step in range(1, 4):
        greedy_step(P, step)
    assert P.eng.last_status() == 0
    print("stats", P.stats)


def test_autoregressive_mode_k0_matches_the_oracle_forward():
    """K = 0: each pard_verify + pard_accept_commit decodes one token with the
    target alone (Eq. 2); logits and tokens against one oracle forward per
    token, teacher-forced onto the GPU's token."""
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["tiny"].replace(n_new=20)
    tw = S.model_weights(wl.target, wl.seed, S.TARGET, wl.norm_jitter)
    dw = S.model_weights(wl.draft, wl.seed, S.DRAFT, wl.norm_jitter)
    prompt = [int(t) for t in wl.prompts()[0]]
    P_len = len(prompt)
    eng = pard.PardEngine(wl.target, S.device_weights(wl.target, 0, 0, host=tw), wl.draft,
                          S.device_weights(wl.draft, 0, 0, host=dw), max_batch=1, max_k=wl.K,
                          max_ctx=P_len + wl.n_new + 2 * wl.K + 16, n_pages=wl.n_pages(), prefill_chunk=64,
                          page_order_target=wl.page_order(S.TARGET), page_order_draft=wl.page_order(S.DRAFT))
    stats = dict(excused_tokens=0, checked_tokens=0)
    m = oracle.OracleModel(wl.target, tw, 1, P_len + wl.n_new + 2)
    lg = m.forward(0, prompt, np.arange(P_len, dtype=np.int32), [P_len - 1])[0]
    tok = int(eng.prefill([prompt], wl.n_new, 0).cpu().numpy()[0])
    check_token(tok, lg, stats, "first token")
    out = eng.alloc_step_outputs(want_logits=True)
    for step in range(1, wl.n_new):
        eng.verify(out, None, 1.0)
        y = out["logits"][0, 0].cpu().numpy()
        lg = m.forward(0, [tok], [P_len + step - 1], [0])[0]
        assert float(np.abs(y - lg).max()) <= LOGIT_TOL, f"step {step}"
        eng.accept_commit(out, False, 1.0, 0, step)
        assert int(out["n_emit"][0]) == 1 and int(out["accept_len"][0]) == 0
        tok = int(out["emitted"][0, 0])
        check_token(tok, lg, stats, f"step {step}")
    n, gen, done = eng.state()
    assert gen == [wl.n_new] and done == [1]
    assert eng.last_status() == 0
    with pytest.raises(RuntimeError):
        eng.draft(out)
    print("stats", stats)


def test_batch16_ragged_full_width_two_layers():
    """The batch-16 ragged configuration (8b_batch16: K = 6, ragged prompts)
    at full width with two layers per model: 16 x 7 = 112 verify rows and 192
    draft rows take the 64-token tiles, and attention covers 16 sequences of
    different lengths.  Prompts are 16..64 tokens here (the configuration's
    128..2048 keep the CPU oracle's prefill within seconds only at this size)."""
    wl = S.WORKLOADS["8b_batch16"].replace(target=S.TARGET_8B.replace(n_layers=2),
                                           draft=S.DRAFT_1B.replace(n_layers=2), prompt_len_range=(16, 64), n_new=12)
    P = Pair(wl, prefill_chunk=64)
    P.prefill()
    for step in range(1, 4):
        greedy_step(P, step)
    assert P.eng.last_status() == 0
    print("stats", P.stats)


# ----------------------------------------------------------------------------
# speculative sampling
# ----------------------------------------------------------------------------
def test_sampling_decisions_on_identical_logits():
    """Level 1: the oracle's logits fed to the GPU acceptance kernels with the
    same Philox streams give the same accept/reject decisions and bonus draws
    (except where u*q and p are within a few ulps)."""
    import torch
    wl = S.WORKLOADS["tiny"].replace(sample=True, n_new=1000, K=4)
    P = Pair(wl)
    P.prefill(seed=5)
    rng = np.random.default_rng(0)
    V, K = wl.target.vocab, wl.K
    mism = 0
    for trial in range(40):
        y = (rng.standard_normal((1, K + 1, V)) * 2.0).astype(np.float32)
        z = (y[:, :K] + rng.standard_normal((1, K, V)).astype(np.float32) * (0.3 + 0.1 * (trial % 5))).astype(np.float32)
        d = np.array([OP.draft_tokens(z[0], True, 1.0, 77 + trial, 3, 0)], dtype=np.int32)
        P.eng.set_logits(torch.as_tensor(y, device="cuda"), torch.as_tensor(z, device="cuda"),
                         torch.as_tensor(d, device="cuda"), 1.0)
        out = P.eng.alloc_step_outputs()
        step = 1000 + trial
        n_before = P.eng.state()[0][0]
        P.eng.accept_commit(out, True, 1.0, 5, step)
        a_g = int(out["accept_len"][0])
        em_g = out["emitted"][0].cpu().numpy()
        a_o, em_o = OP.accept_sampling(d[0], z[0], y[0], 1.0, 5, step, 0)
        if a_o != a_g:
            # excuse only a decision within rounding of the threshold
            i = min(a_o, a_g)
            p = OP.softmax_t(y[0, i], 1.0)[d[0, i]]
            q = OP.softmax_t(z[0, i], 1.0)[d[0, i]]
            u = uniform01(raw_words(5, STREAM_ACCEPT, step, 0, i, np.zeros(1, np.uint64)))[0]
            assert abs(u * q - p) <= 1e-5 * max(p, q), (trial, a_o, a_g)
            mism += 1
            continue
        take = int(out["n_emit"][0])
        assert list(em_g[:take]) == em_o[:take], (trial, em_g, em_o)
    assert mism <= 2


def test_sampling_end_to_end_tiny():
    """Level 2: sampling decode end to end (tiny models, batch 2, ragged
    prompts).  The sampled first token, the draft's Gumbel-max candidates,
    the accept / reject decisions and the bonus draws agree with the
    oracle's on the same Philox streams wherever the margins are clear (the
    margins follow from the measured logit differences); the oracle follows
    the GPU's tokens."""
    wl = S.WORKLOADS["tiny"].replace(sample=True, n_new=40, batch=2, prompt_len=None, prompt_len_range=(20, 45))
    P = Pair(wl)
    seed = 11
    P.prefill(seed)
    step = 1
    while not P.oracle.all_done() and step < 60:
        sampling_step(P, step, seed)
        step += 1
    assert P.oracle.all_done()
    st = P.stats
    print("stats", st)
    assert st["decisions_checked"] > 0
    # draft candidates, first tokens and bonus draws: nearly all have clear margins
    assert st["sampled_exact"] >= 0.9 * st["sampled_checked"]
    assert P.eng.last_status() == 0


def test_sampling_full_width_8b_two_layers():
    """The sampling configuration (8b_sample: T = 1, K = 6) at full width with
    two layers per model, 64-token prompt: logits within tolerance; sampled
    candidates, first token, decisions and bonus draws as in the tiny test;
    KV slots equal."""
    wl = S.WORKLOADS["8b_sample"].replace(target=S.TARGET_8B.replace(n_layers=2),
                                          draft=S.DRAFT_1B.replace(n_layers=2), prompt_len=64, n_new=24)
    P = Pair(wl, prefill_chunk=64)
    seed = 5
    P.prefill(seed)
    for step in range(1, 5):
        sampling_step(P, step, seed)
    st = P.stats
    print("stats", st)
    assert st["sampled_exact"] >= 0.9 * st["sampled_checked"]
    assert P.eng.last_status() == 0


def test_vanilla_sd_sampled_sequential_draft():
    """The sampled form of vanilla speculative decoding's drafting stage
    (Section 2.2): every draft pass draws its candidate by Gumbel-max from
    its own logits (Philox stream 0, row i); candidates, decisions and bonus
    draws against the oracle's sequential draft fed the GPU's candidates,
    margins as in the other sampling tests; batch 2, ragged prompts."""
    wl = S.WORKLOADS["tiny"].replace(sample=True, n_new=30, batch=2, prompt_len=None, prompt_len_range=(20, 45))
    P = Pair(wl)
    seed = 13
    P.prefill(seed)
    step = 1
    while not P.oracle.all_done() and step < 40:
        sampling_step(P, step, seed, sequential=True)
        step += 1
    st = P.stats
    print("stats", st)
    assert P.oracle.all_done()
    assert st["sampled_exact"] >= 0.9 * st["sampled_checked"]
    assert P.eng.last_status() == 0


@pytest.mark.parametrize("vocab", [2048, 128256])
def test_draft_sampler_on_identical_logits(vocab):
    """Level 1 for the draft's candidate selection (Eq. 6, sampled at
    temperature T, and greedy): given draft logits go through the same tile
    statistics and selection kernel as the LM head's, and the candidates
    equal the oracle's Gumbel-max (or argmax) winners on the same Philox
    stream exactly, except where the winner's lead is a few fp32 ulps."""
    import torch
    wl = S.WORKLOADS["tiny"].replace(batch=3, K=6, n_new=100, prompt_len=20)
    if vocab != wl.target.vocab:
        wl = wl.replace(target=wl.target.replace(vocab=vocab, mask_id=vocab - 1),
                        draft=wl.draft.replace(vocab=vocab, mask_id=vocab - 1))
    P = Pair(wl)
    P.prefill()
    B, K, V = wl.batch, wl.K, vocab
    rng = np.random.default_rng(vocab)
    near = exact = 0
    for trial in range(12):
        T = (0.7, 1.0, 1.3)[trial % 3]
        sample = trial % 4 != 3
        z = (rng.standard_normal((B, K, V)) * 2.0).astype(np.float32)
        out = P.eng.alloc_step_outputs()
        seed, step = 31 + trial, 200 + trial
        P.eng.set_draft_logits(torch.as_tensor(z, device="cuda"), out, sample, T, seed, step)
        d_g = out["draft"].cpu().numpy()
        for b in range(B):
            d_o = OP.draft_tokens(z[b], sample, T, seed, step, b)
            for i in range(K):
                if int(d_g[b, i]) == d_o[i]:
                    exact += 1
                    continue
                sc = (gumbel_scores(z[b, i], T, seed, STREAM_DRAFT, step, b, i) if sample
                      else z[b, i].astype(np.float32))
                assert margin(sc) <= GUMBEL_EPS, (trial, b, i, int(d_g[b, i]), d_o[i], margin(sc))
                near += 1
    print("exact", exact, "near ties", near)
    assert near <= 2 and exact >= B * K * 12 - 2


def test_weight_packing_round_trip_restores_every_matrix():
    """Loading packs the weight matrices in place; unpacking restores the
    exact row-major bits (including a draft sharing the target's tensors)."""
    import torch
    wl = S.WORKLOADS["tiny"].replace(target=S.TARGET_8B.replace(n_layers=1, vocab=2048, mask_id=2047),
                                     draft=S.DRAFT_1B.replace(n_layers=1, vocab=2048, mask_id=2047))
    P = Pair(wl)
    host = P.tw_host
    dev = P.tw_dev
    packed_any = not torch.equal(dev["layers"][0]["wq"].view(torch.int16).cpu(),
                                 torch.from_numpy(host["layers"][0]["wq"].view("int16")))
    assert packed_any, "wq should be in the packed layout while loaded"
    P.eng.unpack_weights()
    for name in ("wq", "wk", "wv", "wo", "wg", "wu", "wd"):
        got = dev["layers"][0][name].view(torch.int16).cpu().numpy()
        assert np.array_equal(got, host["layers"][0][name].view("int16")), name
    assert np.array_equal(dev["lm_head"].view(torch.int16).cpu().numpy(), host["lm_head"].view("int16"))
    with pytest.raises(Exception):
        P.eng.prefill([[1, 2, 3]], 4, wl.K)


def test_state_errors_are_reported():
    from paper_2504_18583_gb300 import pard
    wl = S.WORKLOADS["tiny"]
    P = Pair(wl)
    out = P.eng.alloc_step_outputs()
    with pytest.raises(pard.PardError) as e:
        P.eng.draft(out)
    assert e.value.code == -7
    with pytest.raises(pard.PardError) as e:
        P.eng.prefill([list(range(10))], 10_000, wl.K)
    assert e.value.code == -1
