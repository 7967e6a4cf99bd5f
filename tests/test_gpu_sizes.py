"""GPU parity at the configurations' full sizes: long contexts (the paged
attention's pull combine and many K/V ring wraps), the 70B-shaped target's
widths, and the 8B-shaped target at full depth.  The oracle runs every
prefill and step itself (nothing is seeded from the GPU), so these tests
spend minutes of host-core time."""
import numpy as np
import pytest

import synthetic as S

from _parity import LOGIT_TOL, Pair, greedy_step, sampling_step

pytestmark = pytest.mark.gpu

PUSH, PULL, RING2, SPLIT0 = 1 << 0, 1 << 1, 1 << 2, 3


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2504_18583_gb300 import _build
    _build.build()


def split_sizes(bits: int):
    return sorted(n for n in range(1, 17) if bits & (1 << (SPLIT0 + n)))


def test_long_contexts_pull_combine_and_8_cta_clusters():
    """8B widths, two layers per model, two sequences with 2100- and
    4200-token prompts (the C3 range's top and the C4 context), K = 8:
    verify and draft attention walk 66-133 key chunks per unit over 16-CTA
    clusters, which combine their splits by the pull over distributed shared
    memory; three greedy steps against the oracle.  Then the same sequences
    with the key splits capped at 8 (the clusters the launcher falls back to
    on a GPU that cannot place 16 CTAs): three more steps."""
    wl = S.WORKLOADS["8b_greedy"].replace(target=S.TARGET_8B.replace(n_layers=2),
                                          draft=S.DRAFT_1B.replace(n_layers=2), batch=2, prompt_len=None,
                                          prompt_lens_given=(2100, 4200), n_new=40)
    P = Pair(wl, prefill_chunk=512)
    P.prefill()
    P.eng.attention_paths()  # clear the prefill's record
    for step in range(1, 4):
        greedy_step(P, step)
    bits = P.eng.attention_paths()
    print("16-CTA clusters: paths", hex(bits), "cluster sizes", split_sizes(bits), "stats", P.stats)
    assert bits & PULL and not bits & PUSH and not bits & RING2
    assert split_sizes(bits) == [16]
    P.eng.set_attention_split_cap(8)
    for step in range(4, 7):
        greedy_step(P, step)
    bits = P.eng.attention_paths()
    print("8-CTA clusters: paths", hex(bits), "cluster sizes", split_sizes(bits), "stats", P.stats)
    assert bits & PULL and split_sizes(bits) == [8]
    assert P.eng.last_status() == 0


def test_batch16_ragged_c3_prompts_two_layers():
    """The batch-16 configuration at its own sizes (16 prompts of 128..2048
    tokens drawn from its seed, K = 6), two layers per model at full width:
    112 verify and up to 192 draft rows over contexts that differ by 16x.
    The key splits are sized by the contexts' total (nine splits here, more
    units than two per SM), so the attention takes its two-buffer K/V ring
    with four CTAs per SM, and the long sequences' warp pairs split every
    chunk's keys; the clusters combine by the pull.  Three greedy steps."""
    wl = S.WORKLOADS["8b_batch16"].replace(target=S.TARGET_8B.replace(n_layers=2),
                                           draft=S.DRAFT_1B.replace(n_layers=2), n_new=20)
    print("prompt lengths", wl.prompt_lens())
    P = Pair(wl, prefill_chunk=512)
    P.prefill()
    P.eng.attention_paths()
    for step in range(1, 4):
        greedy_step(P, step)
    bits = P.eng.attention_paths()
    print("paths", hex(bits), "cluster sizes", split_sizes(bits), "stats", P.stats)
    assert bits & PULL and bits & RING2
    assert split_sizes(bits) == [9]
    assert P.eng.last_status() == 0


def test_70b_widths_two_layers_4096_context():
    """The 70B-shaped target's widths (d 8192, 64 query / 8 KV heads: GQA
    group 8, FFN 28672) with two layers, the 1B-shaped draft with two layers,
    a 4096-token prompt and K = 8: the group-8 attention instantiation (two
    row blocks for the 9 verify rows) and the 70B GEMM tile counts; three
    greedy steps against the oracle."""
    wl = S.WORKLOADS["70b_greedy"].replace(target=S.TARGET_70B.replace(n_layers=2),
                                           draft=S.DRAFT_1B.replace(n_layers=2), n_new=40)
    P = Pair(wl, prefill_chunk=512)
    P.prefill()
    P.eng.attention_paths()
    for step in range(1, 4):
        greedy_step(P, step)
    bits = P.eng.attention_paths()
    print("paths", hex(bits), "cluster sizes", split_sizes(bits), "stats", P.stats)
    # the 9 verify rows are two row blocks of 8 at group 8; 16-CTA clusters
    assert split_sizes(bits) == [16]
    assert P.eng.last_status() == 0


def test_full_depth_8b_greedy_c1():
    """The greedy configuration at full size: the 32-layer 8B-shaped target
    and 16-layer 1B-shaped draft, 512-token prompt, K = 8; four steps.  The
    largest logit difference over the whole depth is reported."""
    wl = S.WORKLOADS["8b_greedy"].replace(n_new=48)
    P = Pair(wl, prefill_chunk=512)
    P.prefill()
    for step in range(1, 5):
        greedy_step(P, step)
    print("full depth C1: max verify logit err %.4g, max draft logit err %.4g (tolerance %g); stats %s" % (
        P.stats["max_logit_err"], P.stats["max_draft_logit_err"], LOGIT_TOL, P.stats))
    assert P.eng.last_status() == 0


def test_full_depth_8b_sampling_c2():
    """The sampling configuration at full size: 32/16 layers, 1024-token
    prompt, K = 6, T = 1; four speculative-sampling steps with the sampled
    candidates, decisions and bonus draws checked against the oracle's."""
    wl = S.WORKLOADS["8b_sample"].replace(n_new=40)
    P = Pair(wl, prefill_chunk=512)
    seed = 9
    P.prefill(seed)
    for step in range(1, 5):
        sampling_step(P, step, seed)
    st = P.stats
    print("full depth C2: max verify logit err %.4g, max draft logit err %.4g (tolerance %g); stats %s" % (
        st["max_logit_err"], st["max_draft_logit_err"], LOGIT_TOL, st))
    assert st["sampled_exact"] >= 0.8 * st["sampled_checked"]
    assert P.eng.last_status() == 0
