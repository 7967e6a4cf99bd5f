"""The allocation-free acceptance entry point gives the same results as the
context-based path (pard_set_logits + pard_accept_commit) on the same
inputs, for two calls in a row (greedy and sampling), through the C ABI.

This file is collected last on purpose: pard_accept_noalloc is an interface
for callers that cannot provide device memory (no device allocator, or an
engine that forbids allocation on its serving path), and its scratch lives in
a fixed device array shared by all calls."""
import numpy as np
import pytest

import synthetic as S
from oracle import pard as OP

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("batch,K,vocab", [(1, 4, 2048), (3, 4, 2048), (16, 8, 128256)],
                         ids=["b1k4", "b3k4", "b16k8_full_vocab"])
def test_noalloc_acceptance_matches_context_path_twice(batch, K, vocab):
    """Four calls in a row (two sampled, two greedy) at batch 1, at batch 3,
    and at the scratch's limits (batch 16, K = 8, the 128256-entry
    vocabulary: every row pitch and tile count of its fixed layout)."""
    import torch
    from _parity import Pair
    from paper_2504_18583_gb300 import _build, pard
    _build.build()
    wl = S.WORKLOADS["tiny"].replace(sample=True, n_new=100000, K=K, batch=batch, prompt_len=20)
    if vocab != wl.target.vocab:
        wl = wl.replace(target=wl.target.replace(vocab=vocab, mask_id=vocab - 1),
                        draft=wl.draft.replace(vocab=vocab, mask_id=vocab - 1))
    P = Pair(wl)
    P.prefill(seed=3)
    B, V = wl.batch, vocab
    rng = np.random.default_rng(11 + batch)
    lib = pard.lib()
    stream = P.eng.stream.cuda_stream
    for call, sample in enumerate((True, True, False, False)):
        y = (rng.standard_normal((B, K + 1, V)) * 2.0).astype(np.float32)
        z = (y[:, :K] + rng.standard_normal((B, K, V)).astype(np.float32) * 0.5).astype(np.float32)
        d = np.array([OP.draft_tokens(z[b], True, 1.0, 900 + call, 2, b) for b in range(B)], dtype=np.int32)
        if call == 1:
            d[:, 1:] = np.argmax(y[:, 1:K], axis=-1)  # some acceptance deep into the draft
        yt, zt, dt = (torch.as_tensor(a, device="cuda") for a in (y, z, d))
        step = 50 + call
        # existing path
        P.eng.set_logits(yt, zt, dt, 1.0)
        out = P.eng.alloc_step_outputs()
        P.eng.accept_commit(out, sample, 1.0, 7, step)
        # allocation-free path, same inputs
        acc2 = torch.full((B,), -9, dtype=torch.int32, device="cuda")
        em2 = torch.full((B, K + 1), -9, dtype=torch.int32, device="cuda")
        code = lib.pard_accept_noalloc(yt.data_ptr(), zt.data_ptr(), dt.data_ptr(), B, K, V, int(sample), 1.0, 7,
                                       step, acc2.data_ptr(), em2.data_ptr(), stream)
        assert code == 0, pard.pard_last_error()
        torch.cuda.synchronize()
        assert torch.equal(acc2, out["accept_len"]), (call, acc2, out["accept_len"])
        assert torch.equal(em2, out["emitted"]), (call, em2, out["emitted"])
    # sizes beyond the static scratch are refused with a message
    code = lib.pard_accept_noalloc(yt.data_ptr(), zt.data_ptr(), dt.data_ptr(), 17, K, V, 0, 1.0, 0, 0,
                                   acc2.data_ptr(), em2.data_ptr(), stream)
    assert code == -1 and "static scratch" in pard.pard_last_error()
    assert P.eng.last_status() == 0
