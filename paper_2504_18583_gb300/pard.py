"""Python binding of libpard (ctypes): the C ABI's functions under the same
names, plus ``PardEngine``, which allocates the workspace and KV page pool
with torch and passes raw device pointers.  Every step of the decode path
runs in the library's CUDA kernels; there is no CPU fallback: without the
built library (or without a GB300) the calls raise."""
from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Optional, Sequence

from ._build import LIB

PARD_OK = 0
STATUS_NAMES = {0: "PARD_OK", -1: "PARD_ERR_ARG", -2: "PARD_ERR_SHAPE", -3: "PARD_ERR_NO_PAGES",
                -4: "PARD_ERR_CUDA", -5: "PARD_ERR_DEVICE_CHECK", -6: "PARD_ERR_TIMEOUT", -7: "PARD_ERR_STATE"}
LAYER_ORDER = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")


class ModelCfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32), ("n_q_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("ffn", ctypes.c_int32),
                ("vocab", ctypes.c_int32), ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float),
                ("mask_id", ctypes.c_int32)]

    @classmethod
    def of(cls, shape) -> "ModelCfg":
        return cls(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads, shape.head_dim,
                   shape.ffn, shape.vocab, shape.rope_theta, shape.rms_eps, shape.mask_id)


class Weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p), ("lm_head", ctypes.c_void_p),
                ("layers", ctypes.POINTER(ctypes.c_void_p))]


class Limits(ctypes.Structure):
    _fields_ = [("max_batch", ctypes.c_int32), ("max_k", ctypes.c_int32), ("max_ctx", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("prefill_chunk", ctypes.c_int32), ("n_pages", ctypes.c_int32)]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is missing: build it with __graft_entry__.build() "
                               "(there is no CPU fallback for the decode path)")
        L = ctypes.CDLL(LIB)
        vp, i32, u64, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_uint64, ctypes.c_float, ctypes.c_size_t
        P = ctypes.POINTER
        L.pard_workspace_bytes.argtypes = [P(ModelCfg), P(ModelCfg), P(Limits)]
        L.pard_workspace_bytes.restype = sz
        L.pard_kv_pool_bytes.argtypes = [P(ModelCfg), P(ModelCfg), P(Limits)]
        L.pard_kv_pool_bytes.restype = sz
        L.pard_load_weights.argtypes = [P(vp), P(ModelCfg), P(Weights), P(ModelCfg), P(Weights), P(Limits),
                                        vp, sz, vp, sz, vp, vp, vp]
        L.pard_prefill.argtypes = [vp, vp, vp, i32, i32, i32, i32, f32, u64, vp, vp]
        L.pard_draft.argtypes = [vp, i32, f32, u64, u64, vp, vp, vp]
        L.pard_draft_sequential.argtypes = [vp, i32, f32, u64, u64, vp, vp, vp]
        L.pard_set_mask_ids.argtypes = [vp, vp, i32, vp]
        L.pard_selftest_stalled_wait.argtypes = [vp, vp]
        L.pard_cod_select.argtypes = [i32, i32, ctypes.c_double, ctypes.c_double, u64, u64, vp, vp, vp]
        L.pard_verify.argtypes = [vp, vp, f32, vp, vp]
        L.pard_accept_commit.argtypes = [vp, i32, f32, u64, u64, vp, vp, vp, vp, vp]
        L.pard_set_logits.argtypes = [vp, vp, vp, vp, f32, vp]
        L.pard_set_draft_logits.argtypes = [vp, vp, i32, f32, u64, u64, vp, vp]
        L.pard_get_state.argtypes = [vp, vp, vp, vp, vp]
        L.pard_read_kv.argtypes = [vp, i32, i32, i32, vp, i32, vp, vp, vp]
        L.pard_last_status.argtypes = [vp, P(ctypes.c_uint32), vp]
        L.pard_accept_noalloc.argtypes = [vp, vp, vp, i32, i32, i32, i32, f32, u64, u64, vp, vp, vp]
        L.pard_accept_noalloc.restype = ctypes.c_int
        L.pard_attention_paths.argtypes = [vp, P(ctypes.c_uint32), vp]
        L.pard_attention_paths.restype = ctypes.c_int
        L.pard_set_attention_split_cap.argtypes = [vp, i32]
        L.pard_set_attention_split_cap.restype = ctypes.c_int
        L.pard_unpack_weights.argtypes = [vp, vp]
        L.pard_unpack_weights.restype = ctypes.c_int
        L.pard_launch_count.argtypes = [vp]
        L.pard_launch_count.restype = i32
        L.pard_last_error.argtypes = []
        L.pard_last_error.restype = ctypes.c_char_p
        L.pard_destroy.argtypes = [vp]
        L.pard_destroy.restype = None
        for name in ("pard_load_weights", "pard_prefill", "pard_draft", "pard_draft_sequential", "pard_verify",
                     "pard_accept_commit", "pard_set_mask_ids", "pard_selftest_stalled_wait", "pard_cod_select",
                     "pard_set_logits", "pard_set_draft_logits", "pard_get_state", "pard_read_kv", "pard_last_status"):
            getattr(L, name).restype = ctypes.c_int
        _lib = L
    return _lib


def cod_select(n: int, K: int, r: float, r_min: float, seed: int, sample_id: int, stream=None):
    """COD data construction for one sample (pard_cod_select): returns device
    tensors keep [K-1, n] and counts [K] (int32), enqueued on `stream`."""
    import torch
    keep = torch.zeros((max(K - 1, 1), n), dtype=torch.int32, device="cuda")
    counts = torch.zeros(K, dtype=torch.int32, device="cuda")
    s = stream if stream is not None else torch.cuda.current_stream()
    _check(lib().pard_cod_select(n, K, float(r), float(r_min), seed, sample_id, keep.data_ptr(), counts.data_ptr(),
                                 s.cuda_stream), "pard_cod_select")
    return keep[:K - 1], counts


class PardError(RuntimeError):
    def __init__(self, code: int, where: str):
        msg = lib().pard_last_error().decode(errors="replace")
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)}: {msg}")
        self.code = code


def _check(code: int, where: str) -> None:
    if code != PARD_OK:
        raise PardError(code, where)


def _ptr(t) -> Optional[int]:
    return None if t is None else t.data_ptr()


# thin wrappers with the C names --------------------------------------------------
def pard_workspace_bytes(tcfg: ModelCfg, dcfg: ModelCfg, lim: Limits) -> int:
    return lib().pard_workspace_bytes(ctypes.byref(tcfg), ctypes.byref(dcfg), ctypes.byref(lim))


def pard_kv_pool_bytes(tcfg: ModelCfg, dcfg: ModelCfg, lim: Limits) -> int:
    return lib().pard_kv_pool_bytes(ctypes.byref(tcfg), ctypes.byref(dcfg), ctypes.byref(lim))


def pard_last_error() -> str:
    return lib().pard_last_error().decode(errors="replace")


class PardEngine:
    """Owns the device memory (torch) for one target + draft pair and calls
    the library.  ``target_w`` / ``draft_w``: {'embed','final_norm','lm_head',
    'layers': [ {name: tensor} ]} of contiguous bf16 CUDA tensors."""

    def __init__(self, target_shape, target_w: Dict, draft_shape, draft_w: Dict, *, max_batch: int,
                 max_k: int, max_ctx: int, n_pages: int, page_size: int = 16, prefill_chunk: int = 512,
                 page_order_target: Optional[Sequence[int]] = None,
                 page_order_draft: Optional[Sequence[int]] = None, stream=None):
        import torch
        self.torch = torch
        self.dev = torch.device("cuda", torch.cuda.current_device())
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.tcfg, self.dcfg = ModelCfg.of(target_shape), ModelCfg.of(draft_shape)
        self.vocab = target_shape.vocab
        self.lim = Limits(max_batch, max_k, max_ctx, page_size, prefill_chunk, n_pages)
        ws = pard_workspace_bytes(self.tcfg, self.dcfg, self.lim)
        kv = pard_kv_pool_bytes(self.tcfg, self.dcfg, self.lim)
        if ws == 0 or kv == 0:
            raise ValueError("libpard rejected the shapes or limits")
        self.workspace = torch.empty(ws + 256, dtype=torch.uint8, device=self.dev)
        self.kv_pool = torch.empty(kv + 256, dtype=torch.uint8, device=self.dev)
        self._keep = [target_w, draft_w]
        self._tw, self._tl = self._weights(target_shape, target_w)
        self._dw, self._dl = self._weights(draft_shape, draft_w)
        ot = self._order(page_order_target, n_pages)
        od = self._order(page_order_draft, n_pages)
        self.ctx = ctypes.c_void_p()
        _check(lib().pard_load_weights(ctypes.byref(self.ctx), ctypes.byref(self.tcfg), ctypes.byref(self._tw),
                                       ctypes.byref(self.dcfg), ctypes.byref(self._dw), ctypes.byref(self.lim),
                                       self._aligned(self.kv_pool), kv, self._aligned(self.workspace), ws,
                                       ot, od, self.stream.cuda_stream), "pard_load_weights")
        self.batch = 0
        self.K = 0

    @staticmethod
    def _aligned(t) -> int:
        p = t.data_ptr()
        return (p + 255) & ~255

    @staticmethod
    def _order(order, n):
        if order is None:
            return None
        arr = (ctypes.c_int32 * n)(*[int(x) for x in order])
        return ctypes.cast(arr, ctypes.c_void_p)

    def _weights(self, shape, w):
        ptrs = (ctypes.c_void_p * (shape.n_layers * 9))()
        for l in range(shape.n_layers):
            for j, name in enumerate(LAYER_ORDER):
                t = w["layers"][l][name]
                assert t.is_cuda and t.is_contiguous()
                ptrs[l * 9 + j] = t.data_ptr()
        return Weights(w["embed"].data_ptr(), w["final_norm"].data_ptr(), w["lm_head"].data_ptr(),
                       ctypes.cast(ptrs, ctypes.POINTER(ctypes.c_void_p))), ptrs

    def close(self):
        if self.ctx:
            lib().pard_destroy(self.ctx)
            self.ctx = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the decode step ----------------------------------------------------------
    def prefill(self, prompts: Sequence[Sequence[int]], n_new: int, K: int, sample: bool = False,
                temperature: float = 1.0, seed: int = 0):
        torch = self.torch
        toks = torch.tensor([t for p in prompts for t in p], dtype=torch.int32, device=self.dev)
        lens = (ctypes.c_int32 * len(prompts))(*[len(p) for p in prompts])
        first = torch.empty(len(prompts), dtype=torch.int32, device=self.dev)
        _check(lib().pard_prefill(self.ctx, toks.data_ptr(), ctypes.cast(lens, ctypes.c_void_p), len(prompts),
                                  n_new, K, int(sample), temperature, seed, first.data_ptr(),
                                  self.stream.cuda_stream), "pard_prefill")
        self.batch, self.K = len(prompts), K
        return first

    def alloc_step_outputs(self, want_logits: bool = False):
        torch = self.torch
        B, K, V = self.batch, self.K, self.vocab
        o = dict(draft=torch.empty((B, K), dtype=torch.int32, device=self.dev),
                 accept_len=torch.empty(B, dtype=torch.int32, device=self.dev),
                 emitted=torch.empty((B, K + 1), dtype=torch.int32, device=self.dev),
                 kv_slots=torch.empty((B, K + 1), dtype=torch.int32, device=self.dev),
                 n_emit=torch.empty(B, dtype=torch.int32, device=self.dev))
        if want_logits:
            o["draft_logits"] = torch.empty((B, K, V), dtype=torch.float32, device=self.dev)
            o["logits"] = torch.empty((B, K + 1, V), dtype=torch.float32, device=self.dev)
        return o

    def draft(self, out, sample=False, temperature=1.0, seed=0, step=0):
        _check(lib().pard_draft(self.ctx, int(sample), temperature, seed, step, out["draft"].data_ptr(),
                                _ptr(out.get("draft_logits")), self.stream.cuda_stream), "pard_draft")

    def draft_sequential(self, out, sample=False, temperature=1.0, seed=0, step=0):
        """Vanilla speculative decoding's K-pass draft (same outputs as draft())."""
        _check(lib().pard_draft_sequential(self.ctx, int(sample), temperature, seed, step, out["draft"].data_ptr(),
                                           _ptr(out.get("draft_logits")), self.stream.cuda_stream),
               "pard_draft_sequential")

    def set_mask_ids(self, ids=None):
        """One mask id per draft offset (None: the config's shared id)."""
        n = 0 if ids is None else len(ids)
        arr = (ctypes.c_int32 * max(n, 1))(*(ids or [0]))
        _check(lib().pard_set_mask_ids(self.ctx, ctypes.cast(arr, ctypes.c_void_p) if n else None, n,
                                       self.stream.cuda_stream), "pard_set_mask_ids")

    def verify(self, out, draft_in=None, temperature=1.0):
        _check(lib().pard_verify(self.ctx, _ptr(draft_in), temperature, _ptr(out.get("logits")),
                                 self.stream.cuda_stream), "pard_verify")

    def accept_commit(self, out, sample=False, temperature=1.0, seed=0, step=0):
        _check(lib().pard_accept_commit(self.ctx, int(sample), temperature, seed, step,
                                        out["accept_len"].data_ptr(), out["emitted"].data_ptr(),
                                        out["kv_slots"].data_ptr(), out["n_emit"].data_ptr(),
                                        self.stream.cuda_stream), "pard_accept_commit")

    def step(self, out, sample=False, temperature=1.0, seed=0, step=0, sequential=False):
        """One PARD step: draft, verify, accept/commit (K = 0: one autoregressive token, no draft;
        sequential: vanilla speculative decoding's K-pass draft)."""
        if self.K:
            (self.draft_sequential if sequential else self.draft)(out, sample, temperature, seed, step)
        self.verify(out, None, temperature)
        self.accept_commit(out, sample, temperature, seed, step)

    def set_logits(self, target_logits, draft_logits, draft, temperature=1.0):
        _check(lib().pard_set_logits(self.ctx, target_logits.data_ptr(), _ptr(draft_logits), draft.data_ptr(),
                                     temperature, self.stream.cuda_stream), "pard_set_logits")

    def set_draft_logits(self, draft_logits, out, sample=False, temperature=1.0, seed=0, step=0):
        """Candidates from given draft logits [B, K, V] into out['draft'] (pard_set_draft_logits)."""
        _check(lib().pard_set_draft_logits(self.ctx, draft_logits.data_ptr(), int(sample), temperature, seed, step,
                                           out["draft"].data_ptr(), self.stream.cuda_stream), "pard_set_draft_logits")

    def state(self):
        B = max(self.batch, 1)
        n, g, d = (ctypes.c_int32 * B)(), (ctypes.c_int32 * B)(), (ctypes.c_int32 * B)()
        _check(lib().pard_get_state(self.ctx, ctypes.cast(n, ctypes.c_void_p), ctypes.cast(g, ctypes.c_void_p),
                                    ctypes.cast(d, ctypes.c_void_p), self.stream.cuda_stream), "pard_get_state")
        return list(n), list(g), list(d)

    def read_kv(self, model: int, layer: int, b: int, positions: Sequence[int], shape):
        torch = self.torch
        n = len(positions)
        k = torch.empty((n, shape.n_kv_heads, shape.head_dim), dtype=torch.bfloat16, device=self.dev)
        v = torch.empty_like(k)
        pos = (ctypes.c_int32 * n)(*positions)
        _check(lib().pard_read_kv(self.ctx, model, layer, b, ctypes.cast(pos, ctypes.c_void_p), n, k.data_ptr(),
                                  v.data_ptr(), self.stream.cuda_stream), "pard_read_kv")
        return k, v

    def selftest_stalled_wait(self):
        """Enqueue the bounded-wait self test (its wait runs out after 2 s)."""
        _check(lib().pard_selftest_stalled_wait(self.ctx, self.stream.cuda_stream), "pard_selftest_stalled_wait")

    def last_status(self) -> int:
        flags = ctypes.c_uint32(0)
        code = lib().pard_last_status(self.ctx, ctypes.byref(flags), self.stream.cuda_stream)
        if code not in (PARD_OK, -5, -6):
            _check(code, "pard_last_status")
        return flags.value

    def unpack_weights(self) -> None:
        """Restore the row-major weight layout (the engine is unusable after)."""
        _check(lib().pard_unpack_weights(self.ctx, self.stream.cuda_stream), "pard_unpack_weights")

    def launch_count(self) -> int:
        return lib().pard_launch_count(self.ctx)

    def attention_paths(self) -> int:
        """Attention combine forms run since the last call (bit 0 push, bit 1
        pull, bit 3 + n: clusters of n CTAs); the record is cleared."""
        bits = ctypes.c_uint32(0)
        _check(lib().pard_attention_paths(self.ctx, ctypes.byref(bits), self.stream.cuda_stream),
               "pard_attention_paths")
        return bits.value

    def set_attention_split_cap(self, cap: int) -> None:
        """At most `cap` key splits (CTAs of one cluster) per attention unit; 0: the default 16."""
        _check(lib().pard_set_attention_split_cap(self.ctx, int(cap)), "pard_set_attention_split_cap")
