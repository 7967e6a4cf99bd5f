"""Seeded synthetic workloads for the PARD decode step.

This module is shared by the CPU oracle, the tests, ``bench.py`` and the
smoke entry point.  It holds the workload shapes and turns seeds into
inputs (weights, prompt ids, prompt lengths, page orders); it holds none of
the method's arithmetic.

The workloads stand in for the paper's evaluation setting (LLaMA3.1-8B
target with a LLaMA3.2-1B PARD draft, Section 4.1; 70B target, Table 1):
trained weights and the HumanEval / GSM8K / SpecBench prompts are not
available, so every tensor is drawn N(0, 0.02) from a seed and every prompt
is uniform-random token ids.
"""
from __future__ import annotations

import ctypes
import dataclasses
import os
import subprocess
import tempfile
from typing import Dict, Iterator, List, Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB = None

BF16_ONE = 0x3F80
LAYER_TENSORS = ("attn_norm", "wq", "wk", "wv", "wo", "mlp_norm", "wg", "wu", "wd")
GLOBAL_TENSORS = ("embed", "final_norm", "lm_head")
TARGET, DRAFT = 0, 1


def _build_lib() -> str:
    src = os.path.join(_HERE, "gen.c")
    out = os.path.join(_HERE, "_synth_gen.so")
    if os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
    os.close(fd)
    subprocess.check_call(["gcc", "-O2", "-std=c99", "-fopenmp", "-fPIC", "-shared",
                           "-ffp-contract=off", src, "-o", tmp, "-lm"])
    os.replace(tmp, out)
    return out


def build() -> None:
    """Compile the generator's C helper (idempotent)."""
    _lib()


def _lib():
    global _LIB
    if _LIB is None:
        lib = ctypes.CDLL(_build_lib())
        lib.synth_normal_bf16.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_double,
                                          ctypes.c_void_p, ctypes.c_int64]
        lib.synth_fill_bf16.argtypes = [ctypes.c_uint16, ctypes.c_void_p, ctypes.c_int64]
        lib.synth_uniform_int.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                          ctypes.c_int64, ctypes.c_void_p, ctypes.c_int64]
        lib.synth_permutation.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_void_p,
                                          ctypes.c_int64]
        _LIB = lib
    return _LIB


# --------------------------------------------------------------------------
# Shapes
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class ModelShape:
    """Llama-style decoder shape (the model families of Section 4.1)."""
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    ffn: int
    vocab: int
    rope_theta: float
    rms_eps: float
    mask_id: int

    def tensor_shape(self, name: str) -> Tuple[int, ...]:
        d, hq, hkv, hd = self.d_model, self.n_q_heads, self.n_kv_heads, self.head_dim
        return {
            "attn_norm": (d,), "mlp_norm": (d,), "final_norm": (d,),
            "wq": (hq * hd, d), "wk": (hkv * hd, d), "wv": (hkv * hd, d), "wo": (d, hq * hd),
            "wg": (self.ffn, d), "wu": (self.ffn, d), "wd": (d, self.ffn),
            "embed": (self.vocab, d), "lm_head": (self.vocab, d),
        }[name]

    def streamed_weight_bytes(self) -> int:
        """bf16 bytes one forward pass streams: every layer matrix, the norm
        gains and the LM head (the embedding is gathered, not streamed)."""
        per_layer = sum(int(np.prod(self.tensor_shape(n))) for n in LAYER_TENSORS)
        glob = int(np.prod(self.tensor_shape("lm_head"))) + self.d_model
        return 2 * (self.n_layers * per_layer + glob)

    def kv_bytes_per_token(self) -> int:
        """bf16 K and V bytes per token over all layers."""
        return 2 * 2 * self.n_layers * self.n_kv_heads * self.head_dim

    def replace(self, **kw) -> "ModelShape":
        return dataclasses.replace(self, **kw)


@dataclasses.dataclass(frozen=True)
class Workload:
    """One decode-loop workload: target + PARD draft + batch / prompt / K."""
    name: str
    target: ModelShape
    draft: ModelShape
    batch: int
    prompt_len: Optional[int]            # fixed length, or None: drawn per sequence
    prompt_len_range: Optional[Tuple[int, int]]
    K: int
    n_new: int
    sample: bool
    temperature: float
    page_size: int
    seed: int
    norm_jitter: float = 0.0             # 0: norm gains are 1.0
    prompt_lens_given: Optional[Tuple[int, ...]] = None  # one length per sequence (overrides the two above)

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    def prompt_lens(self) -> List[int]:
        if self.prompt_lens_given is not None:
            assert len(self.prompt_lens_given) == self.batch
            return [int(x) for x in self.prompt_lens_given]
        if self.prompt_len is not None:
            return [self.prompt_len] * self.batch
        lo, hi = self.prompt_len_range
        out = np.empty(self.batch, dtype=np.int32)
        _lib().synth_uniform_int(self.seed, 3 << 48, lo, hi - lo + 1, out.ctypes.data, self.batch)
        return [int(x) for x in out]

    def prompts(self) -> List[np.ndarray]:
        """Uniform-random ids in [0, V-1), which excludes the mask id V-1."""
        out = []
        V = self.target.vocab
        assert self.target.mask_id == V - 1 and self.draft.mask_id == V - 1
        for b, L in enumerate(self.prompt_lens()):
            ids = np.empty(L, dtype=np.int32)
            _lib().synth_uniform_int(self.seed, (2 << 48) + b, 0, V - 1, ids.ctypes.data, L)
            out.append(ids)
        return out

    def pages_per_seq(self, prompt_len: int) -> int:
        """Pages reserved per sequence and model: prompt + new tokens + 2K."""
        return -(-(prompt_len + self.n_new + 2 * self.K) // self.page_size)

    def n_pages(self) -> int:
        return sum(self.pages_per_seq(L) for L in self.prompt_lens())

    def page_order(self, model_tag: int, n_pages: Optional[int] = None) -> np.ndarray:
        """Seeded permutation of the page pool, so that no kernel can assume
        that a sequence's pages are contiguous."""
        n = self.n_pages() if n_pages is None else n_pages
        out = np.empty(n, dtype=np.int32)
        _lib().synth_permutation(self.seed, (4 << 48) + model_tag, out.ctypes.data, n)
        return out


def _llama_tiny(n_layers: int) -> ModelShape:
    return ModelShape(n_layers, 256, 4, 2, 64, 688, 2048, 10000.0, 1e-5, 2047)


TARGET_8B = ModelShape(32, 4096, 32, 8, 128, 14336, 128256, 500000.0, 1e-5, 128255)
DRAFT_1B = ModelShape(16, 2048, 32, 8, 64, 8192, 128256, 500000.0, 1e-5, 128255)
TARGET_70B = ModelShape(80, 8192, 64, 8, 128, 28672, 128256, 500000.0, 1e-5, 128255)

WORKLOADS: Dict[str, Workload] = {
    # tiny check: 4-layer target, 2-layer draft, greedy
    "tiny": Workload("tiny", _llama_tiny(4), _llama_tiny(2), 1, 32, None, 4, 16, False, 1.0, 16, 1000),
    # 8B-shaped target, 1B-shaped draft, batch 1, greedy, K=8
    "8b_greedy": Workload("8b_greedy", TARGET_8B, DRAFT_1B, 1, 512, None, 8, 256, False, 1.0, 16, 1001),
    # same models, speculative sampling at T=1, K=6
    "8b_sample": Workload("8b_sample", TARGET_8B, DRAFT_1B, 1, 1024, None, 6, 256, True, 1.0, 16, 1002),
    # same models, batch 16 with ragged prompts in [128, 2048], K=6
    "8b_batch16": Workload("8b_batch16", TARGET_8B, DRAFT_1B, 16, None, (128, 2048), 6, 128, False, 1.0, 16, 1003),
    # 70B-shaped target, 1B-shaped draft, context 4096, K=8
    "70b_greedy": Workload("70b_greedy", TARGET_70B, DRAFT_1B, 1, 4096, None, 8, 128, False, 1.0, 16, 1004),
}
WORKLOAD_ORDER = ["tiny", "8b_greedy", "8b_sample", "8b_batch16", "70b_greedy"]


# --------------------------------------------------------------------------
# Weights
# --------------------------------------------------------------------------
def tensor_tag(model_tag: int, layer: int, name: str) -> int:
    if layer < 0:
        idx = GLOBAL_TENSORS.index(name)
        return (model_tag << 40) + idx
    return (model_tag << 40) + ((layer + 1) << 8) + LAYER_TENSORS.index(name)


def fill_tensor(shape: ModelShape, seed: int, model_tag: int, layer: int, name: str,
                out_ptr: int, numel: int, std: float = 0.02, norm_jitter: float = 0.0) -> None:
    """Write one bf16 tensor (as uint16 bits) to host memory at ``out_ptr``.
    Norm gains are 1.0, or 1 + N(0, norm_jitter^2) when a jitter is given."""
    lib = _lib()
    if name.endswith("norm"):
        if norm_jitter == 0.0:
            lib.synth_fill_bf16(BF16_ONE, out_ptr, numel)
        else:
            tmp = np.empty(numel, dtype=np.uint16)
            lib.synth_normal_bf16(seed, tensor_tag(model_tag, layer, name), norm_jitter,
                                  tmp.ctypes.data, numel)
            g = bf16_to_f32(tmp) + 1.0
            ctypes.memmove(out_ptr, f32_to_bf16(g).ctypes.data, 2 * numel)
        return
    lib.synth_normal_bf16(seed, tensor_tag(model_tag, layer, name), std, out_ptr, numel)


def tensor(shape: ModelShape, seed: int, model_tag: int, layer: int, name: str,
           norm_jitter: float = 0.0) -> np.ndarray:
    dims = shape.tensor_shape(name)
    out = np.empty(dims, dtype=np.uint16)
    fill_tensor(shape, seed, model_tag, layer, name, out.ctypes.data, out.size,
                norm_jitter=norm_jitter)
    return out


def iter_tensors(shape: ModelShape) -> Iterator[Tuple[int, str]]:
    """(layer, name) for every tensor; layer -1 marks the global tensors."""
    for n in GLOBAL_TENSORS:
        yield -1, n
    for l in range(shape.n_layers):
        for n in LAYER_TENSORS:
            yield l, n


def model_weights(shape: ModelShape, seed: int, model_tag: int, norm_jitter: float = 0.0) -> dict:
    """All tensors of one model as bf16 bit arrays (uint16):
    {'embed','final_norm','lm_head','layers': [ {name: array} ]}."""
    w = {"layers": [dict() for _ in range(shape.n_layers)]}
    for layer, name in iter_tensors(shape):
        t = tensor(shape, seed, model_tag, layer, name, norm_jitter)
        if layer < 0:
            w[name] = t
        else:
            w["layers"][layer][name] = t
    return w


def workload_weights(wl: Workload) -> Tuple[dict, dict]:
    return (model_weights(wl.target, wl.seed, TARGET, wl.norm_jitter),
            model_weights(wl.draft, wl.seed, DRAFT, wl.norm_jitter))


# --------------------------------------------------------------------------
# bf16 bit helpers (storage only)
# --------------------------------------------------------------------------
def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def random_normal_f32(seed: int, tag: int, shape: Sequence[int], std: float = 1.0) -> np.ndarray:
    """Seeded N(0, std^2) values rounded through bf16 (for per-op test inputs)."""
    n = int(np.prod(shape))
    bits = np.empty(n, dtype=np.uint16)
    _lib().synth_normal_bf16(seed, (5 << 48) + tag, std, bits.ctypes.data, n)
    return bf16_to_f32(bits).reshape(shape)


def random_ints(seed: int, tag: int, lo: int, hi_exclusive: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.int32)
    _lib().synth_uniform_int(seed, (6 << 48) + tag, lo, hi_exclusive - lo, out.ctypes.data, n)
    return out


# --------------------------------------------------------------------------
# Upload to a CUDA device (torch is used for memory only)
# --------------------------------------------------------------------------
def device_weights(shape: ModelShape, seed: int, model_tag: int, device="cuda", norm_jitter: float = 0.0,
                   host: Optional[dict] = None) -> dict:
    """Same tensors as ``model_weights``, as contiguous bf16 CUDA tensors.
    Generated tensor by tensor into one pinned staging buffer (or taken from
    ``host`` when given) so host memory stays at one tensor."""
    import torch
    biggest = max(int(np.prod(shape.tensor_shape(n))) for _, n in iter_tensors(shape))
    staging = None if host is not None else torch.empty(biggest, dtype=torch.int16, pin_memory=True)
    out = {"layers": [dict() for _ in range(shape.n_layers)]}
    for layer, name in iter_tensors(shape):
        dims = shape.tensor_shape(name)
        numel = int(np.prod(dims))
        dev = torch.empty(dims, dtype=torch.bfloat16, device=device)
        if host is not None:
            src = host[name] if layer < 0 else host["layers"][layer][name]
            dev.view(torch.int16).copy_(torch.from_numpy(np.ascontiguousarray(src).view(np.int16)))
        else:
            fill_tensor(shape, seed, model_tag, layer, name, staging.data_ptr(), numel, norm_jitter=norm_jitter)
            dev.view(torch.int16).view(-1).copy_(staging[:numel])
        if layer < 0:
            out[name] = dev
        else:
            out["layers"][layer][name] = dev
    return out
