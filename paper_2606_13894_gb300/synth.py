"""Seeded synthetic inputs shaped like the workloads the Gefen paper trains.

This module holds no Gefen arithmetic: it only draws parameters and gradients
with the shapes and gradient-scale structure of the paper's models (GPT-2-125M
trained with nanoGPT, Llama 3-1.5B trained with TorchTitan; Appendix I), plus a
tiny set, a flat sweep and a refit micro-benchmark set.  None of the paper's
datasets or trained weights are used; every value comes from torch's seeded
generators (Philox on CUDA, the CPU generator on the host).

Both the CUDA path's tests and the oracle's tests draw their inputs here.

Recipe (all seeds derive from one integer ``seed`` mixed with the tensor index
and the step, so a tensor's gradient at step t is reproducible on its own):
  * parameters theta ~ N(0, 0.02^2), fp32;
  * gradients g = bf16(sigma * N(0, 1)) with a fixed per-tensor sigma
    structure (per row, per 64-wide column stripe, or per head), the sigmas
    drawn once per tensor from a log-uniform law on [1e-4, 1e-2];
  * tensors are packed into flat arenas at offsets rounded up to a multiple of
    ``ALIGN`` elements.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Sequence

import torch

ALIGN = 64  # element alignment of every tensor inside a flat arena

SIGMA_LO, SIGMA_HI = 1e-4, 1e-2


@dataclasses.dataclass(frozen=True)
class TensorSpec:
    """One parameter tensor: its shape and the structure of its gradient scale.

    structure:
      "row"        one sigma per row (last dim contiguous)
      "col64"      one sigma per 64-column stripe, shared by all rows
      "head_row"   rows grouped in heads of 64, sigma_head[r//64] * rho_r,
                   rho_r log-uniform on [1/2, 2]
      "head_col"   one sigma per 64-column stripe (per head of the input dim)
      "const"      one sigma for the whole tensor
      "const:<s>"  the fixed sigma <s> for the whole tensor
    """
    name: str
    shape: tuple
    structure: str = "row"
    period: int = 0  # prescribed block size; 0 = to be inferred

    @property
    def numel(self) -> int:
        return int(math.prod(self.shape))

    @property
    def rows(self) -> int:
        return self.shape[0] if len(self.shape) > 1 else 1

    @property
    def cols(self) -> int:
        return self.shape[-1]


def _mix(*xs: int) -> int:
    h = 0x9E3779B97F4A7C15
    for x in xs:
        h ^= (int(x) + 0x632BE59BD9B4E019 + ((h << 6) & (2**64 - 1)) + (h >> 2))
        h &= 2**64 - 1
    return h & (2**63 - 1)


def _gen(device, *key: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_mix(*key))
    return g


def _log_uniform(n, lo, hi, gen, device):
    u = torch.rand(n, generator=gen, device=device, dtype=torch.float64)
    return torch.exp(math.log(lo) + u * (math.log(hi) - math.log(lo)))


# --------------------------------------------------------------------------
# Workload definitions
# --------------------------------------------------------------------------
def tiny_set() -> List[TensorSpec]:
    """4 tensors, ~0.59M params; blocks are rows (the vector is one block)."""
    return [
        TensorSpec("w0", (256, 256), "row", period=256),
        TensorSpec("w1", (256, 1024), "row", period=1024),
        TensorSpec("w2", (1024, 256), "row", period=256),
        TensorSpec("b0", (256,), "row", period=256),
    ]


def gpt2_125m_set() -> List[TensorSpec]:
    """GPT-2-125M shapes as nanoGPT stores them (Conv1D [in, out]), no linear
    biases: tied wte, wpe, 12 x (qkv, proj, fc, fc2), LayerNorm vectors."""
    d, V, T, L = 768, 50257, 1024, 12
    specs = [TensorSpec("wte", (V, d), "col64"), TensorSpec("wpe", (T, d), "col64")]
    for i in range(L):
        specs += [
            TensorSpec(f"h{i}.ln_1.weight", (d,), "const"),
            TensorSpec(f"h{i}.ln_1.bias", (d,), "const"),
            TensorSpec(f"h{i}.attn.c_attn", (d, 3 * d), "col64"),
            TensorSpec(f"h{i}.attn.c_proj", (d, d), "col64"),
            TensorSpec(f"h{i}.ln_2.weight", (d,), "const"),
            TensorSpec(f"h{i}.ln_2.bias", (d,), "const"),
            TensorSpec(f"h{i}.mlp.c_fc", (d, 4 * d), "col64"),
            TensorSpec(f"h{i}.mlp.c_proj", (4 * d, d), "col64"),
        ]
    specs += [TensorSpec("ln_f.weight", (d,), "const"), TensorSpec("ln_f.bias", (d,), "const")]
    return specs


def llama_1p5b_set() -> List[TensorSpec]:
    """Llama-3-style ~1.5B shapes ([out, in] torch layout): d=2048, 20 layers,
    32 q / 8 kv heads of 64, SwiGLU 8192, RMSNorm vectors, tied 128256 x 2048
    embedding."""
    d, L, ffn, V, hd, nkv = 2048, 20, 8192, 128256, 64, 8
    specs = [TensorSpec("tok_embeddings", (V, d), "row")]
    for i in range(L):
        specs += [
            TensorSpec(f"l{i}.attention_norm", (d,), "const"),
            TensorSpec(f"l{i}.wq", (d, d), "head_row"),
            TensorSpec(f"l{i}.wk", (nkv * hd, d), "head_row"),
            TensorSpec(f"l{i}.wv", (nkv * hd, d), "head_row"),
            TensorSpec(f"l{i}.wo", (d, d), "head_col"),
            TensorSpec(f"l{i}.ffn_norm", (d,), "const"),
            TensorSpec(f"l{i}.w1", (ffn, d), "row"),
            TensorSpec(f"l{i}.w3", (ffn, d), "row"),
            TensorSpec(f"l{i}.w2", (d, ffn), "row"),
        ]
    specs += [TensorSpec("norm", (d,), "const")]
    return specs


def flat_set(n: int, period: int) -> List[TensorSpec]:
    """One flat fp32 tensor of n elements with gradients N(0, 1e-3^2)."""
    return [TensorSpec("flat", (n,), "const:1e-3", period=period)]


CONFIGS = {
    "tiny": tiny_set,
    "gpt2-125m": gpt2_125m_set,
    "llama-1.5b": llama_1p5b_set,
}


# --------------------------------------------------------------------------
# Arena packing and drawing
# --------------------------------------------------------------------------
def pack_offsets(specs: Sequence[TensorSpec], align: int = ALIGN):
    """Element offsets of each tensor in a flat arena, and the arena length."""
    offs, o = [], 0
    for s in specs:
        offs.append(o)
        o += (s.numel + align - 1) // align * align
    return offs, o


def _sigma_full(spec: TensorSpec, seed: int, idx: int, device) -> torch.Tensor:
    """The fixed gradient-scale field of one tensor, broadcastable to its
    (rows, cols) view."""
    gen = _gen(device, seed, idx, 0xA11CE)
    rows, cols = spec.rows, spec.cols
    st = spec.structure
    if st == "row":
        sig = _log_uniform(rows, SIGMA_LO, SIGMA_HI, gen, device)[:, None]
    elif st in ("col64", "head_col"):
        stripes = (cols + 63) // 64
        s = _log_uniform(stripes, SIGMA_LO, SIGMA_HI, gen, device)
        sig = s.repeat_interleave(64)[:cols][None, :]
    elif st == "head_row":
        heads = (rows + 63) // 64
        sh = _log_uniform(heads, SIGMA_LO, SIGMA_HI, gen, device)
        rho = _log_uniform(rows, 0.5, 2.0, gen, device)
        sig = (sh.repeat_interleave(64)[:rows] * rho)[:, None]
    elif st == "const":
        sig = _log_uniform(1, SIGMA_LO, SIGMA_HI, gen, device).view(1, 1)
    elif st.startswith("const:"):
        sig = torch.full((1, 1), float(st.split(":", 1)[1]), dtype=torch.float64, device=device)
    else:
        raise ValueError(f"unknown gradient structure {st!r}")
    return sig.to(torch.float32)


def init_params(specs, seed: int, device="cpu", out: torch.Tensor | None = None,
                align: int = ALIGN) -> torch.Tensor:
    """Flat fp32 parameter arena, theta ~ N(0, 0.02^2); padding is zero."""
    offs, total = pack_offsets(specs, align)
    if out is None:
        out = torch.zeros(total, dtype=torch.float32, device=device)
    for i, (s, o) in enumerate(zip(specs, offs)):
        gen = _gen(device, seed, i, 0x7E7A)
        out[o:o + s.numel].normal_(0.0, 0.02, generator=gen)
    return out


def draw_grads(specs, seed: int, step: int, device="cpu", out: torch.Tensor | None = None,
               align: int = ALIGN) -> torch.Tensor:
    """Flat bf16 gradient arena for one step; padding is zero."""
    offs, total = pack_offsets(specs, align)
    if out is None:
        out = torch.zeros(total, dtype=torch.bfloat16, device=device)
    for i, (s, o) in enumerate(zip(specs, offs)):
        gen = _gen(device, seed, i, step, 0x6EAD)
        sig = _sigma_full(s, seed, i, device)
        z = torch.randn((s.rows, s.cols), generator=gen, device=device, dtype=torch.float32)
        out[o:o + s.numel].copy_((z * sig).reshape(-1).to(torch.bfloat16))
    return out


def refit_values(n: int, seed: int, device="cpu", block: int = 4096,
                 outlier_frac: float = 0.01) -> torch.Tensor:
    """Normalised momentum-like values for the refit micro-benchmark.

    Student-t(nu=4) draws Z / sqrt(chi2_4 / 4); with probability
    ``outlier_frac`` a draw is replaced by +-8 sigma_t (sigma_t = sqrt(2)).
    Each run of ``block`` values is divided by its largest magnitude, so every
    block holds an exact +-1.  n must be a multiple of ``block``.
    """
    assert n % block == 0
    out = torch.empty(n, dtype=torch.float32, device=device)
    chunk = block * 65536
    for c0 in range(0, n, chunk):
        m = min(chunk, n - c0)
        gen = _gen(device, seed, c0 // chunk, 0x5EF1)
        z = torch.randn(m, generator=gen, device=device, dtype=torch.float32)
        # chi-square with 4 degrees of freedom = sum of 4 squared normals
        e = torch.randn((m, 4), generator=gen, device=device, dtype=torch.float32)
        chi2 = (e * e).sum(dim=1)
        t = z / torch.sqrt(chi2 / 4.0)
        u = torch.rand(m, generator=gen, device=device, dtype=torch.float32)
        sgn = torch.where(torch.rand(m, generator=gen, device=device) < 0.5, -1.0, 1.0)
        t = torch.where(u < outlier_frac, sgn * (8.0 * math.sqrt(2.0)), t)
        t = t.view(-1, block)
        t = t / t.abs().amax(dim=1, keepdim=True)
        out[c0:c0 + m] = t.reshape(-1)
    return out


def bf16_bits(t: torch.Tensor):
    """uint16 numpy view of a bf16 tensor's bit patterns (host copy)."""
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view("uint16")


def total_params(specs) -> int:
    return sum(s.numel for s in specs)
