"""Seeded synthetic inputs shaped like the attribution runs Bergson targets.

This module only draws random tensors and describes shapes; it holds none of
the method's arithmetic, so both the CUDA path and the CPU oracle can be fed
from it.  Every draw comes from a ``torch.Generator`` seeded explicitly.

Workloads (module lists follow the Pythia and Llama layer shapes):
  tiny        one Linear 64->64, B=8, T=32, k=16, second moments on
  pythia160m  12 blocks x {qkv 768->2304, out 768->768, mlp 768->3072,
              3072->768}, B=32, T=2048, ~10% right padding, k=16
  pythia1b4   24 blocks x {2048->6144, 2048->2048, 2048->8192, 8192->2048},
              B=16, T=2048, no padding, k=32, second moments on, one block at
              a time
  llama8b     32 blocks x {4096->6144, 4096->4096, 4096->14336 (gate),
              4096->14336 (up), 14336->4096}, B=8, T=4096, k=16, one block at
              a time; gate and up read the same input (one A tensor)
  score4m     fp16 store 4,000,000 x 8192, 1024 queries, top-100
"""
from __future__ import annotations

import dataclasses

import torch


@dataclasses.dataclass(frozen=True)
class ModuleSpec:
    name: str
    d_in: int
    d_out: int
    shares_input: bool = False   # reads the same input tensor as the module before it


@dataclasses.dataclass(frozen=True)
class CollectWorkload:
    name: str
    modules: tuple
    B: int
    T: int
    k: int
    max_pad: int          # right padding per example drawn from U{0..max_pad}; 0 = no mask
    second_moments: bool
    blocks: int           # modules are grouped per transformer block (streaming unit)
    input_scale: bool     # A ~ N(0,1)/sqrt(d_in), G ~ N(0,1)/sqrt(d_out) when True

    @property
    def modules_per_block(self) -> int:
        return len(self.modules) // self.blocks

    @property
    def k_total(self) -> int:
        return len(self.modules) * self.k * self.k

    def block_modules(self, blk: int):
        n = self.modules_per_block
        return self.modules[blk * n:(blk + 1) * n]

    def col_offset(self, module_index: int) -> int:
        return module_index * self.k * self.k


def _blocks(n_blocks, shapes):
    mods = []
    for b in range(n_blocks):
        for shape in shapes:
            name, di, do = shape[:3]
            mods.append(ModuleSpec(f"h{b}.{name}", di, do, *shape[3:]))
    return tuple(mods)


def input_bytes(specs, tokens: int) -> int:
    """bf16 bytes of distinct A and G tensors of `tokens` tokens (a shared input counts once)."""
    dims = sum(s.d_out + (0 if s.shares_input else s.d_in) for s in specs)
    return 2 * dims * tokens


TINY = CollectWorkload("tiny: Linear 64->64, B=8, T=32, k=16, Adafactor r,c",
                       (ModuleSpec("linear", 64, 64),), 8, 32, 16, 0, True, 1, False)

PYTHIA160M = CollectWorkload(
    "pythia160m-shaped: 12 blocks x {768->2304, 768->768, 768->3072, 3072->768}, "
    "B=32, T=2048, ~10% right padding, k=16",
    _blocks(12, [("qkv", 768, 2304), ("attn_out", 768, 768), ("mlp_up", 768, 3072),
                 ("mlp_down", 3072, 768)]),
    32, 2048, 16, 409, False, 12, True)

PYTHIA1B4 = CollectWorkload(
    "pythia1.4b-shaped: 24 blocks x {2048->6144, 2048->2048, 2048->8192, 8192->2048}, "
    "B=16, T=2048, k=32, Adafactor r,c, one block per call",
    _blocks(24, [("qkv", 2048, 6144), ("attn_out", 2048, 2048), ("mlp_up", 2048, 8192),
                 ("mlp_down", 8192, 2048)]),
    16, 2048, 32, 0, True, 24, True)

LLAMA8B = CollectWorkload(
    "llama8b-shaped: 32 blocks x {4096->6144, 4096->4096, 4096->14336 x2, 14336->4096}, "
    "B=8, T=4096, k=16, one block per call, gate and up share their input",
    _blocks(32, [("qkv", 4096, 6144), ("attn_out", 4096, 4096), ("gate", 4096, 14336),
                 ("up", 4096, 14336, True), ("down", 14336, 4096)]),
    8, 4096, 16, 0, False, 32, True)

COLLECT_WORKLOADS = {"tiny": TINY, "pythia160m": PYTHIA160M, "pythia1b4": PYTHIA1B4,
                     "llama8b": LLAMA8B}


@dataclasses.dataclass(frozen=True)
class ScoreWorkload:
    name: str
    N: int
    K: int
    Q: int
    topk: int


SCORE4M = ScoreWorkload("score4m: fp16 store 4,000,000 x 8192, Q=1024, top-100",
                        4_000_000, 8192, 1024, 100)


def generator(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def layer_inputs(spec: ModuleSpec, B: int, T: int, seed: int, device="cpu",
                 input_scale: bool = False):
    """A [B, T, d_in] and G [B, T, d_out], bf16, N(0,1) (optionally / sqrt(d))."""
    g = generator(seed, device)
    A = torch.randn((B, T, spec.d_in), generator=g, device=device, dtype=torch.float32)
    G = torch.randn((B, T, spec.d_out), generator=g, device=device, dtype=torch.float32)
    if input_scale:
        A.mul_(spec.d_in ** -0.5)
        G.mul_(spec.d_out ** -0.5)
    return A.to(torch.bfloat16), G.to(torch.bfloat16)


def module_inputs(specs, B: int, T: int, seeds, device="cpu", input_scale: bool = False):
    """[(A, G)] per module as layer_inputs draws them, except that a module with
    shares_input takes the previous module's A tensor itself (same storage)."""
    out = []
    for spec, seed in zip(specs, seeds):
        A, G = layer_inputs(spec, B, T, seed=seed, device=device, input_scale=input_scale)
        if spec.shares_input:
            if not out or out[-1][0].shape[-1] != spec.d_in:
                raise ValueError(f"{spec.name}: no preceding module with d_in={spec.d_in}")
            A = out[-1][0]
        out.append((A, G))
    return out


def right_padding_mask(B: int, T: int, max_pad: int, seed: int, device="cpu"):
    """u8 [B, T]: example b keeps its first T - pad_b tokens, pad_b ~ U{0..max_pad}."""
    g = generator(seed, "cpu")
    pad = torch.randint(0, max_pad + 1, (B,), generator=g)
    t = torch.arange(T)
    mask = (t[None, :] < (T - pad)[:, None]).to(torch.uint8)
    return mask.to(device)


def second_moments(d_out: int, d_in: int, seed: int, device="cpu"):
    """Factored second moments r [d_out], c [d_in] ~ U(0.5, 2), fp32."""
    g = generator(seed, "cpu")
    r = torch.rand((d_out,), generator=g) * 1.5 + 0.5
    c = torch.rand((d_in,), generator=g) * 1.5 + 0.5
    return r.to(device), c.to(device)


def gaussian_rows(n: int, K: int, seed: int, device="cpu", dtype=torch.float32):
    """n rows of N(0, I_K) (not normalised), e.g. queries or raw store rows."""
    g = generator(seed, device)
    return torch.randn((n, K), generator=g, device=device, dtype=dtype)


def planted_rows(queries: torch.Tensor, per_query: int, seed: int):
    """Rows x = t * q + n with n ~ N(0, I) and t spread over [0.35, 2.0].

    Their cosine to q is about t / sqrt(1 + t^2), i.e. 0.33 .. 0.89, far above
    the ~0.06 maximum cosine of independent Gaussian rows at K = 8192.
    Returns rows [Q * per_query, K] (query-major) on the queries' device.
    """
    Q, K = queries.shape
    g = generator(seed, queries.device)
    t = torch.linspace(2.0, 0.35, per_query, device=queries.device)
    noise = torch.randn((Q, per_query, K), generator=g, device=queries.device,
                        dtype=queries.dtype)
    rows = t[None, :, None] * queries[:, None, :] + noise
    return rows.reshape(Q * per_query, K)


def planted_positions(N: int, Q: int, per_query: int, seed: int):
    """Distinct store row indices [Q, per_query] for the planted rows."""
    g = generator(seed, "cpu")
    perm = torch.randperm(N, generator=g)[: Q * per_query]
    return perm.reshape(Q, per_query)
