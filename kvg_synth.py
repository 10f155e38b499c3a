"""Seeded synthetic inputs shaped like the paper's serving workloads.

This module holds none of the method's arithmetic: it only draws bf16 values
and integer choices from seeded generators and describes the workload
geometry.  Both sides of every parity check (the CUDA library and the CPU
oracle) receive the same bytes from here; neither regenerates them.

Workloads (the paper's models are Gemma-4-12B / Gemma-4-31B served with a
32,768-token window, Sec. 3.4 and Sec. 4.4; their weights and benchmarks are
not used, so K, V and q are N(0, 1) draws rounded to bf16):

* tiny      — 2 layers, Hq/Hkv 4/2, D 64, page 16; one 256-token block.
* 12b       — 48 layers, Hq/Hkv 16/8, D 256, page 64; an 8,192-token block
              grafted into a 32,768-token context (24,576 tokens fresh).
* batched   — 12b geometry; 32 sequences x 4 blocks of U{2048..6144} tokens
              from a 512-block store, then 64 decode steps.
* 31b       — 60 layers, Hq/Hkv 32/16, D 128, page 64, theta 1e6; a
              16,384-token block re-based by delta in {0, 1, 4096, 100000};
              batch 8 over 65,536-token contexts.
* deep      — 2-layer slice of 12b; 1,394 blocks x 2,048 tokens in pinned
              host memory; 1,000 uniform random grafts.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    page_size: int
    rope_theta: float
    seed: int

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def page_bytes(self) -> int:
        return self.n_kv_heads * self.page_size * self.head_dim * 2

    @property
    def token_bytes(self) -> int:
        """K+V bytes of one token over all layers."""
        return self.n_layers * 2 * self.n_kv_heads * self.head_dim * 2

    def with_layers(self, n_layers: int) -> "Workload":
        return dataclasses.replace(self, n_layers=n_layers)


TINY = Workload("tiny", 2, 4, 2, 64, 16, 10000.0, 0x4B5647001)
B12 = Workload("12b", 48, 16, 8, 256, 64, 10000.0, 0x4B5647002)
BATCHED = Workload("batched", 48, 16, 8, 256, 64, 10000.0, 0x4B5647003)
B31 = Workload("31b", 60, 32, 16, 128, 64, 1000000.0, 0x4B5647004)
DEEP = Workload("deep", 2, 16, 8, 256, 64, 10000.0, 0x4B5647005)

TINY_BLOCK = 256
B12_BLOCK, B12_CTX = 8192, 32768
# per-tensor scales of the fp8 (E4M3) KV variant: N(0,1) rows span roughly
# +-5, so code values up to ~80 (the E4M3 grid reaches 448)
FP8_K_SCALE, FP8_V_SCALE = 0.0625, 0.0625
BATCHED_SEQS, BATCHED_BLOCKS_PER_SEQ, BATCHED_STORE, BATCHED_STEPS = 32, 4, 512, 64
BATCHED_LEN_RANGE = (2048, 6144)
B31_BLOCK, B31_CTX, B31_BATCH = 16384, 65536, 8
B31_DELTAS = (0, 1, 4096, 100000)
DEEP_BLOCKS, DEEP_BLOCK, DEEP_GRAFTS, DEEP_CTX = 1394, 2048, 1000, 32768


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) & 0x7FFFFFFFFFFFFFFF)
    return g


def normal_bf16(shape, seed: int, device="cpu") -> torch.Tensor:
    """N(0, 1) draws rounded to bf16, as a bf16 tensor on `device`."""
    g = _gen(seed, device)
    return torch.randn(tuple(shape), generator=g, device=device, dtype=torch.float32).to(
        torch.bfloat16)


def as_u16(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit patterns (copied to host)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def from_u16(a: np.ndarray, device="cpu") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)


def kv_rows(w: Workload, n_tokens: int, seed: int, device="cpu"):
    """Prefill-shaped K and V rows: two bf16 tensors [L][n][Hkv][D]."""
    shape = (w.n_layers, n_tokens, w.n_kv_heads, w.head_dim)
    return normal_bf16(shape, seed * 2 + 1, device), normal_bf16(shape, seed * 2 + 2, device)


def queries(w: Workload, n_layers: int, batch: int, seed: int, device="cpu") -> torch.Tensor:
    """Decode queries, bf16 [L][B][Hq][D] (already position-encoded)."""
    return normal_bf16((n_layers, batch, w.n_q_heads, w.head_dim), seed * 2 + 3, device)


def positions(start: int, n: int) -> np.ndarray:
    return np.arange(start, start + n, dtype=np.int32)


def batched_plan(seed: int = BATCHED.seed, n_store: int = BATCHED_STORE):
    """Per sequence: 4 distinct block ids from the n_store-block store (512 in
    the workload; fewer for small profiling cases) and the store's block
    lengths, U{2048..6144} each."""
    rng = np.random.default_rng(seed)
    lens = rng.integers(BATCHED_LEN_RANGE[0], BATCHED_LEN_RANGE[1] + 1, size=n_store)
    ids = np.stack([rng.choice(n_store, BATCHED_BLOCKS_PER_SEQ, replace=False)
                    for _ in range(BATCHED_SEQS)])
    return lens.astype(np.int64), ids.astype(np.int64)


def deep_plan(seed: int = DEEP.seed, n_grafts: int = DEEP_GRAFTS, n_blocks: int = DEEP_BLOCKS):
    """Block index of each random-access graft, uniform over store depth."""
    rng = np.random.default_rng(seed)
    return rng.integers(0, n_blocks, size=n_grafts).astype(np.int64)


def permutation(n: int, seed: int) -> np.ndarray:
    return np.random.default_rng(seed).permutation(n).astype(np.int32)


def splitmix64(seed: int, n: int) -> np.ndarray:
    """The first n outputs of SplitMix64 seeded with `seed` (Steele, Lea and
    Flood, "Fast splittable pseudorandom number generators", 2014: the state
    advances by the golden-ratio increment, each output is the state mixed by
    two xor-shift-multiply rounds).  Integer-only, so the same bytes on every
    machine and library version."""
    with np.errstate(over="ignore"):
        z = (np.uint64(seed & 0xFFFFFFFFFFFFFFFF)
             + (np.arange(1, n + 1, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15)))
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def portable_bf16(shape, seed: int) -> np.ndarray:
    """bf16 bit patterns drawn with integer operations only (for stored
    fixtures that must not depend on a library's random generator): random
    sign, binade uniform over 2^-4 ... 2^0 (so |x| < 2, the scale of the
    N(0, 1) workloads), mantissa uniform."""
    n = int(np.prod(shape))
    r = splitmix64(seed, n)
    sign = (r & np.uint64(1)) << np.uint64(15)
    expo = (np.uint64(123) + (r >> np.uint64(8)) % np.uint64(5)) << np.uint64(7)
    mant = (r >> np.uint64(16)) & np.uint64(0x7F)
    return (sign | expo | mant).astype(np.uint16).reshape(shape)
