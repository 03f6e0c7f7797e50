"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds no arithmetic of the method: it only draws random vectors.
Both the CUDA path and the CPU oracle consume exactly the fp32 arrays made
here, so the two sides always see identical inputs.

Shapes follow the paper: D = 768 (bge-base-en-v1.5 embeddings, Tab. "config"),
unit-normalised rows whose coordinate RMS 1/sqrt(768) = 0.0361 matches the
measured sigma of the encoder's output (App. "Band-width study"), and memory
sizes equal to the paper's corpus counts (27,986 chunks; 361,802 records).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np
import torch

D_EMBED = 768
SEED_MEMORY = 0
SEED_QUERY = 1


def _gen(seed: int, device: str = "cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def unit_rows(n: int, d: int = D_EMBED, seed: int = SEED_MEMORY) -> np.ndarray:
    """n rows of i.i.d. N(0, 1) entries, each row scaled to unit L2 norm."""
    x = torch.randn(n, d, generator=_gen(seed), dtype=torch.float32)
    x = x / x.norm(dim=1, keepdim=True).clamp_min(1e-30)
    return x.numpy()


def planted_rows(n: int, d: int = D_EMBED, seed: int = SEED_MEMORY,
                 frac: float = 0.05, sigma: float = 0.01) -> np.ndarray:
    """Unit rows where a fraction are near-duplicates of other rows.

    A planted row j is normalise(row_src + N(0, sigma^2 I)), src drawn
    uniformly among the rows that are not planted.
    """
    g = _gen(seed)
    x = torch.randn(n, d, generator=g, dtype=torch.float32)
    x = x / x.norm(dim=1, keepdim=True).clamp_min(1e-30)
    n_plant = int(round(frac * n))
    perm = torch.randperm(n, generator=g)
    planted = perm[:n_plant]
    sources = perm[n_plant:]
    pick = torch.randint(0, sources.numel(), (n_plant,), generator=g)
    src = sources[pick]
    noise = torch.randn(n_plant, d, generator=g, dtype=torch.float32) * sigma
    y = x[src] + noise
    x[planted] = y / y.norm(dim=1, keepdim=True).clamp_min(1e-30)
    return x.numpy()


def flat_values(n: int, seed: int = SEED_MEMORY, d_scale: int = D_EMBED) -> np.ndarray:
    """n values ~ N(0, 1/d_scale) clipped to [-1, 1] (flat quantize microbench)."""
    x = torch.randn(n, generator=_gen(seed), dtype=torch.float32)
    x = (x * (1.0 / math.sqrt(d_scale))).clamp_(-1.0, 1.0)
    return x.numpy()


def queries(b: int, d: int = D_EMBED, seed: int = SEED_QUERY) -> np.ndarray:
    """b unit-normalised Gaussian query vectors."""
    return unit_rows(b, d, seed)


def unit_rows_device(n: int, d: int, seed: int, device) -> torch.Tensor:
    """Unit Gaussian rows drawn directly on a CUDA device (large memories).

    Used where the fp32 memory is too large to draw on the host; the oracle
    side then reads back the sampled rows it checks.
    """
    g = _gen(seed, device=str(device))
    x = torch.randn(n, d, generator=g, dtype=torch.float32, device=device)
    x /= x.norm(dim=1, keepdim=True).clamp_min(1e-30)
    return x


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: memory size, query batches, eps sweep, metric."""
    name: str
    n: int
    d: int
    batches: tuple
    eps: tuple
    width: int          # 0 = narrowest width that holds the codes
    metric: int         # 0 inner product, 1 cosine, 2 squared L2
    k: int
    planted: bool = False
    slab_rows: int = 0  # >0: memory drawn and quantized in slabs of this many rows
    notes: str = field(default="")


WORKLOADS = {
    "pr1_n4096_cos": Workload("pr1_n4096_cos", 4096, 768, (16,), (1e-3,), 2, 1, 10,
                              notes="unit Gaussian rows, int16 codes, cosine top-10"),
    "chunks_n27986_ip": Workload("chunks_n27986_ip", 27986, 768, (1024,),
                                 (1e-2, 1e-3, 1e-4), 0, 0, 10, planted=True,
                                 notes="5% planted near-duplicates, narrowest width"),
    "flat_2p26": Workload("flat_2p26", 1 << 26, 1, (), (1e-2, 1e-3, 1e-4), 0, 0, 0,
                          notes="flat N(0,1/768) clipped values, quantize+dequant"),
    "records_n361802_ip": Workload("records_n361802_ip", 361802, 768, (1, 64, 4096),
                                   (1e-3,), 2, 0, 10,
                                   notes="int16 codes, inner-product top-10"),
    "mem_n8388608_l2": Workload("mem_n8388608_l2", 8388608, 768, (1, 256), (1e-2,), 1,
                                2, 100, slab_rows=1 << 20,
                                notes="int8 codes quantized in 1M-row slabs, L2 top-100"),
}
