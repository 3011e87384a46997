"""Seeded synthetic workloads: shapes, sizes and random inputs only.

This module holds none of the method's arithmetic.  It serves both the CUDA
path (bench, tests) and the oracle (tests), so that both see the same inputs.
The shapes follow the five evaluation configurations of the adapter hot path;
the paper's GLUE / Alpaca / ImageNet data are replaced by N(0, 1) activations
of the same shapes (Sec. 4: RoBERTa q/v adapters, Llama q/v/k/o, ViT blocks).

Seeds: support seed 1 per (m, n) shape (101 + matrix index with per-layer
supports); C values seed 2 + matrix index; X seed 3 (+ matrix index); dY
seed 4 (+ matrix index); W0 seed 5.
"""
from __future__ import annotations

from dataclasses import dataclass, field

UNIFORM, ZIPF_ROWS, BLOCKDIAG = 0, 1, 2


@dataclass(frozen=True)
class MatSpec:
    name: str
    n: int   # in features
    m: int   # out features


@dataclass(frozen=True)
class Workload:
    name: str
    mats: tuple
    N: int                       # tokens per matrix
    nnz: int                     # support size per shape
    dtype: str                   # "f32" or "bf16" activations
    c_std: float                 # C values ~ N(0, c_std)
    support_mode: int = UNIFORM
    zipf_s: float = 1.1
    k: int = 16                  # subspaces of every frame; rho = d / k
    alpha: float = 200.0         # s = alpha / sqrt(m n)  (Sec. 4 instruction tuning uses alpha = 200)
    merge_tenants: int = 0
    merge_shape: tuple = ()      # (m, n) of the merged W0
    w0_std: float = 0.02
    support_seed: int = 1
    per_layer_support: bool = False  # one support per matrix instead of one per shape
    frames: tuple = ()           # (d, k, rho) frame parameters overriding k = 16, rho = d / 16 for dimension d
    notes: str = ""

    def shapes(self):
        """Distinct (m, n) shapes in first-seen order."""
        out = []
        for s in self.mats:
            if (s.m, s.n) not in out:
                out.append((s.m, s.n))
        return out

    def dims(self):
        out = []
        for s in self.mats:
            for d in (s.n, s.m):
                if d not in out:
                    out.append(d)
        return out


def _layers(nl, per_layer):
    return tuple(MatSpec(f"l{i}.{nm}", n, m) for i in range(nl) for (nm, n, m) in per_layer)


WORKLOADS = {
    "single_256_fp32": Workload(
        "single_256_fp32", (MatSpec("w", 256, 256),), N=8, nnz=128, dtype="f32", c_std=0.02,
        merge_tenants=4, merge_shape=(256, 256),
        notes="one 256x256 layer, 16 subspaces of dim 16, fp32; forward, dX, dC and merge"),
    "roberta_base_qv": Workload(
        "roberta_base_qv", _layers(12, [("q", 768, 768), ("v", 768, 768)]), N=32 * 128, nnz=1000, dtype="bf16",
        c_std=0.02, notes="RoBERTa-base q/v adapters, 32 sequences x 128 tokens"),
    "llama2_7b_qkvo": Workload(
        "llama2_7b_qkvo", _layers(32, [("q", 4096, 4096), ("k", 4096, 4096), ("v", 4096, 4096), ("o", 4096, 4096)]),
        N=4 * 2048, nnz=4096, dtype="bf16", c_std=0.01,
        notes="LLaMA-2-7B q/k/v/o adapters, 4 sequences x 2048 tokens, fused fwd + dX + dC"),
    "llama3_8b_all": Workload(
        "llama3_8b_all", _layers(32, [("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
                                      ("gate", 4096, 14336), ("up", 4096, 14336), ("down", 14336, 4096)]),
        N=16384, nnz=8192, dtype="bf16", c_std=0.01, support_mode=ZIPF_ROWS, zipf_s=1.1,
        notes="LLaMA-3-8B attention (GQA k/v) and MLP adapters, Zipf(1.1) rows of C, 16384 tokens"),
    "vit_b16_merge": Workload(
        "vit_b16_merge", _layers(12, [("q", 768, 768), ("k", 768, 768), ("v", 768, 768), ("proj", 768, 768),
                                      ("fc1", 768, 3072), ("fc2", 3072, 768)]),
        N=64 * 197, nnz=2000, dtype="bf16", c_std=0.02, merge_tenants=64, merge_shape=(768, 768),
        notes="ViT-B/16 blocks, 64 images x 197 tokens; merge of 64 tenants over a 768x768 W0"),
}

# Support variants of the scope table's next rows, at RoBERTa shapes: supports
# restricted to the k diagonal blocks (Sec. 3.3), and one support per layer
# instead of one per shape.
WORKLOADS["roberta_blockdiag"] = Workload(
    "roberta_blockdiag", _layers(2, [("q", 768, 768), ("v", 768, 768), ("fc1", 768, 3072)]), N=4096, nnz=1000,
    dtype="bf16", c_std=0.02, support_mode=BLOCKDIAG,
    notes="supports uniform inside the 16 diagonal blocks of C")
WORKLOADS["roberta_zipf"] = Workload(
    "roberta_zipf", _layers(2, [("q", 768, 768), ("v", 768, 768)]), N=4096, nnz=1000, dtype="bf16", c_std=0.02,
    support_mode=ZIPF_ROWS, zipf_s=1.1,
    notes="heavy-tailed Zipf(1.1) rows at RoBERTa shapes: long runs split over chunks (overflow and fix-up)")
WORKLOADS["roberta_per_layer"] = Workload(
    "roberta_per_layer", _layers(3, [("q", 768, 768), ("v", 768, 768)]), N=4096, nnz=1000, dtype="bf16",
    c_std=0.02, per_layer_support=True, notes="a distinct uniform support for every matrix")

# The paper's own frame regime, rho = 2 (k = d / 2 subspaces of real dimension
# 2, k*rho = d): every frame is one dense realified DFT of size d / 2
# (Sec. 4 fine-tuning setup and the subspace-dimension ablation), at the
# LLaMA-2 and RoBERTa shapes; and redundant frames with T blocks (k*rho > d,
# the (6,3,11)-style construction of the appendix) at small odd shapes.
WORKLOADS["llama2_rho2"] = Workload(
    "llama2_rho2", _layers(32, [("q", 4096, 4096), ("k", 4096, 4096), ("v", 4096, 4096), ("o", 4096, 4096)]),
    N=4 * 2048, nnz=4096, dtype="bf16", c_std=0.01, frames=((4096, 2048, 2),),
    notes="LLaMA-2-7B q/k/v/o adapters with rho = 2 frames (dense DFT_2048 per token)")
WORKLOADS["roberta_rho2"] = Workload(
    "roberta_rho2", _layers(12, [("q", 768, 768), ("v", 768, 768)]), N=32 * 128, nnz=1000, dtype="bf16",
    c_std=0.02, frames=((768, 384, 2),), notes="RoBERTa-base q/v adapters with rho = 2 frames (dense DFT_384)")
WORKLOADS["tblock_tff"] = Workload(
    "tblock_tff", (MatSpec("a", 40, 22), MatSpec("b", 46, 46), MatSpec("c", 22, 40)), N=300, nnz=200,
    dtype="bf16", c_std=0.02, frames=((40, 7, 8), (22, 6, 6), (46, 10, 10)),
    notes="redundant tight fusion frames with T blocks: (d, k, rho) = (40, 7, 8), (22, 6, 6), (46, 10, 10)")

# The configuration the headline metric is quoted on.
HEADLINE = "llama2_7b_qkvo"


def frame_params(w: Workload, d: int):
    """(k, rho) of the frame of dimension d in workload w."""
    for dd, k, rho in w.frames:
        if dd == d:
            return k, rho
    return w.k, d // w.k


def coef_dims(w: Workload, spec: MatSpec):
    """(K_m, K_n): rows and columns of C (frame columns k*rho of each side)."""
    km, rm = frame_params(w, spec.m)
    kn, rn = frame_params(w, spec.n)
    return km * rm, kn * rn


def support_key(w: Workload, mat_index: int):
    """Key of the support (and plan) matrix `mat_index` uses: its shape, or
    the matrix itself with per-layer supports."""
    spec = w.mats[mat_index]
    return (spec.m, spec.n, mat_index) if w.per_layer_support else (spec.m, spec.n)


def support_seed_of(w: Workload, mat_index: int) -> int:
    return w.support_seed + (100 + mat_index if w.per_layer_support else 0)


def scale_of(w: Workload, spec: MatSpec) -> float:
    return w.alpha / (spec.m * spec.n) ** 0.5


# ---------------------------------------------------------------------------
# seeded random tensors (torch Philox / CPU generators)
# ---------------------------------------------------------------------------
def normal(shape, seed: int, std: float = 1.0, dtype=None, device="cpu"):
    """N(0, std^2) tensor from a seeded torch generator on `device`, cast to dtype."""
    import torch
    dtype = dtype or torch.float32
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(dtype)


def torch_dtype(w: Workload):
    import torch
    return torch.float32 if w.dtype == "f32" else torch.bfloat16


def c_values(w: Workload, mat_index: int, device="cpu"):
    return normal((w.nnz,), 2 + mat_index, w.c_std, device=device)


def x_input(w: Workload, mat_index: int, N: int | None = None, device="cpu"):
    spec = w.mats[mat_index]
    return normal((w.N if N is None else N, spec.n), 3 + 1000 * mat_index, 1.0, torch_dtype(w), device)


def dy_input(w: Workload, mat_index: int, N: int | None = None, device="cpu"):
    spec = w.mats[mat_index]
    return normal((w.N if N is None else N, spec.m), 4 + 1000 * mat_index, 1.0, torch_dtype(w), device)


def w0_input(w: Workload, device="cpu"):
    m, n = w.merge_shape
    return normal((m, n), 5, w.w0_std, torch_dtype(w), device)


def merge_c_values(w: Workload, device="cpu"):
    return normal((w.merge_tenants, w.nnz), 6, w.c_std, device=device)
