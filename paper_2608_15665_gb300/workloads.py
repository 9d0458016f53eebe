"""Synthetic workloads of the SubZero+ weight path and their seeded input generators.

This module holds shapes, hyper-parameters and random INPUTS only (initial
weights and the per-step loss values that stand in for the caller's forward
passes); it contains none of the method's arithmetic.  Inputs come from
PyTorch's / numpy's own generators, not from the method's Philox contract.

The paper fine-tunes OPT, LLaMA and Qwen checkpoints on SuperGLUE (Sec. 5.1,
App. A.2); neither the weights nor the datasets are used here.  Each workload
keeps the SHAPES of such a model's trainable matrices (nn.Linear [out, in]),
weights drawn i.i.d. N(0, 0.02^2), and losses L = 2.0 + 0.01 N(0, 1) per
evaluation, which is what the weight path sees of a real run.
"""

from dataclasses import dataclass, field

import numpy as np


@dataclass
class Workload:
    name: str
    shapes: list            # [(m, n), ...] per trainable matrix, row-major W is m x n
    dtype: str              # "bf16" or "f32" weight storage
    r: int
    q: int
    eps: float
    lr: float
    beta1: float
    beta2: float
    eps_adam: float
    steps: int
    F: int                  # subspace refresh period (Alg. 3: refresh when t mod F == 0)
    seed: int
    zero_init: list = field(default_factory=list)   # indices of matrices initialised to zero
    note: str = ""

    @property
    def n_mats(self):
        return len(self.shapes)

    @property
    def params(self):
        return int(sum(m * n for m, n in self.shapes))

    @property
    def elem_bytes(self):
        return 2 if self.dtype == "bf16" else 4

    def bytes_per_pass(self):
        """Algorithmic HBM bytes of one weight pass: read and write every element of W once."""
        return 2 * self.elem_bytes * self.params


def _opt13b_lora_shapes():
    shapes, zero = [], []
    for _layer in range(40):
        for _proj in ("q", "v"):
            shapes.append((8, 5120))        # LoRA A: r_L x in, ~N(0, 0.02)
            shapes.append((5120, 8))        # LoRA B: out x r_L, zero at init
            zero.append(len(shapes) - 1)
    return shapes, zero


def _build():
    wl = {}
    wl["single256_f32_r8"] = Workload(
        "single256_f32_r8", [(256, 256)], "f32", r=8, q=4, eps=1e-3, lr=1e-4, beta1=0.9,
        beta2=0.999, eps_adam=1e-8, steps=10, F=5, seed=1001,
        note="one fp32 256x256 matrix, 10 steps, refresh at steps 0 and 5")
    opt = []
    for _ in range(24):
        opt += [(2048, 2048)] * 4 + [(8192, 2048), (2048, 8192)]
    wl["opt1.3b_bf16_r16"] = Workload(
        "opt1.3b_bf16_r16", opt, "bf16", r=16, q=4, eps=1e-3, lr=1e-3, beta1=0.9, beta2=0.95,
        eps_adam=1e-8, steps=100, F=50, seed=1002,
        note="OPT-1.3B shapes: 24 x {q,k,v,o 2048x2048, fc1 8192x2048, fc2 2048x8192}")
    llama = []
    for _ in range(32):
        llama += [(4096, 4096)] * 4 + [(11008, 4096)] * 2 + [(4096, 11008)]
    wl["llama7b_bf16_r32"] = Workload(
        "llama7b_bf16_r32", llama, "bf16", r=32, q=4, eps=1e-3, lr=1e-3, beta1=0.9, beta2=0.95,
        eps_adam=1e-8, steps=50, F=25, seed=1003,
        note="LLaMA-7B shapes: 32 x {q,k,v,o 4096x4096, gate,up 11008x4096, down 4096x11008}")
    lora, zero = _opt13b_lora_shapes()
    wl["lora_opt13b_f32_r4"] = Workload(
        "lora_opt13b_f32_r4", lora, "f32", r=4, q=8, eps=1e-3, lr=1e-2, beta1=0.9, beta2=0.95,
        eps_adam=1e-8, steps=200, F=50, seed=1004, zero_init=zero,
        note="OPT-13B LoRA on q,v: 40 x 2 x {A 8x5120, B 5120x8}, B zero at init")
    wl["llama7b_bf16_r128_q99"] = Workload(
        "llama7b_bf16_r128_q99", llama, "bf16", r=128, q=99, eps=1e-3, lr=1e-3, beta1=0.9,
        beta2=0.95, eps_adam=1e-8, steps=400, F=50, seed=1006,
        note="the paper's default scale (App. A.2, Table 7): r = 128, K = 99 queries, "
             "F = 50, on the LLaMA-7B shapes")
    llama13 = []
    for _ in range(40):
        llama13 += [(5120, 5120)] * 4 + [(13824, 5120), (13824, 5120), (5120, 13824)]
    wl["llama13b_bf16_r128_q99"] = Workload(
        "llama13b_bf16_r128_q99", llama13, "bf16", r=128, q=99, eps=1e-3, lr=1e-3, beta1=0.9,
        beta2=0.95, eps_adam=1e-8, steps=400, F=100, seed=1007,
        note="the paper's default scale on the LLaMA-13B shapes: 40 x {q,k,v,o 5120x5120, "
             "gate,up 13824x5120, down 5120x13824}, r = 128, K = 99, F = 100")
    big = []
    for _ in range(64):
        big += [(8192, 5120), (1024, 5120), (1024, 5120), (5120, 8192),
                (25600, 5120), (25600, 5120), (5120, 25600)]
    wl["dense32b_bf16_r64"] = Workload(
        "dense32b_bf16_r64", big, "bf16", r=64, q=8, eps=1e-3, lr=1e-3, beta1=0.9, beta2=0.95,
        eps_adam=1e-8, steps=10, F=5, seed=1005,
        note="32B shapes: 64 x {q 8192x5120, k,v 1024x5120, o 5120x8192, gate,up 25600x5120, down 5120x25600}")
    return wl


WORKLOADS = _build()


def get(name):
    return WORKLOADS[name]


def loss_table(wl, scheme, steps=None, start=0):
    """Per-step fp32 losses standing in for the forward passes: 2.0 + 0.01 N(0, 1).

    central: 2q values per step (L+_0, L-_0, ...); forward: q+1 (l_0, l_1, ...); direct: q.
    Row t is the same whatever ``start``/``steps`` window is asked for.
    """
    n = {"central": 2 * wl.q, "forward": wl.q + 1, "direct": wl.q}[scheme]
    steps = wl.steps if steps is None else steps
    rows = []
    for t in range(start, start + steps):
        g = np.random.default_rng([wl.seed, t, n])
        rows.append((2.0 + 0.01 * g.standard_normal(n)).astype(np.float32))
    return np.stack(rows) if rows else np.zeros((0, n), np.float32)


def partition(wl, rank, world):
    """Layer partition of a `world`-times larger parameter set: rank `rank` owns the
    global matrix indices [rank * n_mats, (rank + 1) * n_mats) with this workload's
    shapes.  Every rank uses the same Philox seed; the global index alone selects the
    random streams, so the split changes no Z or Omega.  No data crosses ranks."""
    if not 0 <= rank < world:
        raise ValueError("rank out of range")
    base = rank * wl.n_mats
    return {"matrix_index_base": base, "global_indices": range(base, base + wl.n_mats),
            "seed": wl.seed}


def init_weight(wl, i, device="cpu", index_base=0):
    """Initial W_i: N(0, 0.02^2) in the workload dtype (zero for LoRA B), via torch's
    generator, seeded by the global matrix index index_base + i."""
    import torch
    m, n = wl.shapes[i]
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    if i in wl.zero_init:
        return torch.zeros(m, n, dtype=dt, device=device)
    g = torch.Generator(device=device)
    g.manual_seed(wl.seed * 100003 + index_base + i)
    w = torch.randn(m, n, generator=g, device=device, dtype=torch.float32)
    return w.mul_(0.02).to(dt)


def scaled(wl, name=None, **changes):
    """A copy of a workload with some fields replaced (for small parity cases)."""
    d = dict(wl.__dict__)
    d.update(changes)
    if name:
        d["name"] = name
    return Workload(**d)
