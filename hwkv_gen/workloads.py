"""The synthetic workloads: shapes, lengths and per-head window policies.

Inputs stand in for the paper's long-context runs (Qwen3.6-27B at 112K/128K,
the 161K capacity point): seeded generator tensors with those shapes and
lengths, no dataset content. Window levels are drawn per (layer, KV head) with
splitmix64 draws; the budget workload lowers heads one level at a time until a
target fraction of all-full residency is met.
"""
from dataclasses import dataclass, field
from typing import List, Optional

FULL = 0
_M64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15


def _mix(z):
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _M64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _M64
    return z ^ (z >> 31)


def draw(seed, stream, i):
    """i-th 64-bit draw of a splitmix64 stream keyed by (seed, stream)."""
    return _mix((((seed ^ (stream * 0xD1B54A32D192ED03)) & _M64) + (i + 1) * _GAMMA) & _M64)


@dataclass
class Workload:
    name: str
    n_layers: int
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    prompt: int              # tokens before decode
    decode_steps: int
    chunk: int               # prefill chunk length (0 = prompt filled by append only)
    levels: List[int]        # window levels the policy draws from (0 = full)
    fixed_windows: Optional[List[int]] = None  # per (layer, kv head), overrides the draw
    per_head_scale: bool = False
    seed: int = 0
    budget: Optional[float] = None  # target fraction of all-full residency (budget sweep)
    note: str = ""
    windows: List[int] = field(default_factory=list)

    @property
    def max_ctx(self):
        return self.prompt + self.decode_steps

    @property
    def group(self):
        return self.n_q_heads // self.n_kv_heads

    @property
    def n_units(self):
        return self.n_layers * self.n_kv_heads


def _drawn_windows(wl):
    return [wl.levels[draw(wl.seed, 1, u) % len(wl.levels)] for u in range(wl.n_units)]


BUDGET_LEVELS = [FULL, 65536, 32768, 16384, 8192, 4096, 2048, 512]


def budget_windows(n_units, C, target, seed, levels=BUDGET_LEVELS):
    """Start all full; visit units in a seeded shuffled order, cyclically, lowering
    each by one level until the retained fraction sum(min(W, C)) / (n_units C)
    is at most `target` (or nothing can be lowered)."""
    order = list(range(n_units))
    for i in range(n_units - 1, 0, -1):  # Fisher-Yates with splitmix64 draws
        j = draw(seed, 2, i) % (i + 1)
        order[i], order[j] = order[j], order[i]
    level = [0] * n_units

    def retained():
        return sum(C if levels[l] == FULL else min(levels[l], C) for l in level)

    k = 0
    while retained() > target * n_units * C:
        movable = [u for u in order if level[u] + 1 < len(levels)]
        if not movable:
            break
        u = order[k % n_units]
        k += 1
        if level[u] + 1 < len(levels):
            level[u] += 1
    return [levels[l] for l in level]


def make(name, budget=None):
    """The workload `name` with its window policy filled in."""
    if name == "tiny":
        wl = Workload("tiny", 1, 1, 8, 2, 64, 512, 16, 512, [FULL, 128],
                      fixed_windows=[FULL, 128],
                      note="1 layer, batch 1, 8q/2kv, d64, 512-token prompt + 16 decode steps")
    elif name == "single32k":
        wl = Workload("single32k", 1, 1, 24, 4, 256, 32768, 256, 8192,
                      [FULL, 16384, 4096, 1024], fixed_windows=[FULL, 16384, 4096, 1024],
                      per_head_scale=True,
                      note="1 layer, batch 1, 24q/4kv, d256, 32K prompt + 256 decode, "
                           "K/V scaled per KV head by U[0.5,2)")
    elif name == "layers16_112k":
        wl = Workload("layers16_112k", 16, 16, 24, 4, 256, 114688 - 128, 128, 0,
                      [FULL, 32768, 8192, 2048, 512],
                      note="16 layers, batch 16, 24q/4kv, d256, 112K context, 128 decode "
                           "steps; windows drawn from {full, 32768, 8192, 2048, 512}")
    elif name == "prefill64k":
        wl = Workload("prefill64k", 1, 2, 32, 8, 128, 65536, 0, 8192, [FULL, 16384, 4096],
                      note="64K prompt in 8K chunks, batch 2, 32q/8kv, d128; windows drawn "
                           "from {full, 16384, 4096}")
    elif name == "budget161k":
        b = 1.0 if budget is None else budget
        wl = Workload("budget161k", 16, 4, 24, 4, 256, 164864 - 64, 64, 0, BUDGET_LEVELS,
                      budget=b,
                      note="161K context, batch 4, 16 layers, 24q/4kv, d256, 64 decode steps, "
                           "windows lowered to %.0f%% of all-full residency" % (100 * b))
        wl.name = "budget161k_r%02d" % int(round(100 * b))
    else:
        raise KeyError(name)
    if wl.fixed_windows is not None:
        wl.windows = list(wl.fixed_windows)
    elif wl.budget is not None:
        wl.windows = budget_windows(wl.n_units, wl.max_ctx, wl.budget, wl.seed)
    else:
        wl.windows = _drawn_windows(wl)
    return wl


NAMES = ["tiny", "single32k", "layers16_112k", "prefill64k", "budget161k"]
