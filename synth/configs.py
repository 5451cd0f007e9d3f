"""Workload shapes and recipes.

Shapes follow the models the paper evaluates (Table 7, model architectures) plus a
GPT-2-small shape; the value recipes are synthetic stand-ins for pretrained weights,
which are not available here.  Every recipe draws bf16 weights in the nn.Linear
layout ``Wq[l]: [n_q*d_h, d]``, ``Wk[l]: [n_kv*d_h, d]`` (row-major).
"""

from dataclasses import dataclass, field


@dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    d: int
    n_q: int
    n_kv: int
    d_h: int
    iters: int
    recipe: str  # "spike1", "lognormal", "planted", "spike4"
    seed: int
    steps: int = 0  # >0: transient refresh workload (warm-started, iters per step)
    cold_iters: int = 0  # iterations of the cold start that precedes step 0
    notes: str = field(default="", compare=False)

    @property
    def group(self) -> int:
        return self.n_q // self.n_kv

    @property
    def heads(self) -> int:
        return self.layers * self.n_q

    def weight_bytes(self) -> int:
        return 2 * self.layers * (self.n_q + self.n_kv) * self.d_h * self.d

    def vector_bytes(self) -> int:
        """fp32 start vectors read plus fp32 written-back vectors."""
        return 2 * 4 * self.layers * self.n_q * self.d

    def algorithmic_bytes(self) -> int:
        """Least any exact k-step implementation must move: every W^Q_h and every
        (unexpanded) W^K_g once, v_in read, v_out written."""
        return self.weight_bytes() + self.vector_bytes()

    def scaled(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


_BASE_SEED = 1885100

WORKLOADS = {
    # GPT-2-small shape, MHA, d_h=64, rank-1 planted spike per head.
    "gpt2-small": Workload("gpt2-small", 12, 768, 12, 12, 64, 20, "spike1", _BASE_SEED + 1),
    # GPT-2-XL shape (Table 7), MHA 25/25, per-head log-normal norm multiplier.
    "gpt2-xl": Workload("gpt2-xl", 48, 1600, 25, 25, 64, 20, "lognormal", _BASE_SEED + 2),
    # Llama-2-7B shape, MHA 32/32, planted singular spectra (closed-form sigma).
    "llama2-7b-planted": Workload("llama2-7b-planted", 32, 4096, 32, 32, 128, 30, "planted",
                                  _BASE_SEED + 3),
    # Llama-2-70B shape (Table 7), GQA 64/8, rank-4 spikes.
    "llama2-70b-gqa": Workload("llama2-70b-gqa", 80, 8192, 64, 8, 128, 30, "spike4", _BASE_SEED + 4),
    # Llama-2-70B transient refresh: cold start (30 iterations) then 100 warm steps of 2.
    "llama2-70b-transient": Workload("llama2-70b-transient", 80, 8192, 64, 8, 128, 2, "spike4",
                                     _BASE_SEED + 4, steps=100, cold_iters=30),
    # Small cases for the CPU suite and quick parity tests (several tiles, ragged tails).
    "tiny-mha": Workload("tiny-mha", 2, 256, 4, 4, 64, 12, "spike1", _BASE_SEED + 11),
    "tiny-gqa": Workload("tiny-gqa", 2, 256, 8, 2, 64, 12, "spike4", _BASE_SEED + 12),
    "tiny-gqa128": Workload("tiny-gqa128", 3, 512, 8, 2, 128, 15, "spike4", _BASE_SEED + 13),
    "ragged": Workload("ragged", 3, 200, 6, 3, 64, 10, "lognormal", _BASE_SEED + 14),
    "ragged128": Workload("ragged128", 2, 1000, 5, 5, 128, 9, "spike1", _BASE_SEED + 15),
    # Group-size edge cases: 16 and 32 query heads per KV head (the latter gives the
    # widest z0 / write-back operand, 128 rows).
    "tiny-g16": Workload("tiny-g16", 2, 384, 16, 1, 128, 8, "spike4", _BASE_SEED + 16),
    "tiny-g32": Workload("tiny-g32", 2, 320, 32, 1, 64, 8, "spike4", _BASE_SEED + 17),
    # The largest group at d_h 128: 64 query heads per KV head (a 128-row v operand and
    # 64 heads' start vectors per key tile).
    "tiny-g64": Workload("tiny-g64", 2, 256, 64, 1, 128, 6, "spike4", _BASE_SEED + 21),
    # Head widths outside {64, 128} (streaming back end): 80 and 96 as in several
    # published models, 256 as in wide-head ones.
    "tiny-dh80": Workload("tiny-dh80", 2, 320, 4, 2, 80, 10, "spike4", _BASE_SEED + 18),
    "tiny-dh96": Workload("tiny-dh96", 2, 384, 6, 3, 96, 10, "lognormal", _BASE_SEED + 19),
    "tiny-dh256": Workload("tiny-dh256", 2, 512, 4, 2, 256, 10, "spike1", _BASE_SEED + 20),
    # A full-size model with d_h 80 (Phi-2-like: 32 layers, d 2560, 32/32 heads), for
    # timing the tensor-core back ends on a head width that does not fill 128-row tiles.
    "dh80-mha": Workload("dh80-mha", 32, 2560, 32, 32, 80, 30, "spike4", _BASE_SEED + 22),
    # A full-size model with d_h 256 (Gemma-7B-like: 28 layers, d 3072, 16/16 heads), for
    # timing the streaming back end that such head widths run on.
    "dh256-mha": Workload("dh256-mha", 28, 3072, 16, 16, 256, 30, "spike4", _BASE_SEED + 23),
}

# Transient recipe (per step, per weight matrix W of one head or KV group):
#   W_master += eps * ||W_master||_F * P Q^T / ||P Q^T||_F,  P: d_h x 8, Q: d x 8 Gaussian,
#   eps = 1e-3, except 5e-2 for steps 40..45 inclusive; the bf16 weights are the
#   round-to-nearest-even of the fp32 master copy.
TRANSIENT_RANK = 8
TRANSIENT_EPS = 1e-3
TRANSIENT_SPIKE_EPS = 5e-2
TRANSIENT_SPIKE_STEPS = range(40, 46)


def get_workload(name: str) -> Workload:
    try:
        return WORKLOADS[name]
    except KeyError as e:
        raise KeyError(f"unknown workload {name!r}; known: {sorted(WORKLOADS)}") from e
