"""Workload table and seeded generators.

Every tensor here is a function of (workload, seed, tags) only.  Random draws use
``torch.Generator`` objects whose seeds are derived with BLAKE2b from the
workload seed and a tag naming the draw, so that one draw never depends on
another draw's length or order.  Per-sequence quantities use per-sequence seeds,
so a sequence's data is the same whatever the batch size.

Value distributions (shapes follow the paper's Qwen3-8B-class workloads, §5.1):

* ``planted``      fp32 logits ~ N(0, 1) plus +4 at one seeded token per row.
* ``zipf_gumbel``  bf16(z + g + beta_v): z ~ N(0, sigma_z), g ~ Gumbel(0, 1),
                   beta_v = -1.1 * ln(1 + pi(v)) with pi a seeded permutation of
                   the vocabulary (a Zipf(1.1) token-frequency prior).
* ``zipf_temp``    bf16((z + beta_v) / tau_d), tau_d ~ U[0.5, 2] per row.

The trigram prefix signal (the paper instantiates rho_d with an n-gram model,
n = 3, §5.1) is a synthetic table: each triple over the ``n_frequent`` most
frequent tokens is present with probability ``table_density``, plus
``n_background`` uniform random triples; its log-probabilities are exact binary
fractions -(h & 63) / 8 in [-7.875, 0], h a SplitMix64 hash of the triple.
"""

from __future__ import annotations

import hashlib
from dataclasses import dataclass, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int                 # sequences in the batch
    L: int                 # drafter block length (tree depth limit)
    V: int                 # vocabulary size
    k: int                 # candidates kept per position
    N: int                 # node budget, root included
    lam: float             # prefix-correction strength lambda_d
    use_table: bool        # False: marginal-only scoring (no prefix signal)
    logits: str            # "planted" | "zipf_gumbel" | "zipf_temp"
    logits_dtype: str      # "f32" | "bf16"
    Hq: int                # query heads
    Hkv: int               # key/value heads
    D: int                 # head dim
    T: int                 # KV-cache length (maximum when ragged)
    T_min: int             # minimum KV length (== T unless ragged)
    layers: int = 1        # independent attention layers per round
    seed: int = 0
    b: int = 0             # branching factor; 0 means b = k
    table_log2_cap: int = 22
    n_background: int = 1_000_000
    n_frequent: int = 64
    table_density: float = 0.3
    sigma_z: float = 2.0
    target_noise: float = 1.5
    p_target_argmax: float = 0.7
    miss_logrho: float = -12.0

    @property
    def branching(self) -> int:
        return self.b or self.k

    @property
    def rows(self) -> int:
        return self.B * self.L

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    # 1 x 8 x 4096 fp32 logits, k=4, N=16; 4 q-heads / 1 kv-head, D=64, T=256.
    "tiny": Workload("tiny", B=1, L=8, V=4096, k=4, N=16, lam=0.2, use_table=True,
                     logits="planted", logits_dtype="f32", Hq=4, Hkv=1, D=64,
                     T=256, T_min=256, seed=0, table_log2_cap=19,
                     n_background=20_000, sigma_z=1.0),
    # Qwen3-8B-shaped dedicated-drafter round: B=1, L=16, k=8, N=64, GQA 32/8,
    # D=128, T=4096.
    "qwen3_8b": Workload("qwen3_8b", B=1, L=16, V=151936, k=8, N=64, lam=0.2,
                         use_table=True, logits="zipf_gumbel", logits_dtype="bf16",
                         Hq=32, Hkv=8, D=128, T=4096, T_min=4096, seed=1),
    # Batched serving: B=16, N=128, ragged T ~ U{1024..16384}.
    "batched_ragged": Workload("batched_ragged", B=16, L=16, V=151936, k=8, N=128,
                               lam=0.2, use_table=True, logits="zipf_gumbel",
                               logits_dtype="bf16", Hq=32, Hkv=8, D=128,
                               T=16384, T_min=1024, seed=2),
    # Self-speculative dLLM round, marginal-only scoring: B=4, L=32, k=6, N=256.
    "self_spec": Workload("self_spec", B=4, L=32, V=151936, k=6, N=256, lam=0.0,
                          use_table=False, logits="zipf_temp", logits_dtype="bf16",
                          Hq=32, Hkv=8, D=128, T=8192, T_min=8192, seed=3),
    # Long-context stress: B=8, k=10, N=256, T=32768, 36 layers of attention.
    "long_ctx": Workload("long_ctx", B=8, L=16, V=151936, k=10, N=256, lam=0.2,
                         use_table=True, logits="zipf_gumbel", logits_dtype="bf16",
                         Hq=32, Hkv=8, D=128, T=32768, T_min=32768, layers=36,
                         seed=4),
}


# --------------------------------------------------------------------------- seeds

def _seed(*parts) -> int:
    h = hashlib.blake2b(repr(parts).encode(), digest_size=8).digest()
    return int.from_bytes(h, "little") & ((1 << 63) - 1)


def _gen(device, *parts) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(_seed(*parts))
    return g


def _splitmix64(x: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser (Steele, Lea, Flood 2014), vectorised over uint64."""
    z = (x.astype(np.uint64) + np.uint64(0x9E3779B97F4A7C15))
    z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
    z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
    return z ^ (z >> np.uint64(31))


# --------------------------------------------------------------------------- logits

def zipf_rank(w: Workload) -> torch.Tensor:
    """pi(v): a seeded permutation of the vocabulary; rank 0 is the most frequent."""
    return torch.randperm(w.V, generator=_gen("cpu", w.seed, "zipf"))


def planted_peaks(w: Workload, b: int) -> torch.Tensor:
    return torch.randint(0, w.V, (w.L,), generator=_gen("cpu", w.seed, "peak", b))


def drafter_logits(w: Workload, seqs=None) -> torch.Tensor:
    """Drafter per-position logits [len(seqs), L, V] on the CPU (fp32 or bf16)."""
    seqs = range(w.B) if seqs is None else seqs
    out = []
    beta = None
    if w.logits != "planted":
        beta = -1.1 * torch.log1p(zipf_rank(w).to(torch.float32))
    for b in seqs:
        g = _gen("cpu", w.seed, "logits", b)
        if w.logits == "planted":
            x = torch.randn(w.L, w.V, generator=g, dtype=torch.float32) * w.sigma_z
            x[torch.arange(w.L), planted_peaks(w, b)] += 4.0
        elif w.logits == "zipf_gumbel":
            z = torch.randn(w.L, w.V, generator=g, dtype=torch.float32) * w.sigma_z
            u = torch.rand(w.L, w.V, generator=g, dtype=torch.float32).clamp_min(1e-20)
            x = z - torch.log(-torch.log(u)) + beta
        elif w.logits == "zipf_temp":
            z = torch.randn(w.L, w.V, generator=g, dtype=torch.float32) * w.sigma_z
            tau = 0.5 + 1.5 * torch.rand(w.L, 1, generator=g, dtype=torch.float32)
            x = (z + beta) / tau
        else:
            raise ValueError(w.logits)
        out.append(x)
    x = torch.stack(out)
    return x.to(torch.bfloat16) if w.logits_dtype == "bf16" else x.contiguous()


# --------------------------------------------------------------------------- context / table

def frequent_tokens(w: Workload) -> np.ndarray:
    """The token set the synthetic trigram table concentrates on (sorted)."""
    if w.logits == "planted":
        peaks = torch.cat([planted_peaks(w, b) for b in range(w.B)]).numpy()
        extra = torch.randint(0, w.V, (w.n_frequent,),
                              generator=_gen("cpu", w.seed, "freq")).numpy()
        return np.unique(np.concatenate([peaks, extra]))
    rank = zipf_rank(w).numpy()
    return np.sort(np.nonzero(rank < w.n_frequent)[0])


def ctx_tokens(w: Workload) -> torch.Tensor:
    """Last two committed tokens per sequence, int32 [B, 2]; column 1 is the root."""
    freq = torch.from_numpy(frequent_tokens(w))
    idx = torch.randint(0, len(freq), (w.B, 2), generator=_gen("cpu", w.seed, "ctx"))
    return freq[idx].to(torch.int32)


def trigram_entries(w: Workload):
    """Synthetic trigram table as parallel arrays (a, b, t, logrho).

    Keys are unique.  Returns int64 token arrays and float32 log-probabilities
    (exact binary fractions <= 0).  Empty arrays when the workload has no table.
    """
    if not w.use_table:
        e = np.zeros(0, np.int64)
        return e, e.copy(), e.copy(), np.zeros(0, np.float32)
    freq = frequent_tokens(w).astype(np.int64)
    nf = len(freq)
    g = _gen("cpu", w.seed, "table")
    keep = (torch.rand(nf ** 3, generator=g) < w.table_density).numpy()
    ia, ib, it = np.unravel_index(np.nonzero(keep)[0], (nf, nf, nf))
    a, b, t = freq[ia], freq[ib], freq[it]
    bg = torch.randint(0, w.V, (3, w.n_background), generator=g).numpy().astype(np.int64)
    a = np.concatenate([a, bg[0]])
    b = np.concatenate([b, bg[1]])
    t = np.concatenate([t, bg[2]])
    code = (a * w.V + b) * w.V + t
    code, first = np.unique(code, return_index=True)
    a, b, t = a[first], b[first], t[first]
    h = _splitmix64(code.astype(np.uint64))
    logrho = -((h & np.uint64(63)).astype(np.float32)) / np.float32(8.0)
    return a, b, t, logrho.astype(np.float32)


# --------------------------------------------------------------------------- attention

def kv_lengths(w: Workload) -> torch.Tensor:
    if w.T_min == w.T:
        return torch.full((w.B,), w.T, dtype=torch.int32)
    g = _gen("cpu", w.seed, "kvlen")
    return torch.randint(w.T_min, w.T + 1, (w.B,), generator=g).to(torch.int32)


def attention_inputs(w: Workload, layer: int = 0, device="cpu") -> dict:
    """One layer's tree-attention inputs, bf16 ~ N(0, 1), generated on `device`.

    q       [B, N, Hq, D]      query rows of the N tree tokens (RoPE already applied)
    k_cache [B, Hkv, T, D]     committed-prefix keys; rows >= kv_len[b] are padding
    v_cache [B, Hkv, T, D]
    k_tree  [B, N, Hkv, D]     keys / values of the tree tokens themselves
    v_tree  [B, N, Hkv, D]
    kv_len  [B] int32
    """
    g = _gen(device, w.seed, "attn", layer)
    bf = torch.bfloat16

    def rn(*shape):
        return torch.randn(*shape, generator=g, device=device, dtype=torch.float32).to(bf)

    return {
        "q": rn(w.B, w.N, w.Hq, w.D),
        "k_cache": rn(w.B, w.Hkv, w.T, w.D),
        "v_cache": rn(w.B, w.Hkv, w.T, w.D),
        "k_tree": rn(w.B, w.N, w.Hkv, w.D),
        "v_tree": rn(w.B, w.N, w.Hkv, w.D),
        "kv_len": kv_lengths(w).to(device),
    }


# --------------------------------------------------------------------------- target model

def node_paths(node_token, node_parent, n_nodes):
    """Token path (root excluded) of every used node, per sequence: list of lists of tuples."""
    node_token = np.asarray(node_token)
    node_parent = np.asarray(node_parent)
    out = []
    for b in range(node_token.shape[0]):
        paths = []
        for i in range(int(n_nodes[b])):
            toks = []
            j = i
            while j > 0:
                toks.append(int(node_token[b, j]))
                j = int(node_parent[b, j])
            paths.append(tuple(reversed(toks)))
        out.append(paths)
    return out


def target_token_for_path(w: Workload, logits_row_fn, b: int, path: tuple, device="cpu") -> int:
    """The synthetic target model's greedy next token after root + `path`.

    planted workloads: the drafter argmax of the next position with probability
    p_target_argmax, else a uniform token.  Other workloads: argmax over the
    vocabulary of (drafter logit of the next position + N(0, target_noise)).
    Past the block (len(path) == L) the token is uniform.  The draw is seeded by
    (seed, b, path), so it does not depend on node order or tree size.
    """
    g = _gen(device, w.seed, "target", b, path)
    d = len(path)
    if d >= w.L:
        return int(torch.randint(0, w.V, (1,), generator=g, device=device).item())
    row = logits_row_fn(d).to(device=device, dtype=torch.float32)
    if w.logits == "planted":
        u = torch.rand(1, generator=g, device=device).item()
        if u < w.p_target_argmax:
            return int(torch.argmax(row).item())
        return int(torch.randint(0, w.V, (1,), generator=g, device=device).item())
    eps = torch.randn(w.V, generator=g, device=device, dtype=torch.float32) * w.target_noise
    return int(torch.argmax(row + eps).item())


def target_tokens(w: Workload, logits, node_token, node_parent, n_nodes, device="cpu") -> torch.Tensor:
    """target_token[b, i]: the target's greedy token after node i (int32 [B, N], -1 unused)."""
    logits = logits.to(device)
    out = torch.full((w.B, w.N), -1, dtype=torch.int32)
    for b, paths in enumerate(node_paths(node_token, node_parent, n_nodes)):
        for i, p in enumerate(paths):
            out[b, i] = target_token_for_path(w, lambda d: logits[b, d], b, p, device)
    return out
