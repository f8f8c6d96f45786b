"""Seeded synthetic inputs for the transfer: token segmentations, sender
K/V caches, folded maps and paged-cache block tables.

This module draws random numbers and lays them out; it holds none of the
method's arithmetic (no alignment, layer map, affine map or RoPE).  Both the
CUDA path and the CPU oracle are fed from it.

The shapes and value distributions stand in for the paper's QuALITY
contexts (4K-32K receiver tokens, Section 4.4 / Appendix G) and its model
pairs (Llama-3.1-8B, Qwen-family and Ministral-family KV widths), none of
which are available offline:

* segmentation: token lengths 1 + Binomial(12, (m - 1)/12) characters (mean
  m; 4.0 for the Llama-shaped side, 3.6 for the other), receiver lengths
  drawn first, sender lengths drawn over the same characters with the last
  one cut so both sides end at the same offset; the tiny case uses lengths
  uniform on 1..7 over a 1,024-character string;
* sender K/V: N(0, 1) times a per-(layer, role, channel) scale
  10 ** U(-1, 1) (outlier channels), stored in bf16; fp32 N(0, 1) for the
  tiny case;
* maps: W = A_final transposed, entries N(0, 1/K) with K the map input width,
  bias N(0, 0.1^2), and a positive per-(layer, role) normaliser r equal to
  the root-mean-square channel scale of that role times U(0.9, 1.1), so the
  mapped features have roughly unit variance;
* paged cache: 16-token blocks, a pool with 10% spare blocks and a seeded
  random permutation as the block table;
* KV Ridge apply: per receiver layer the 8 sender layers with the smallest
  |t - p| + U(0, 3) (p the proportional depth; a stand-in for the
  calibrated R^2 ranking), maps drawn as above and divided by the scale r
  would have had, with r = 1 (ridge maps have no normaliser).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field, replace
from typing import List, Optional, Tuple

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    L_s: int
    H_s: int
    D_s: int
    L_r: int
    H_r: int
    D_r: int
    theta_s: float
    theta_r: float
    r_tokens: Tuple[int, ...]          # receiver tokens per request (nominal when n_chars is set)
    mean_s: float = 4.0                # sender characters per token
    mean_r: float = 3.6                # receiver characters per token
    dtype: str = "bf16"                # "bf16" or "f32"
    align_mode: str = "ta"             # "ta", "overlap_mean", "same_index"
    layer_mode: str = "paper3"         # "paper3", "interp" or "explicit"
    paged: bool = False
    block_size: int = 16
    spare_frac: float = 0.10
    seed: int = 0
    uniform_lengths: Optional[Tuple[int, int]] = None  # tiny case: (lo, hi)
    n_chars: Optional[int] = None      # tiny case: fixed text length
    channel_scales: bool = True
    knorm: bool = False
    r_pos0: Optional[Tuple[int, ...]] = None
    # optional descriptor fields
    seg_layer: Optional[tuple] = None  # explicit layer table [L_r][n_seg][n_terms]
    seg_w: Optional[tuple] = None
    sender_k_rotated: bool = False     # sender keys stored with RoPE (base theta_s)
    s_pos0: Optional[Tuple[int, ...]] = None
    rope_table: bool = False           # receiver RoPE from a caller table (inv_freq_r_table)
    span_gap: int = 0                  # message spans: cache rows before each request's span
    kv_ridge: bool = False             # KV Ridge apply: explicit k-layer table, maps without r

    @property
    def d_s(self) -> int:
        return self.H_s * self.D_s

    @property
    def d_r(self) -> int:
        return self.H_r * self.D_r

    @property
    def n_seg(self) -> int:
        if self.layer_mode == "explicit":
            return len(self.seg_layer[0])
        return 3 if self.layer_mode == "paper3" else 1

    @property
    def K(self) -> int:
        return self.n_seg * self.d_s

    @property
    def n_req(self) -> int:
        return len(self.r_tokens)

    @property
    def torch_dtype(self):
        return torch.bfloat16 if self.dtype == "bf16" else torch.float32

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workload families (sizes of the paper's model pairs).
def tiny() -> Workload:
    """4 sender layers (2 x 64) -> 6 receiver layers (4 x 32), ~256 tokens a
    side over a 1,024-character string, overlap mean-pooling, two-layer
    interpolation, fp32 end to end."""
    return Workload("tiny_overlap_interp_f32", L_s=4, H_s=2, D_s=64, L_r=6, H_r=4, D_r=32,
                    theta_s=10000.0, theta_r=10000.0, r_tokens=(256,), dtype="f32",
                    align_mode="overlap_mean", layer_mode="interp", seed=0,
                    uniform_lengths=(1, 7), n_chars=1024, channel_scales=False)


def llama_to_qwen25(T_r: int = 4096) -> Workload:
    return Workload(f"llama8b_to_qwen25_7b_{T_r}", L_s=32, H_s=8, D_s=128, L_r=28, H_r=4,
                    D_r=128, theta_s=500000.0, theta_r=1e6, r_tokens=(T_r,),
                    mean_s=4.0, mean_r=3.6, seed=1)


def llama_to_ministral(T_r: int = 32768) -> Workload:
    return Workload(f"llama8b_to_ministral_{T_r}", L_s=32, H_s=8, D_s=128, L_r=40, H_r=8,
                    D_r=128, theta_s=500000.0, theta_r=1e8, r_tokens=(T_r,),
                    mean_s=4.0, mean_r=3.6, seed=2)


def qwen25_to_llama_batched(n_req: int = 8, lo: int = 2048, hi: int = 32768,
                            seed: int = 3) -> Workload:
    rng = np.random.default_rng(seed)
    lens = tuple(int(x) for x in rng.integers(lo, hi + 1, size=n_req))
    return Workload(f"qwen25_7b_to_llama8b_batch{n_req}_paged", L_s=28, H_s=4, D_s=128,
                    L_r=32, H_r=8, D_r=128, theta_s=1e6, theta_r=500000.0, r_tokens=lens,
                    mean_s=3.6, mean_r=4.0, paged=True, block_size=16, seed=seed)


def ministral_to_llama(T_r: int) -> Workload:
    return Workload(f"ministral_to_llama8b_{T_r}", L_s=40, H_s=8, D_s=128, L_r=32, H_r=8,
                    D_r=128, theta_s=1e8, theta_r=500000.0, r_tokens=(T_r,),
                    mean_s=3.6, mean_r=4.0, seed=4)


def kv_ridge_selection(L_s: int, L_r: int, k: int = 8, seed: int = 0):
    """A stand-in for KV Ridge's calibrated layer selection (k sender layers
    per receiver layer, ranked by calibration R^2, which favours layers near
    the proportional depth): the k sender layers with the smallest
    |t - p| + U(0, 3), p = l (L_s - 1)/(L_r - 1), in ascending order."""
    rng = np.random.default_rng([seed, 1010])
    out = []
    for l in range(L_r):
        p = l * (L_s - 1) / (L_r - 1) if L_r > 1 else 0.0
        score = np.abs(np.arange(L_s) - p) + rng.uniform(0.0, 3.0, size=L_s)
        out.append(tuple(sorted(int(t) for t in np.argsort(score, kind="stable")[:k])))
    return tuple(out)


def qwen25_to_llama_kv_ridge(T_r: int = 4096, k: int = 8, align_mode: str = "ta") -> Workload:
    """KV Ridge + TA apply on the Qwen2.5-7B-shaped -> Llama-3.1-8B-shaped
    direction: k = 8 selected sender layers per receiver layer, one dense
    [k d_S, d_R] map per layer and role (the per-head maps stacked), no
    Eq. 3 normaliser."""
    sel = kv_ridge_selection(28, 32, k, seed=13)
    layers = tuple(tuple((t,) for t in s) for s in sel)
    weights = tuple(tuple((1.0,) for _ in s) for s in sel)
    return Workload(f"qwen25_7b_to_llama8b_kv_ridge{k}_{T_r}", L_s=28, H_s=4, D_s=128, L_r=32,
                    H_r=8, D_r=128, theta_s=1e6, theta_r=500000.0, r_tokens=(T_r,),
                    mean_s=3.6, mean_r=4.0, seed=13, align_mode=align_mode,
                    layer_mode="explicit", seg_layer=layers, seg_w=weights, kv_ridge=True)


SWEEP_TOKENS = (256, 512, 1024, 4096, 16384, 32768, 65536, 131072)

# Model shapes (layers, KV heads, head width, RoPE base, characters per token).
MODEL_SHAPES = {
    "llama8b": (32, 8, 128, 500000.0, 4.0),
    "qwen25_7b": (28, 4, 128, 1e6, 3.6),
    "ministral": (40, 8, 128, 1e8, 3.6),
}


def direction(sender: str, receiver: str, T_r: int, seed: int, **kw) -> Workload:
    """A transfer between two of MODEL_SHAPES."""
    Ls, Hs, Ds, ths, ms = MODEL_SHAPES[sender]
    Lr, Hr, Dr, thr, mr = MODEL_SHAPES[receiver]
    return Workload(f"{sender}_to_{receiver}_{T_r}", L_s=Ls, H_s=Hs, D_s=Ds, L_r=Lr, H_r=Hr,
                    D_r=Dr, theta_s=ths, theta_r=thr, r_tokens=(T_r,), mean_s=ms, mean_r=mr,
                    seed=seed, **kw)


def message_round(msg_tokens: int = 160, ctx_tokens: int = 2048, seed: int = 20):
    """One communication round of three agents of different families (the
    multi-agent setting of the paper's HiddenBench evaluation): every agent's
    message goes to the two others, six directions.  Each message is a span
    of msg_tokens receiver tokens that follows ctx_tokens of context in the
    sender's cache; the receiver places it after its own context."""
    names = ("llama8b", "qwen25_7b", "ministral")
    out = []
    k = 0
    for a in names:
        for b in names:
            if a == b:
                continue
            out.append(direction(a, b, msg_tokens, seed + k, span_gap=ctx_tokens,
                                 r_pos0=(ctx_tokens,)))
            k += 1
    return out


# ---------------------------------------------------------------------------
# Segmentations
# ---------------------------------------------------------------------------

def _binomial_lengths(rng: np.random.Generator, n: int, mean: float) -> np.ndarray:
    return 1 + rng.binomial(12, (mean - 1.0) / 12.0, size=n)


def _cover(rng: np.random.Generator, n_chars: int, draw) -> List[int]:
    ends: List[int] = []
    e = 0
    while e < n_chars:
        chunk = draw(max(16, (n_chars - e) // 2))
        for ln in chunk:
            e = min(n_chars, e + int(ln))
            ends.append(e)
            if e >= n_chars:
                break
    return ends


@dataclass
class Tokens:
    """Character-end offsets of both tokenisations, concatenated over
    requests; request q owns [s_tok_ptr[q], s_tok_ptr[q+1]) and
    [r_tok_ptr[q], r_tok_ptr[q+1]); offsets restart at zero per request."""
    s_tok_ptr: np.ndarray
    r_tok_ptr: np.ndarray
    s_end: np.ndarray
    r_end: np.ndarray

    @property
    def T_s(self) -> int:
        return int(self.s_tok_ptr[-1])

    @property
    def T_r(self) -> int:
        return int(self.r_tok_ptr[-1])


def tokens(w: Workload) -> Tokens:
    rng = np.random.default_rng([w.seed, 101])
    s_all: List[np.ndarray] = []
    r_all: List[np.ndarray] = []
    for T_q in w.r_tokens:
        if w.uniform_lengths is not None:
            lo, hi = w.uniform_lengths
            n_chars = int(w.n_chars)
            r = _cover(rng, n_chars, lambda n: rng.integers(lo, hi + 1, size=n))
            s = _cover(rng, n_chars, lambda n: rng.integers(lo, hi + 1, size=n))
        else:
            if T_q == 0:
                r_all.append(np.zeros(0, np.int32))
                s_all.append(np.zeros(0, np.int32))
                continue
            r = list(np.cumsum(_binomial_lengths(rng, T_q, w.mean_r)))
            n_chars = int(r[-1])
            s = _cover(rng, n_chars, lambda n: _binomial_lengths(rng, n, w.mean_s))
        r_all.append(np.asarray(r, np.int32))
        s_all.append(np.asarray(s, np.int32))
    s_ptr = np.concatenate([[0], np.cumsum([len(x) for x in s_all])]).astype(np.int32)
    r_ptr = np.concatenate([[0], np.cumsum([len(x) for x in r_all])]).astype(np.int32)
    cat = lambda xs: np.concatenate(xs).astype(np.int32) if xs else np.zeros(0, np.int32)
    return Tokens(s_ptr, r_ptr, cat(s_all), cat(r_all))


# ---------------------------------------------------------------------------
# Values
# ---------------------------------------------------------------------------

def channel_scales(w: Workload) -> np.ndarray:
    """[L_s, 2, d_s] per-channel scales 10 ** U(-1, 1) (ones if disabled)."""
    rng = np.random.default_rng([w.seed, 202])
    if not w.channel_scales:
        return np.ones((w.L_s, 2, w.d_s), np.float32)
    return (10.0 ** rng.uniform(-1.0, 1.0, size=(w.L_s, 2, w.d_s))).astype(np.float32)


def sender_kv(w: Workload, T_s: int, device="cpu") -> torch.Tensor:
    """[L_s, 2, T_s, d_s] sender cache in the workload's dtype."""
    scales = torch.from_numpy(channel_scales(w)).to(device)
    g = torch.Generator(device=device)
    g.manual_seed(int(w.seed) * 1000 + 303)
    out = torch.empty((w.L_s, 2, T_s, w.d_s), dtype=w.torch_dtype, device=device)
    for t in range(w.L_s):
        for c in range(2):
            x = torch.randn((T_s, w.d_s), generator=g, device=device, dtype=torch.float32)
            out[t, c] = (x * scales[t, c][None, :]).to(w.torch_dtype)
    return out


def maps(w: Workload, device="cpu"):
    """Folded maps: W [L_r, 2, d_r, K] (= A_final transposed, workload
    dtype), bias [L_r, 2, d_r] fp32, r [L_r, 2] fp32 (host numpy).

    KV Ridge workloads have no normaliser: their maps come out of the same
    draw divided by the scale r would have had (so the outputs keep unit
    variance) and r is 1."""
    rng = np.random.default_rng([w.seed, 505])
    sc = channel_scales(w).astype(np.float64)
    rms_role = np.sqrt(np.mean(sc ** 2, axis=(0, 2)))  # per role
    r = (rms_role[None, :] * rng.uniform(0.9, 1.1, size=(w.L_r, 2))).astype(np.float32)
    g = torch.Generator(device=device)
    g.manual_seed(int(w.seed) * 1000 + 404)
    std = 1.0 / math.sqrt(w.K)
    W = torch.empty((w.L_r, 2, w.d_r, w.K), dtype=w.torch_dtype, device=device)
    for l in range(w.L_r):
        for c in range(2):
            scale = std / float(r[l, c]) if w.kv_ridge else std
            W[l, c] = (torch.randn((w.d_r, w.K), generator=g, device=device) * scale).to(w.torch_dtype)
    b = torch.randn((w.L_r, 2, w.d_r), generator=g, device=device, dtype=torch.float32) * 0.1
    if w.kv_ridge:
        r = np.ones((w.L_r, 2), np.float32)
    return W, b, r


def knorm_weight(w: Workload) -> Optional[np.ndarray]:
    if not w.knorm:
        return None
    rng = np.random.default_rng([w.seed, 606])
    return rng.uniform(0.5, 1.5, size=w.D_r).astype(np.float32)


def r_pos0(w: Workload) -> Optional[np.ndarray]:
    return None if w.r_pos0 is None else np.asarray(w.r_pos0, np.int32)


def s_pos0(w: Workload) -> Optional[np.ndarray]:
    return None if w.s_pos0 is None else np.asarray(w.s_pos0, np.int32)


def inv_freq_r_table(w: Workload) -> Optional[np.ndarray]:
    """A caller-supplied receiver RoPE frequency table (stand-in for a scaled
    RoPE variant): D_r/2 fp32 values log-uniform in [1e-6, 1], descending."""
    if not w.rope_table:
        return None
    rng = np.random.default_rng([w.seed, 808])
    return np.sort(10.0 ** rng.uniform(-6.0, 0.0, size=w.D_r // 2))[::-1].astype(np.float32)


def explicit_table(L_s: int, L_r: int, n_seg: int, n_terms: int, seed: int):
    """A seeded explicit layer table: random sender layers and weights in
    [-1, 1] (any structure the descriptor allows)."""
    rng = np.random.default_rng([seed, 909])
    layers = rng.integers(0, L_s, size=(L_r, n_seg, n_terms))
    weights = rng.uniform(-1.0, 1.0, size=(L_r, n_seg, n_terms)).astype(np.float32)
    return (tuple(tuple(tuple(int(x) for x in t) for t in s) for s in layers),
            tuple(tuple(tuple(float(x) for x in t) for t in s) for s in weights))


def span_layout(w: Workload, tok) -> Optional[Tuple[np.ndarray, int]]:
    """Message spans: each request's sender span sits after span_gap context
    rows of its own, so request q's span starts at cache row
    (q + 1) * span_gap + s_tok_ptr[q]; returns (s_row0, sender_rows)."""
    if w.span_gap <= 0:
        return None
    ptr = np.asarray(tok.s_tok_ptr, np.int64)
    s_row0 = (np.arange(1, len(ptr)) * w.span_gap + ptr[:-1]).astype(np.int32)
    return s_row0, int(ptr[-1] + (len(ptr) - 1) * w.span_gap)


def sender_cache_rows(w: Workload, tok) -> int:
    sp = span_layout(w, tok)
    return tok.T_s if sp is None else sp[1]


def desc_options(w: Workload, tok=None) -> dict:
    """The optional descriptor fields a workload asks for."""
    opts = {}
    if w.span_gap > 0:
        s_row0, rows = span_layout(w, tok)
        opts.update(s_row0=s_row0, sender_rows=rows)
    if w.layer_mode == "explicit":
        opts.update(seg_layer=np.asarray(w.seg_layer, np.int32),
                    seg_w=np.asarray(w.seg_w, np.float32))
    if w.sender_k_rotated:
        opts.update(sender_k_rotated=True, theta_s=w.theta_s, s_pos0=s_pos0(w))
    if w.rope_table:
        opts.update(inv_freq_r=inv_freq_r_table(w))
    return opts


@dataclass
class Paged:
    block_table: np.ndarray   # [n_req, max_blocks] int32, -1 = unused
    n_blocks: int             # blocks in the pool
    max_blocks: int


def paged_layout(w: Workload, tok: Tokens) -> Paged:
    rng = np.random.default_rng([w.seed, 707])
    bs = w.block_size
    per_req = [(int(tok.r_tok_ptr[q + 1] - tok.r_tok_ptr[q]) + bs - 1) // bs for q in range(w.n_req)]
    used = sum(per_req)
    pool = max(1, int(math.ceil(used * (1.0 + w.spare_frac))))
    perm = rng.permutation(pool).astype(np.int32)
    mb = max(1, max(per_req) if per_req else 1)
    table = np.full((w.n_req, mb), -1, np.int32)
    k = 0
    for q, n in enumerate(per_req):
        table[q, :n] = perm[k:k + n]
        k += n
    return Paged(table, pool, mb)
