"""Seeded synthetic inputs shaped like the fuzzy token-matching workloads.

Both the CUDA path (tests, bench) and the CPU oracle (tests, the bench's CPU baseline)
draw their inputs from here, so the two sides see identical bytes.  This module only
draws random numbers and arranges them into prompt-shaped arrays: it contains none of
the method's arithmetic (no rotary encoding, no projection, no hashing, no Hamming
distance, no gather).

The paper evaluates on summarization prompts of up to 5k tokens (Sec. 4.1, Sec. 4.3)
with reference/target pairs that share most of their content.  Those datasets are not
available, so each workload below builds a reference prompt of i.i.d. N(0,1) embedding
rows and target prompts whose rows are either noisy copies of reference rows (moved to
other positions) or fresh N(0,1) rows.  The generator records the reference row each
target row was copied from (-1 for fresh rows) as a recall diagnostic.

bf16 arrays are carried as uint16 bit patterns (numpy has no bfloat16).
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

# Independent random substreams of one workload seed.
_S_REF, _S_SRC, _S_NOISE, _S_FRESH_MASK, _S_FRESH, _S_HYPER, _S_KV, _S_POOL = range(1, 9)


def rng(seed: int, *stream: int) -> np.random.Generator:
    """A PCG64 generator for substream `stream` of `seed` (platform independent)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(entropy=seed, spawn_key=tuple(stream))))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even) and return the bit patterns.

    Only used to produce bf16 *inputs*; finite values only (the generator draws no NaN)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    u = u + (np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1)))
    return (u >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (exact)."""
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass(frozen=True)
class Workload:
    """Shape and synthetic recipe of one matching workload.

    n_ref     reference tokens in total (for a pool: the sum over its n_seg members)
    n_tgt     tokens per target prompt
    n_batch   number of target prompts matched against the same reference
    d         embedding dimension; emb_dtype 'f32' or 'bf16'
    nbits     LSH code length in bits (multiple of 32)
    kv        (layers, kv heads, head_dim) of the bf16 K/V caches
    reuse     fraction of target rows copied from the reference
    noise     standard deviation of the Gaussian noise added to copied rows
    recipe    how copied rows are placed: 'perm' (global random permutation),
              'window' (local shuffle of +-window positions), 'subset' (sorted random
              subset, order kept), 'pool' (uniform pool member and row),
              'retrieve' (the rows of one pool member in order: the target is a rewrite of
              one stored prompt, the reference retrieval case of Sec. 3.2 and Sec. 4.4)
    """
    name: str
    n_ref: int
    n_tgt: int
    d: int
    emb_dtype: str
    nbits: int
    kv: tuple
    reuse: float
    noise: float
    recipe: str
    n_batch: int = 1
    n_seg: int = 1
    window: int = 64
    base_seed: int = 0x5E4D5AE0

    @property
    def n_layers(self):
        return self.kv[0]

    @property
    def n_heads(self):
        return self.kv[1]

    @property
    def head_dim(self):
        return self.kv[2]

    @property
    def seg_len(self):
        return self.n_ref // self.n_seg

    def scaled(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads (sizes of the paper's prompts: up to 5k tokens; Llama-3-8B-like
# embedding width 4096 and KV cache 32 layers x 8 KV heads x 128).
WORKLOADS = {
    "tiny": Workload("tiny", n_ref=256, n_tgt=256, d=512, emb_dtype="f32", nbits=64,
                     kv=(2, 4, 64), reuse=0.75, noise=0.1, recipe="perm", base_seed=0x5E4D5AE0 + 0),
    "llama8b-1k": Workload("llama8b-1k", n_ref=1024, n_tgt=1024, d=4096, emb_dtype="bf16", nbits=128,
                           kv=(32, 8, 128), reuse=0.70, noise=0.1, recipe="perm", base_seed=0x5E4D5AE0 + 1),
    "llama8b-5k": Workload("llama8b-5k", n_ref=5120, n_tgt=5120, d=4096, emb_dtype="bf16", nbits=256,
                           kv=(32, 8, 128), reuse=0.50, noise=0.2, recipe="window", window=64,
                           base_seed=0x5E4D5AE0 + 2),
    "batched-64x2048": Workload("batched-64x2048", n_ref=4096, n_tgt=2048, n_batch=64, d=4096, emb_dtype="bf16",
                                nbits=256, kv=(32, 8, 128), reuse=0.60, noise=0.2, recipe="subset",
                                base_seed=0x5E4D5AE0 + 3),
    "pool-16x4096": Workload("pool-16x4096", n_ref=65536, n_seg=16, n_tgt=4096, d=4096, emb_dtype="bf16",
                             nbits=256, kv=(32, 8, 128), reuse=0.60, noise=0.2, recipe="pool",
                             base_seed=0x5E4D5AE0 + 4),
}

# Reference retrieval (Sec. 3.2): 16 stored prompts of 4096 tokens, and a target that is one of
# them with 3% of its rows replaced and light noise on the rest (the replace study of Sec. 4.4);
# its retrieval codes are taken without rotary encoding (retrieval precedes it in Sec. 3.2).
RETRIEVAL_WORKLOADS = {
    "retrieve-16x4096": Workload("retrieve-16x4096", n_ref=65536, n_seg=16, n_tgt=4096, d=4096, emb_dtype="bf16",
                                 nbits=256, kv=(32, 8, 128), reuse=0.97, noise=0.02, recipe="retrieve",
                                 base_seed=0x5E4D5AE0 + 5),
}


def retrieval_member(wl: Workload, seed: int | None = None, b: int = 0) -> int:
    """The pool member target prompt `b` of a 'retrieve' workload was rewritten from."""
    seed = wl.base_seed if seed is None else seed
    return int(rng(seed, _S_POOL, b).integers(0, wl.n_seg))


def _emb_out(x: np.ndarray, emb_dtype: str) -> np.ndarray:
    return x.astype(np.float32) if emb_dtype == "f32" else f32_to_bf16_bits(x)


def reference_embeddings(wl: Workload, seed: int | None = None) -> np.ndarray:
    """Reference (or pool) embedding rows [n_ref][d]: i.i.d. N(0,1)."""
    seed = wl.base_seed if seed is None else seed
    out = np.empty((wl.n_ref, wl.d), dtype=np.float32 if wl.emb_dtype == "f32" else np.uint16)
    g = rng(seed, _S_REF)
    step = max(1, (1 << 24) // wl.d)
    for r0 in range(0, wl.n_ref, step):
        r1 = min(wl.n_ref, r0 + step)
        out[r0:r1] = _emb_out(g.standard_normal((r1 - r0, wl.d), dtype=np.float32), wl.emb_dtype)
    return out


def reference_positions(wl: Workload) -> np.ndarray:
    """Each reference prompt's own 0-based token positions (a pool restarts per member)."""
    return np.tile(np.arange(wl.seg_len, dtype=np.int32), wl.n_seg)


def _source_rows(wl: Workload, seed: int, b: int) -> np.ndarray:
    """Reference row each target row is copied from, -1 where the row is fresh."""
    n = wl.n_tgt
    g = rng(seed, _S_SRC, b)
    if wl.recipe == "perm":
        src = g.permutation(wl.n_ref)[:n].astype(np.int64)
    elif wl.recipe == "window":
        key = np.arange(n, dtype=np.float64) + g.uniform(-wl.window, wl.window, size=n)
        src = np.argsort(key, kind="stable").astype(np.int64) % wl.n_ref
    elif wl.recipe == "subset":
        src = np.sort(g.choice(wl.n_ref, size=n, replace=False)).astype(np.int64)
    elif wl.recipe == "retrieve":
        if n > wl.seg_len:
            raise ValueError("a rewritten prompt is at most one member long")
        src = (retrieval_member(wl, seed, b) * wl.seg_len + np.arange(n)).astype(np.int64)
    elif wl.recipe == "pool":
        member = g.integers(0, wl.n_seg, size=n)
        row = g.integers(0, wl.seg_len, size=n)
        src = (member * wl.seg_len + row).astype(np.int64)
    else:
        raise ValueError(wl.recipe)
    n_fresh = int(round((1.0 - wl.reuse) * n))
    fresh = rng(seed, _S_FRESH_MASK, b).permutation(n)[:n_fresh]
    src[fresh] = -1
    return src


def target_prompt(wl: Workload, b: int = 0, ref: np.ndarray | None = None, seed: int | None = None):
    """Target prompt `b`: (embeddings [n_tgt][d], positions [n_tgt], source rows [n_tgt]).

    Copied rows are reference rows plus N(0, noise^2); fresh rows are N(0,1).  Each target
    prompt of a batch has its own substreams, so any one can be drawn alone."""
    seed = wl.base_seed if seed is None else seed
    if ref is None:
        ref = reference_embeddings(wl, seed)
    src = _source_rows(wl, seed, b)
    ref_f = ref if wl.emb_dtype == "f32" else None
    x = np.empty((wl.n_tgt, wl.d), dtype=np.float32)
    copied = src >= 0
    rows = src[copied]
    x[copied] = ref_f[rows] if ref_f is not None else bf16_bits_to_f32(ref[rows])
    x[copied] += np.float32(wl.noise) * rng(seed, _S_NOISE, b).standard_normal((int(copied.sum()), wl.d),
                                                                                 dtype=np.float32)
    x[~copied] = rng(seed, _S_FRESH, b).standard_normal((int((~copied).sum()), wl.d), dtype=np.float32)
    pos = np.arange(wl.n_tgt, dtype=np.int32)
    return _emb_out(x, wl.emb_dtype), pos, src.astype(np.int32)


def hyperplanes(wl: Workload, seed: int | None = None) -> np.ndarray:
    """LSH hyperplanes [nbits][d]: N(0,1) draws stored as bf16 bit patterns."""
    seed = wl.base_seed if seed is None else seed
    return f32_to_bf16_bits(rng(seed, _S_HYPER).standard_normal((wl.nbits, wl.d), dtype=np.float32))


def kv_cache(wl: Workload, seed: int | None = None, segment: int | None = None):
    """Reference K and V caches as bf16 bit patterns, each [n_seg][L][H][seg_len][hd].

    With `segment` given, only that pool member's [L][H][seg_len][hd] pair is drawn."""
    seed = wl.base_seed if seed is None else seed
    L, H, hd = wl.kv
    segs = range(wl.n_seg) if segment is None else [segment]
    ks, vs = [], []
    for s in segs:
        g = rng(seed, _S_KV, s)
        shape = (L, H, wl.seg_len, hd)
        ks.append(f32_to_bf16_bits(g.standard_normal(shape, dtype=np.float32)))
        vs.append(f32_to_bf16_bits(g.standard_normal(shape, dtype=np.float32)))
    if segment is not None:
        return ks[0], vs[0]
    return np.stack(ks), np.stack(vs)


def random_codes(n: int, nbits: int, seed: int, stream: int = 0) -> np.ndarray:
    """Uniform random packed codes [n][nbits/32] (uint32) for search-only tests."""
    return rng(seed, 100 + stream).integers(0, 1 << 32, size=(n, nbits // 32), dtype=np.uint64).astype(np.uint32)


def kv_cache_device(wl: Workload, device, seed: int | None = None, segment: int = 0):
    """One reference prompt's K and V caches drawn on the device: bf16 N(0,1), each
    [L][H][seg_len][hd].  For the multi-GB caches of the batched and pool workloads, where
    drawing on the host would dominate; seeded through a device generator."""
    import torch

    seed = wl.base_seed if seed is None else seed
    L, H, hd = wl.kv
    g = torch.Generator(device=device).manual_seed((seed * 1000003 + 7919 * (segment + 1)) & 0x7FFFFFFFFFFFFFFF)
    k = torch.randn((L, H, wl.seg_len, hd), generator=g, device=device).to(torch.bfloat16)
    v = torch.randn((L, H, wl.seg_len, hd), generator=g, device=device).to(torch.bfloat16)
    return k, v


def prompt_rows(wl: Workload, seed: int | None = None, batches=None):
    """Host rows of one matching problem, reference rows first:
    (emb [n_ref + B*n_tgt][d], positions, source rows [B][n_tgt]) for target prompts `batches`
    (default: all n_batch of them)."""
    seed = wl.base_seed if seed is None else seed
    batches = range(wl.n_batch) if batches is None else list(batches)
    ref = reference_embeddings(wl, seed)
    rows, pos, src = [ref], [reference_positions(wl)], []
    for b in batches:
        x, p, s = target_prompt(wl, b=b, ref=ref, seed=seed)
        rows.append(x)
        pos.append(p)
        src.append(s)
    return np.concatenate(rows), np.concatenate(pos).astype(np.int32), np.stack(src)


def recomputed_kv_device(wl: Workload, device, k_ref, v_ref, src, seed: int | None = None, noise: float = 0.05):
    """A synthetic recomputed cache for the target prompt, [L][H][n_tgt][hd] bf16 each: a target
    token copied from reference row src[t] gets that row's K/V plus N(0, noise^2); a fresh token
    (src[t] = -1) gets fresh N(0,1) values.  k_ref/v_ref: the reference cache's layers to
    recompute ([L][H][N][hd]); seeded through a device generator."""
    import torch

    seed = wl.base_seed if seed is None else seed
    g = torch.Generator(device=device).manual_seed((seed * 7919 + 104729) & 0x7FFFFFFFFFFFFFFF)
    s = torch.as_tensor(np.asarray(src), device=device).long()
    copied = s >= 0
    out = []
    for ref in (k_ref, v_ref):
        L, H, _, hd = ref.shape
        x = torch.randn((L, H, len(s), hd), generator=g, device=device)
        base = ref.float()[:, :, s.clamp(min=0)]
        x = torch.where(copied.view(1, 1, -1, 1), base + noise * x, x)
        out.append(x.to(torch.bfloat16).contiguous())
    return out[0], out[1]


# Retention schedule for the synthetic workloads (Sec. 3.3.4, App. A: alpha_retain larger in
# shallow layers, smaller in deep ones; the first layer keeps max(0.8, r_dynamic)): 0.8 on the
# first layer, then 0.98 per layer.
RETAIN_DEN = 1000  # the synthetic retention ratios are given in thousandths


def retain_alphas(n_layers: int) -> list:
    """Numerators over RETAIN_DEN of the synthetic per-layer retention ratios: 0.8 on the first
    layer, then 0.98 per layer."""
    return [800] + [980] * (n_layers - 1)


def retained_tokens(n_tok: int, counts, seed: int) -> list:
    """Nested retained sets: a seeded ranking of the target tokens stands in for the attention
    scores; layer l keeps the counts[l] best-ranked tokens, listed in ascending order."""
    rank = rng(seed, 200).permutation(n_tok)
    return [np.sort(rank[:c]).astype(np.int32) for c in counts]
