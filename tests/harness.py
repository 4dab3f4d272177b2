"""Shared helpers of the GPU tests: run a workload through the CUDA path (via
the C ABI binding) and through the oracle, and compare."""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np

from oracle import compile_grammar


def unpack(mask_words: np.ndarray, V: int) -> np.ndarray:
    """[B, W] uint32 words -> [B, V] uint8 bits (LSB first)."""
    m = mask_words.astype(np.uint32).view(np.uint8).reshape(mask_words.shape[0], -1)
    bits = np.unpackbits(m, axis=1, bitorder="little")
    return bits[:, :V]


def pack_bits(bits: np.ndarray) -> np.ndarray:
    B, V = bits.shape
    W = (V + 31) // 32
    padded = np.zeros((B, W * 32), dtype=np.uint8)
    padded[:, :V] = bits
    return np.packbits(padded, axis=1, bitorder="little").view(np.uint32).reshape(B, W)


class GpuRun:
    """Compile + load + specialize + build B configurations from prefixes."""

    def __init__(self, wl, device="cuda:0"):
        import torch
        from paper_2607_11951_gb300 import grid as G
        self.G = G
        self.torch = torch
        self.wl = wl
        self.dev = torch.device(device)
        self.grammar = G.Grammar(wl["grammar"], wl["role"], wl["lexicons"], wl.get("max_depth", 4096))
        self.vocab = G.Vocab(wl["tokens"], wl["eos"], wl["specials"])
        self.spec = G.Spec(self.grammar, self.vocab)
        self.V = len(wl["tokens"])
        self.W = (self.V + 31) // 32
        self.B = len(wl["prefixes"])
        self.cfg = G.Configs(self.spec, self.B)
        self.status = torch.zeros(self.B, dtype=torch.int32, device=self.dev)
        self.mask = torch.zeros((self.B, self.W), dtype=torch.int32, device=self.dev)

    def build_configs(self, cfg=None, prefixes=None):
        """Advance every row through its prefix tokens in one launch."""
        torch = self.torch
        cfg = cfg or self.cfg
        prefixes = prefixes if prefixes is not None else self.wl["prefixes"]
        n = max(1, max(len(p) for p in prefixes))
        toks = np.full((len(prefixes), n), -1, dtype=np.int32)
        for i, p in enumerate(prefixes):
            toks[i, :len(p)] = p
        t = torch.from_numpy(toks).to(self.dev)
        cfg.reset()
        self.G.grid_advance(self.spec.h, cfg.h, cfg.h, t, self.status)
        torch.cuda.synchronize()
        return self.status.cpu().numpy().copy()

    def masks(self, cfg=None):
        torch = self.torch
        self.G.grid_masks(self.spec.h, (cfg or self.cfg).h, self.mask, self.status)
        torch.cuda.synchronize()
        words = self.mask.cpu().numpy().view(np.uint32)
        return words, self.status.cpu().numpy().copy()


# ---- oracle side (multiprocessing with spawn so CUDA state is never forked) ----
_OG = None
_VOCAB = None


def _init_worker(grammar, role, lexicons, vocab=None):
    """Worker set-up: the oracle grammar, and optionally (tokens, eos,
    specials) so that jobs need not carry the vocabulary."""
    global _OG, _VOCAB
    _OG = (compile_grammar(grammar, role, lexicons))
    _VOCAB = vocab


def _oracle_rows(args):
    if len(args) == 2:
        prefix, ids = args
        tokens, eos, specials = _VOCAB
    else:
        prefix, tokens, eos, specials, ids = args
    og = _OG
    cfg = og.config_from_ids(prefix, tokens, eos, specials)
    if cfg is None:
        return None
    return og.mask(cfg, tokens, eos, specials, ids=ids)


_CFG_CACHE = {}


def _oracle_rows_timed(args):
    """Like _oracle_rows, plus the seconds spent in the mask itself (building
    the configuration from its prefix is not part of a mask step)."""
    import time
    prefix, tokens, eos, specials, ids = args
    og = _OG
    key = tuple(prefix)
    if key not in _CFG_CACHE:
        _CFG_CACHE[key] = og.config_from_ids(prefix, tokens, eos, specials)
    cfg = _CFG_CACHE[key]
    if cfg is None:
        return None, 0.0
    t0 = time.perf_counter()
    bits = og.mask(cfg, tokens, eos, specials, ids=ids)
    return bits, time.perf_counter() - t0


def oracle_masks(wl, rows=None, ids_per_row=None, procs=None):
    """Oracle bits for the given rows (all by default) over all ids or the
    per-row id subsets ``ids_per_row``.  Returns a list of lists of bits."""
    rows = list(range(len(wl["prefixes"]))) if rows is None else rows
    jobs = []
    for k, r in enumerate(rows):
        ids = None if ids_per_row is None else list(ids_per_row[k])
        jobs.append((list(wl["prefixes"][r]), ids))
    vocab = (wl["tokens"], wl["eos"], wl["specials"])
    procs = procs or min(len(jobs), os.cpu_count() or 1)
    if procs <= 1:
        _init_worker(wl["grammar"], wl["role"], wl["lexicons"], vocab)
        return [_oracle_rows(j) for j in jobs]
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs, initializer=_init_worker,
                  initargs=(wl["grammar"], wl["role"], wl["lexicons"], vocab)) as pool:
        return pool.map(_oracle_rows, jobs, chunksize=1)


def oracle_masks_split(wl, rows=None, procs=None, parts=8):
    """Full oracle masks, splitting each row's vocabulary into ``parts`` jobs."""
    rows = list(range(len(wl["prefixes"]))) if rows is None else rows
    V = len(wl["tokens"])
    bounds = np.linspace(0, V, parts + 1).astype(int)
    jobs = []
    for r in rows:
        for a, b in zip(bounds[:-1], bounds[1:]):
            jobs.append((list(wl["prefixes"][r]), list(range(a, b))))
    procs = procs or (os.cpu_count() or 1)
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs, initializer=_init_worker,
                  initargs=(wl["grammar"], wl["role"], wl["lexicons"], (wl["tokens"], wl["eos"], wl["specials"]))) as pool:
        res = pool.map(_oracle_rows, jobs, chunksize=1)
    out = []
    for i in range(len(rows)):
        chunk = res[i * parts:(i + 1) * parts]
        if any(c is None for c in chunk):
            out.append(None)
        else:
            out.append([x for c in chunk for x in c])
    return out
