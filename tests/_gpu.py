"""Helpers of the GPU parity tests: device copies of generator inputs and the
output tolerance.  The CUDA path is always reached through the C ABI."""
from __future__ import annotations

import numpy as np
import torch

from paper_2608_17402_gb300 import moevie

# Output tolerance of the layer (bf16 inputs, fp32 accumulation, bf16 hidden
# activations and bf16 output): relative L2 error <= 1e-2 and every element within
# 5e-2 of the RMS of the oracle output.
REL_L2 = 1e-2
MAX_ABS_OF_RMS = 5e-2
# Oracle margins below this are not trusted to decide an exact tie-free order
# between two independent fp64 evaluations (summation order, libm vs CUDA exp).
MARGIN_PINNED = 1e-11


def dev_bf16(a_u16: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a_u16).view(np.int16)).view(torch.bfloat16).cuda()


def dev(a) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def to_np_f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def dev_rows(a_u16: np.ndarray) -> torch.Tensor:
    """bf16 [..., h] with the row stride the entry points take for W1, W3, Ws1, Ws3."""
    return moevie.moevie_pad_rows(dev_bf16(a_u16))


def layer_to_device(lay):
    W = moevie.LayerWeights(
        W_r=dev(lay.Wr), b=dev(lay.b), W1=dev_rows(lay.W1), W2=dev_bf16(lay.W2), k=lay.cfg.k,
        Ws1=None if lay.Ws1 is None else dev_rows(lay.Ws1),
        Ws2=None if lay.Ws2 is None else dev_bf16(lay.Ws2), lam=lay.cfg.lam,
        W3=None if lay.W3 is None else dev_rows(lay.W3),
        Ws3=None if lay.Ws3 is None else dev_rows(lay.Ws3))
    return dev_bf16(lay.x), W


def workspace_for(lay):
    c = lay.cfg
    return moevie.Workspace(c.T, c.d, c.E, c.k, c.h, c.h_s)


def assert_close(got: np.ndarray, want: np.ndarray, what: str = "y"):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (got.shape, want.shape)
    assert np.all(np.isfinite(got)), f"{what}: non-finite values"
    rms = float(np.sqrt(np.mean(want ** 2))) if want.size else 0.0
    err = got - want
    rel = float(np.linalg.norm(err) / max(np.linalg.norm(want), 1e-300))
    mx = float(np.abs(err).max()) if err.size else 0.0
    assert rel <= REL_L2, f"{what}: relative L2 error {rel:.3e} > {REL_L2}"
    assert mx <= MAX_ABS_OF_RMS * rms + 1e-30, f"{what}: max |err| {mx:.3e} > {MAX_ABS_OF_RMS} * RMS {rms:.3e}"
    return rel, mx / max(rms, 1e-300)


def check_status(ws):
    code, detail = moevie.moevie_get_device_status(ws)
    assert code == 0, f"device status {moevie.STATUS_NAMES.get(code, code)} detail={detail}"


def stratified_tokens(T, k, counts, offsets, perm, n_random=256, seed=0, bm=256, max_bands=16):
    """Output rows (tokens) to compare against the oracle on a full-size layer, chosen
    to cover the paths that only the full launch takes, by stratum:

    * ``last_tile``: for every non-empty expert, the first and last two rows of its
      last (usually partial) m-tile of ``bm`` rows;
    * ``hot``: rows on both sides of every m-tile boundary of the most loaded expert;
    * ``band_edges``: the tokens on both sides of every token-band boundary
      ``ceil(b T / nb)`` of a band-ordered down-projection, for every band count
      ``nb <= max_bands``;
    * ``small``: the rows of the eight least loaded non-empty experts (all of them,
      or the first and last 64 of a segment longer than 128);
    * ``random``: ``n_random`` uniformly drawn tokens.

    Returns the sorted unique tokens and a dict of stratum -> number of tokens."""
    counts = np.asarray(counts)
    offsets = np.asarray(offsets)
    perm = np.asarray(perm)
    strata = {}

    def rows_to_tokens(rows):
        rows = np.asarray([r for r in rows if 0 <= r < T * k], dtype=np.int64)
        return np.unique(perm[rows] // k) if rows.size else np.zeros(0, np.int64)

    rows = []
    for e in np.flatnonzero(counts > 0):
        c, o = int(counts[e]), int(offsets[e])
        first = o + (c - 1) // bm * bm
        rows += [first, first + 1, o + c - 2, o + c - 1]
    strata["last_tile"] = rows_to_tokens(rows)
    hot = int(np.argmax(counts))
    rows = []
    for m in range(bm, int(counts[hot]), bm):
        rows += [offsets[hot] + m - 1, offsets[hot] + m]
    strata["hot"] = rows_to_tokens(rows)
    edges = set()
    for nb in range(2, max_bands + 1):
        for b in range(1, nb):
            t0 = -(-b * T // nb)
            edges.update({t0 - 1, t0})
    strata["band_edges"] = np.array(sorted(t for t in edges if 0 <= t < T), np.int64)
    nz = np.flatnonzero(counts > 0)
    small = nz[np.argsort(counts[nz], kind="stable")[:8]]
    rows = []
    for e in small:   # every row, or the first and last 64 of a larger segment
        o, c = int(offsets[e]), int(counts[e])
        rows += list(range(o, o + c)) if c <= 128 else list(range(o, o + 64)) + list(range(o + c - 64, o + c))
    strata["small"] = rows_to_tokens(rows)
    strata["random"] = np.random.default_rng(seed).choice(T, min(n_random, T), replace=False)
    toks = np.unique(np.concatenate([v for v in strata.values()] + [np.array([0, T - 1])]))
    return toks.astype(np.int32), {k2: int(v.size) for k2, v in strata.items()}
