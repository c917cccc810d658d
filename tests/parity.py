"""Element-by-element comparison of the CUDA commit step with the float64 oracle.

Tolerances are the stated ones: tokens and commit masks bit-exact except at
positions whose top-2 logits differ by less than 1e-3 or whose confidence is
within 2e-3 of a threshold; confidence within 2e-3 absolute for bf16 (and
fp32) weights, 1e-2 for FP8 weights. One addition: a block whose two highest
masked confidences are closer than the confidence tolerance may take its
top-1 fallback at either of them.
"""

from dataclasses import dataclass, field

import numpy as np

GAP_TOL = 1e-3
TAU_TOL = 2e-3
# NVFP4 heads decode exactly to bf16 on the device and take the bf16 path's arithmetic
CONF_TOL = {"f32": 2e-3, "bf16": 2e-3, "e4m3": 1e-2, "nvfp4": 2e-3}


@dataclass
class ParityReport:
    n_live: int = 0
    max_dconf: float = 0.0
    token_mismatch_exempt: int = 0
    commit_mismatch_exempt: int = 0
    failures: list = field(default_factory=list)

    def ok(self):
        return not self.failures


def compare(gpu, ref, taus, weight_dtype, block_len, n_slots, pos_masked=None, block_flags=None,
            max_exempt_frac=0.05):
    """gpu: dict of numpy arrays tokens/conf/commit(/counts); ref: oracle dict."""
    rep = ParityReport()
    ev = ref["evaluated"]
    tol = CONF_TOL[weight_dtype]
    taus32 = np.array([float(np.float32(t)) for t in taus])
    T = len(taus32)
    t_g, c_g = gpu["tokens"][ev], gpu["conf"][ev].astype(np.float64)
    k_g = gpu["commit"][ev].astype(np.uint32)
    t_r, c_r, k_r, gap = ref["tokens"][ev], ref["conf"][ev], ref["commit"][ev], ref["gap"][ev]
    live = t_r >= 0
    rep.n_live = int(live.sum())
    # positions without a prediction: exactly -1 / 0 / 0
    if not np.array_equal(t_g < 0, ~live):
        rep.failures.append(f"prediction set differs at {np.flatnonzero((t_g < 0) != ~live)[:10]}")
        return rep
    if np.any(c_g[~live] != 0) or np.any(k_g[~live] != 0) or np.any(t_g[~live] != -1):
        rep.failures.append("positions without a prediction are not -1/0/0")
    if rep.n_live:
        d = np.abs(c_g[live] - c_r[live])
        rep.max_dconf = float(d.max())
        if rep.max_dconf > tol:
            rep.failures.append(f"confidence off by {rep.max_dconf:.3e} > {tol}")
        if np.any((c_g[live] <= 0) | (c_g[live] > 1)):
            rep.failures.append("confidence outside (0, 1]")
    # tokens
    bad = live & (t_g != t_r)
    exempt = bad & (gap < GAP_TOL)
    rep.token_mismatch_exempt = int(exempt.sum())
    if np.any(bad & ~exempt):
        i = np.flatnonzero(bad & ~exempt)[:5]
        rep.failures.append(f"tokens differ at {i}: gpu {t_g[i]} oracle {t_r[i]} gap {gap[i]}")
    # commit masks, per bit
    idx_ev = np.flatnonzero(ev)
    blk_of = idx_ev // block_len
    fb_tol = tol
    for k in range(T):
        bg = (k_g >> np.uint32(k)) & 1
        br = (k_r >> np.uint32(k)) & 1
        diff = bg != br
        if not diff.any():
            continue
        ok = (gap < GAP_TOL) | (np.abs(c_r - taus32[k]) < TAU_TOL)
        for i in np.flatnonzero(diff & ~ok):
            b = blk_of[i]
            in_blk = (blk_of == b) & live
            cb = np.sort(c_r[in_blk])[::-1]
            near_tie = cb.size >= 2 and (cb[0] - cb[1]) < fb_tol
            if near_tie:
                ok[i] = True
        rep.commit_mismatch_exempt += int((diff & ok).sum())
        if np.any(diff & ~ok):
            i = np.flatnonzero(diff & ~ok)[:5]
            rep.failures.append(f"commit bit {k} (tau {taus32[k]}) differs at {idx_ev[i]}: "
                                f"gpu {bg[i]} oracle {br[i]} conf {c_r[i]}")
    n_ex = rep.token_mismatch_exempt
    if rep.n_live and n_ex > max(2, max_exempt_frac * rep.n_live):
        rep.failures.append(f"too many exempt token mismatches: {n_ex} of {rep.n_live}")
    # counts are the popcounts of the GPU's own commit masks
    if "counts" in gpu and gpu["counts"] is not None and ev.all():
        P = k_g.size
        per_seq = n_slots * block_len
        kk = gpu["commit"].astype(np.uint32).reshape(P // per_seq, per_seq)
        for k in range(T):
            pc = ((kk >> np.uint32(k)) & 1).sum(axis=1)
            if not np.array_equal(pc, gpu["counts"][:, k]):
                rep.failures.append(f"counts for tau {k} are not the popcounts of the commit masks")
                break
    return rep
