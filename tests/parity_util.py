"""Helpers for the GPU-vs-oracle parity tests: moving arrays between the two sides and the
near-tie exemption rules (code indices must match the fp64 oracle exactly except where the
oracle's own decision margin is below 1e-6 relative)."""
import numpy as np
import torch

from oracle import crvq_oracle as O

REL_TIE = 1e-6


def dev(a, dtype=None):
    t = torch.as_tensor(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def host(t):
    return t.detach().cpu().numpy()


def oracle_cbs(gpu_cbs):
    """GPU Codebook list -> oracle Codebook list (codes copied to host)."""
    out = []
    for cb in gpu_cbs:
        codes = None if cb.codes is None else host(cb.codes).astype(np.int64)
        out.append(O.Codebook(host(cb.C), codes, cb.G_cov))
    return out


def tuple_err(T, d, Hb, cbs, codes_of, i, g):
    """fp64 err of the tuple codes_of[s] (None -> fixed codebook's own code) at (i, g)."""
    t = np.asarray(T[i, g * d:(g + 1) * d], np.float64)
    r = t.copy()
    for s, cb in enumerate(cbs):
        if g >= cb.G_cov:
            continue
        k = codes_of[s]
        r -= cb.C[k].astype(np.float64)
    H = np.asarray(Hb[g], np.float64)
    return float(r @ H @ r), float(t @ H @ t)


def check_codes_with_ties(T, d, Hb, cbs_or, n_fixed, gpu_codes, or_codes, rel=REL_TIE):
    """Every vector whose searched tuple differs must be an fp64 near-tie: the oracle's err of
    the GPU tuple is within rel * (err_best + t^T H t) of the oracle's best err. Returns the
    number of exempted vectors."""
    M = T.shape[0]
    G_sub = Hb.shape[0]
    searched = list(range(n_fixed, len(cbs_or)))
    diff = np.zeros((M, G_sub), bool)
    for s in searched:
        G = cbs_or[s].G_cov
        diff[:, :G] |= gpu_codes[s][:, :G] != or_codes[s][:, :G]
    bad = []
    for i, g in zip(*np.nonzero(diff)):
        fixed = [cbs_or[s].codes[i, g] if s < n_fixed else None for s in range(len(cbs_or))]
        tg = list(fixed)
        to = list(fixed)
        for s in searched:
            if g < cbs_or[s].G_cov:
                tg[s] = gpu_codes[s][i, g]
                to[s] = or_codes[s][i, g]
        eg, tt = tuple_err(T, d, Hb, cbs_or, tg, i, g)
        eo, _ = tuple_err(T, d, Hb, cbs_or, to, i, g)
        if abs(eg - eo) > rel * (eo + tt):
            bad.append((int(i), int(g), eg, eo))
    assert not bad, f"{len(bad)} code mismatches beyond the near-tie exemption, e.g. {bad[:5]}"
    return int(diff.sum())


def beam_boundary_gap(t, Hg, Cs, B):
    """Smallest relative gap, over the stages of the oracle's stage-wise beam for one vector,
    between ranked partial tuples j and j+1 for j < B (only rank 0 vs 1 at the last stage)."""
    Hg = np.asarray(Hg, np.float64)
    tt = float(t @ Hg @ t)
    res = [np.asarray(t, np.float64)]
    gap = np.inf
    for si, C in enumerate(Cs):
        C = np.asarray(C, np.float64)
        errs, kids = [], []
        for h, r in enumerate(res):
            D = r[None, :] - C
            e = np.einsum("kd,kd->k", D @ Hg, D)
            errs.append(e)
            kids += [(h, k) for k in range(len(C))]
        e = np.concatenate(errs)
        order = np.argsort(e, kind="stable")
        last = si == len(Cs) - 1
        lim = 1 if last else min(B, len(e) - 1)
        for j in range(min(lim, len(e) - 1)):
            gap = min(gap, (e[order[j + 1]] - e[order[j]]) / (e[order[0]] + tt))
        keep = order[:min(B, len(e))]
        res = [res[kids[o][0]] - C[kids[o][1]] for o in keep]
    return gap
