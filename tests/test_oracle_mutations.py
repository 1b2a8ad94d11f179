"""Planted mistakes in the oracle, on the CPU: each plausible slip (a dropped term or factor,
a wrong sign, index or scale, an operand left unpermuted, a sampling rule broken) is patched
into one oracle function for the duration of a test, and at least one of the pins in
test_oracle_pins.py must then fail. This checks that the pins constrain the oracle rather
than restate it. CPU only."""
import importlib.util
import os

import numpy as np
import pytest

from oracle import crvq_oracle as O

_HERE = os.path.dirname(os.path.abspath(__file__))
_spec = importlib.util.spec_from_file_location("oracle_pins_for_mutation",
                                               os.path.join(_HERE, "test_oracle_pins.py"))
pins = importlib.util.module_from_spec(_spec)
_spec.loader.exec_module(pins)


# ------------------------------------------------------------------ the planted mistakes
def _hessian_without_1_over_n(orig):
    def f(X, damp_rel, d):
        H, xsq, Hb, delta = orig(X, damp_rel, d)
        n = np.asarray(X).shape[0]
        return ((H * n).astype(np.float32), (xsq * n).astype(np.float32),
                (Hb * n).astype(np.float32), np.float32(delta * n))
    return f


def _hessian_damping_everywhere(orig):
    def f(X, damp_rel, d):
        H, xsq, Hb, delta = orig(X, damp_rel, d)
        N = H.shape[0]
        H2 = (H + float(delta) * (np.ones((N, N)) - np.eye(N))).astype(np.float32)
        Hb2 = np.stack([H2[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(N // d)])
        return H2, xsq, Hb2, delta
    return f


def _hessian_delta_from_sum(orig):
    def f(X, damp_rel, d):
        H, xsq, Hb, delta = orig(X, damp_rel, d)
        N = H.shape[0]
        extra = float(delta) * (N - 1)
        return ((H + extra * np.eye(N)).astype(np.float32), xsq,
                (Hb + extra * np.eye(d)).astype(np.float32), np.float32(delta * N))
    return f


def _encode_plus_instead_of_minus(orig):
    """err = (t + c)^T H (t + c): the codeword's sign flipped in the residual."""
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        neg = [O.Codebook(-np.asarray(cb.C), cb.codes, cb.G_cov) for cb in cbs]
        return orig(T, d, H_blocks, neg, n_fixed, B, keep_if_better, **kw)
    return f


def _encode_ignores_H(orig):
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        eye = np.broadcast_to(np.eye(d, dtype=np.float32), np.shape(H_blocks)).copy()
        return orig(T, d, eye, cbs, n_fixed, B, keep_if_better, **kw)
    return f


def _encode_ignores_fixed(orig):
    """The fixed codebooks' codewords are not subtracted from the target."""
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        if n_fixed == 0:
            return orig(T, d, H_blocks, cbs, n_fixed, B, keep_if_better, **kw)
        free = [O.Codebook(cb.C, None if not keep_if_better else cb.codes, cb.G_cov)
                for cb in cbs[n_fixed:]]
        codes, verr = orig(T, d, H_blocks, free, 0, B, keep_if_better, **kw)
        return [cb.codes for cb in cbs[:n_fixed]] + list(codes), verr
    return f


def _update_ignores_H(orig):
    def f(T, d, H_blocks, cbs, which):
        eye = np.broadcast_to(np.eye(d, dtype=np.float32), np.shape(H_blocks)).copy()
        return orig(T, d, eye, cbs, which)
    return f


def _update_zeroes_empty_clusters(orig):
    def f(T, d, H_blocks, cbs, which):
        C, counts = orig(T, d, H_blocks, cbs, which)
        C = np.array(C, copy=True)
        C[np.asarray(counts) == 0] = 0
        return C, counts
    return f


def _update_residual_sign(orig):
    """The other codebooks' codewords are added to the target instead of subtracted."""
    def f(T, d, H_blocks, cbs, which):
        flipped = [cb if s == which else O.Codebook(-np.asarray(cb.C), cb.codes, cb.G_cov)
                   for s, cb in enumerate(cbs)]
        return orig(T, d, H_blocks, flipped, which)
    return f


def _importance_without_half(orig):
    def f(W, W_pre, xsq, mode, seed, hinv=None):
        return orig(W, W_pre, xsq, mode, seed, hinv) * 2.0
    return f


def _importance_mean_over_rows(orig):
    """Mean over the output rows instead of the maximum."""
    def f(W, W_pre, xsq, mode, seed, hinv=None):
        if mode != O.MODE_WA:
            return orig(W, W_pre, xsq, mode, seed, hinv)
        dW = np.asarray(W, np.float64) - np.asarray(W_pre, np.float64)
        return 0.5 * np.asarray(xsq, np.float64) * (dW ** 2).mean(axis=0)
    return f


def _reorder_ascending(orig):
    def f(W, d, W_pre, xsq, H, crit_frac, mode, seed):
        perm, I, Ws, Hb, Gc = orig(W, d, W_pre, xsq, H, crit_frac, mode, seed)
        p = np.ascontiguousarray(perm[::-1])
        Hp = np.asarray(H)[np.ix_(p, p)]
        Hb2 = np.stack([Hp[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(len(p) // d)])
        return p, I, np.asarray(W)[:, p], Hb2, Gc
    return f


def _reorder_blocks_unpermuted(orig):
    def f(W, d, W_pre, xsq, H, crit_frac, mode, seed):
        perm, I, Ws, Hb, Gc = orig(W, d, W_pre, xsq, H, crit_frac, mode, seed)
        H = np.asarray(H)
        Hb2 = np.stack([H[g * d:(g + 1) * d, g * d:(g + 1) * d] for g in range(len(perm) // d)])
        return perm, I, Ws, Hb2, Gc
    return f


def _loss_full_block_only(orig):
    def f(W_sorted, d, H_blocks, perm, cbs, G_c, X=None, delta=0.0):
        W_hat, lb, lc, lf = orig(W_sorted, d, H_blocks, perm, cbs, G_c, X, delta)
        return W_hat, lb, lc, (lb if lf is not None else lf)
    return f


def _loss_full_without_damping(orig):
    def f(W_sorted, d, H_blocks, perm, cbs, G_c, X=None, delta=0.0):
        return orig(W_sorted, d, H_blocks, perm, cbs, G_c, X, 0.0)
    return f


def _sample_indices_not_stratified(orig):
    def f(n, K, seed):
        return np.sort(np.random.default_rng(seed).choice(n, K, replace=False))
    return f


def _init_residual_sign(orig):
    def f(T, d, G_sub, K, seed, fixed=()):
        flipped = [O.Codebook(-np.asarray(cb.C), cb.codes, cb.G_cov) for cb in fixed]
        return orig(T, d, G_sub, K, seed, fixed=flipped)
    return f


def _avg_bits_without_extended(orig):
    def f(e, d, m, lam, M=4096, N=4096, include_perm=False, n_base=1):
        return orig(e, d, 1, lam, M, N, include_perm, n_base)
    return f


def _avg_bits_one_base(orig):
    """Every further base codebook's codes and codewords left out of the count."""
    def f(e, d, m, lam, M=4096, N=4096, include_perm=False, n_base=1):
        return orig(e, d, m, lam, M, N, include_perm, 1)
    return f


def _crit_groups_floor(orig):
    def f(N, d, crit_frac):
        return min(N // d, int(np.floor(np.float32(crit_frac) * N / d)))
    return f


def _splitmix64_wrong_constant(orig):
    def f(stream, counter):
        return orig(stream, counter) ^ 1
    return f


def _hinv_is_diag_of_H(orig):
    """The inverse forgotten: diag(H) instead of diag(H^-1)."""
    def f(H):
        return np.diag(np.asarray(H, np.float64)).copy()
    return f


def _hinv_ignores_correlations(orig):
    """1 / H_ii: the inverse of the diagonal, not the diagonal of the inverse."""
    def f(H):
        return 1.0 / np.diag(np.asarray(H, np.float64))
    return f


def _eq_wa_multiplies(orig):
    """Eq. (wa) with the inverse-Hessian diagonal in the numerator."""
    def f(W, W_pre, xsq, mode, seed, hinv=None):
        if mode != O.MODE_WA_INV:
            return orig(W, W_pre, xsq, mode, seed, hinv)
        dW = np.asarray(W, np.float64) - np.asarray(W_pre, np.float64)
        return np.max(dW * dW, axis=0) * np.asarray(hinv, np.float64) / 2.0
    return f


def _coupled_variant(shift_sign, exclude_own_block):
    """The coupled Gauss-Seidel sweep with one slip: the shift H_gg^-1 b_g subtracted instead
    of added, or b_g formed with the group's own block left in."""
    def plant(orig):
        def f(W_sorted, d, H_sorted, cbs, which, sweeps=1):
            W = np.asarray(W_sorted, np.float64)
            H = np.asarray(H_sorted, np.float64)
            M, N = W.shape
            cb = cbs[which]
            C = cb.C.astype(np.float64)
            codes = cb.codes.copy()
            cur = [O.Codebook(c.C, c.codes, c.G_cov) for c in cbs]
            cur[which] = O.Codebook(cb.C, codes, cb.G_cov)
            D = W - O.decode(M, N, d, cur)
            hist = []
            for _ in range(sweeps):
                for g in range(cb.G_cov):
                    sl = slice(g * d, (g + 1) * d)
                    Hgg = H[sl, sl]
                    b = D @ H[:, sl] - (D[:, sl] @ Hgg if exclude_own_block else 0.0)
                    t = D[:, sl] + C[codes[:, g]]
                    shift = shift_sign * np.linalg.solve(Hgg, b.T).T
                    k = np.argmin(O.quad_err(t + shift, C, Hgg), axis=1)
                    codes[:, g] = k
                    D[:, sl] = t - C[k]
                    hist.append(float(np.einsum("ij,jk,ik->", D, H, D)))
            return codes, hist
        return f
    return plant


def _lut_inverse_perm(orig):
    """Inputs permuted with the inverse order."""
    def f(Xin, perm, cbs, d):
        return orig(Xin, None if perm is None else np.argsort(perm), cbs, d)
    return f


def _lut_base_only(orig):
    """Extended codebooks left out of the product."""
    def f(Xin, perm, cbs, d):
        return orig(Xin, perm, cbs[:1], d)
    return f


def _ties_to_larger_index(orig):
    """Equal errors resolved toward the larger codeword index (codebooks searched reversed)."""
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        rev = []
        for s, cb in enumerate(cbs):
            K = cb.C.shape[0]
            codes = None if cb.codes is None else (K - 1 - cb.codes)
            rev.append(O.Codebook(cb.C[::-1], codes, cb.G_cov))
        codes, verr = orig(T, d, H_blocks, rev, n_fixed, B, keep_if_better, **kw)
        return [cb.C.shape[0] - 1 - c for cb, c in zip(cbs, codes)], verr
    return f


def _beam_width_ignored(orig):
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        return orig(T, d, H_blocks, cbs, n_fixed, 1, keep_if_better, **kw)
    return f


def _keep_if_better_ignored(orig):
    def f(T, d, H_blocks, cbs, n_fixed, B, keep_if_better=False, **kw):
        if keep_if_better:
            cbs = [cb if s < n_fixed else O.Codebook(cb.C, None, cb.G_cov)
                   for s, cb in enumerate(cbs)]
        return orig(T, d, H_blocks, cbs, n_fixed, B, False, **kw)
    return f


def _reconstruction_forward_perm(orig):
    """The sorted reconstruction is scattered back with perm instead of its inverse."""
    def f(W_sorted, d, H_blocks, perm, cbs, G_c, X=None, delta=0.0):
        W_hat, lb, lc, lf = orig(W_sorted, d, H_blocks, perm, cbs, G_c, X, delta)
        if perm is not None:
            W_hat = np.asarray(W_hat)[:, perm][:, perm]
        return W_hat, lb, lc, lf
    return f


def _schedule_variant(slip):
    """The per-matrix schedule with one wiring slip: the base codebook fitted on W instead of
    the reordered W ("base_on_W"), warm-started from the prequantize codebook ("warm_start"),
    extended codebooks fitted on the raw critical vectors instead of the residual of the base
    ("ext_without_base"), the refinement updating the codebooks in reverse order
    ("refine_reversed"), a second base codebook fitted on the reordered W instead of the
    residual of the first ("base2_on_W_sorted") or on the critical groups only
    ("base2_critical_only"). Otherwise the same steps as the oracle's quantize_layer."""
    def plant(orig):
        def f(W, X, cfg):
            d = cfg.d
            W = np.asarray(W, dtype=np.float32)
            M, N = W.shape
            G = N // d
            out = {}
            H, xsq, Hb0, delta = O.hessian(X, cfg.damp_rel, d)
            C0 = O.kmeans_init(W, d, G, cfg.K_base, O.phase_seed(cfg.seed, O.PHASE_PREQUANT, 0))
            pre, _ = O.lloyd(W, d, Hb0, [], C0, G, cfg.kmeans_iters)
            W_pre, pre_loss, _, _ = O.reconstruct_error(W, d, Hb0, None, [pre], 0)
            out.update(C_pre=pre.C, codes_pre=pre.codes, W_pre=W_pre, loss_pre=pre_loss)
            perm, I, Ws, Hb, Gc = O.select_reorder_channels(
                W, d, W_pre, xsq, H, cfg.crit_frac, cfg.importance_mode,
                O.phase_seed(cfg.seed, O.PHASE_RANDOM, 0))
            out.update(perm=perm, importance=I, W_sorted=Ws, H_blocks=Hb, n_crit_groups=Gc)
            T_base = W if slip == "base_on_W" else Ws
            if slip == "warm_start":
                Cb0 = pre.C
            else:
                Cb0 = O.kmeans_init(T_base, d, G, cfg.K_base,
                                    O.phase_seed(cfg.seed, O.PHASE_BASE, 0))
            base, obj = O.lloyd(T_base, d, Hb, [], Cb0, G, cfg.kmeans_iters)
            out["base_objective"] = obj
            cbs = [base]
            for b in range(1, getattr(cfg, "n_base", 1)):
                if slip == "base2_on_W_sorted":        # not on the residual of base 1
                    fixed, Gb = [], G
                elif slip == "base2_critical_only":    # only the critical groups
                    fixed, Gb = [O.Codebook(cb.C, cb.codes[:, :Gc], Gc) for cb in cbs], Gc
                else:
                    fixed, Gb = list(cbs), G
                Tb = Ws[:, :Gb * d]
                Cb0 = O.kmeans_init(Tb, d, Gb, cfg.K_base,
                                    O.phase_seed(cfg.seed, O.PHASE_BASE, b), fixed)
                nb, _ = O.lloyd(Tb, d, Hb[:Gb], fixed, Cb0, Gb, cfg.kmeans_iters)
                cbs.append(nb)
            Tc, Hbc = Ws[:, :Gc * d], Hb[:Gc]
            for t in range(1, cfg.n_ext + 1):
                fixed = [] if slip == "ext_without_base" else \
                    [O.Codebook(cb.C, cb.codes[:, :Gc], Gc) for cb in cbs]
                Ct0 = O.kmeans_init(Tc, d, Gc, cfg.K_ext, O.phase_seed(cfg.seed, O.PHASE_EXT, t),
                                    fixed)
                ext, _ = O.lloyd(Tc, d, Hbc, fixed, Ct0, Gc, cfg.kmeans_iters)
                cbs.append(O.Codebook(ext.C, ext.codes, Gc))
            _, lb, _, _ = O.reconstruct_error(Ws, d, Hb, perm, cbs, Gc)
            history = [lb]
            order = range(len(cbs))
            for _ in range(cfg.refine_rounds):
                for j in (reversed(order) if slip == "refine_reversed" else order):
                    C, _ = O.update_codebook(Ws, d, Hb, cbs, j)
                    cbs[j] = O.Codebook(C, cbs[j].codes, cbs[j].G_cov)
                codes, _ = O.encode_beam(Ws, d, Hb, cbs, n_fixed=0, B=cfg.B, keep_if_better=True)
                cbs = [O.Codebook(cb.C, codes[q], cb.G_cov) for q, cb in enumerate(cbs)]
                _, lb, _, _ = O.reconstruct_error(Ws, d, Hb, perm, cbs, Gc)
                history.append(lb)
            out["loss_history"] = history
            W_hat, lb, lc, lf = O.reconstruct_error(Ws, d, Hb, perm, cbs, Gc, X, float(delta))
            out.update(codebooks=cbs, W_hat=W_hat, loss_block=lb, loss_crit=lc, loss_full=lf)
            return out
        return f
    return plant


_SCHEDULE_PINS = ["test_schedule_with_one_codeword_per_codebook_is_a_sequence_of_weighted_means",
                  "test_schedule_without_lloyd_iterations_keeps_the_sampled_codewords",
                  "test_schedule_with_a_codeword_per_vector_reconstructs_exactly"]
_TWO_BASE_PINS = ["test_schedule_with_two_base_codebooks_of_one_codeword_each",
                  "test_schedule_with_two_base_codebooks_without_lloyd_iterations"]


# (name, oracle attribute, planted version, pins that must catch it: a test name, or a test
# name with its arguments)
MUTATIONS = [
    ("hessian: 1/n dropped", "hessian", _hessian_without_1_over_n,
     ["test_hessian_closed_form_scaled_identity", "test_hessian_matches_matrix_free_product"]),
    ("hessian: damping on every entry", "hessian", _hessian_damping_everywhere,
     ["test_hessian_closed_form_scaled_identity", "test_hessian_matches_matrix_free_product"]),
    ("hessian: delta from the sum, not the mean", "hessian", _hessian_delta_from_sum,
     ["test_hessian_closed_form_scaled_identity", "test_hessian_matches_matrix_free_product"]),
    ("encode: t + c instead of t - c", "encode_beam", _encode_plus_instead_of_minus,
     ["test_encode_isotropic_is_euclidean_nearest_codeword",
      "test_encode_general_H_equals_whitened_nearest_codeword"]),
    ("encode: H ignored", "encode_beam", _encode_ignores_H,
     ["test_encode_isotropic_is_euclidean_nearest_codeword",
      "test_encode_general_H_equals_whitened_nearest_codeword"]),
    ("encode: fixed codebooks not subtracted", "encode_beam", _encode_ignores_fixed,
     ["test_encode_with_fixed_codebook_equals_encode_of_residual"]),
    ("update: H ignored (plain cluster mean)", "update_codebook", _update_ignores_H,
     ["test_update_is_a_minimiser_and_single_member_is_exact"]),
    ("update: empty clusters zeroed", "update_codebook", _update_zeroes_empty_clusters,
     ["test_update_isotropic_is_cluster_mean"]),
    ("update: residual with the wrong sign", "update_codebook", _update_residual_sign,
     ["test_update_of_second_codebook_targets_residual"]),
    ("importance: factor 1/2 dropped", "importance", _importance_without_half,
     ["test_importance_wa_equals_literal_app_a2_sum"]),
    ("importance: mean over rows instead of max", "importance", _importance_mean_over_rows,
     ["test_importance_wa_equals_literal_app_a2_sum"]),
    ("reorder: ascending importance", "select_reorder_channels", _reorder_ascending,
     ["test_reorder_bijection_roundtrip_and_blocks"]),
    ("reorder: H blocks taken unpermuted", "select_reorder_channels",
     _reorder_blocks_unpermuted, ["test_reorder_bijection_roundtrip_and_blocks"]),
    ("losses: loss_full without cross-group terms", "reconstruct_error", _loss_full_block_only,
     ["test_loss_full_two_routes_and_block_loss_matches_encode"]),
    ("losses: damping left out of the X route", "reconstruct_error",
     _loss_full_without_damping, ["test_loss_full_two_routes_and_block_loss_matches_encode"]),
    ("init: indices not stratified", "kmeans_sample_indices", _sample_indices_not_stratified,
     ["test_kmeans_init_strata_distinct_deterministic"]),
    ("init: residual with the wrong sign", "kmeans_init", _init_residual_sign,
     ["test_kmeans_init_takes_sampled_vectors_and_residuals"]),
    ("bit-width: extended codebooks dropped", "avg_bits", _avg_bits_without_extended,
     ["test_avg_bits_paper_values"]),
    ("bit-width: one base codebook counted", "avg_bits", _avg_bits_one_base,
     ["test_avg_bits_of_base_codebooks_alone_is_sec_3_2_eq_bitwidth"]),
    ("critical groups: floor instead of ceiling", "n_crit_groups", _crit_groups_floor,
     ["test_n_crit_groups_closed_form"]),
    ("splitmix64: wrong output", "splitmix64", _splitmix64_wrong_constant,
     ["test_splitmix64_published_sequence"]),
    ("beam: width ignored", "encode_beam", _beam_width_ignored,
     [("test_beam_with_full_width_equals_exhaustive_search", (4, 2, 4)),
      ("test_beam_with_full_width_equals_exhaustive_search", (4, 3, 2))]),
    ("encode: ties to the larger index", "encode_beam", _ties_to_larger_index,
     ["test_beam_ties_follow_err_then_parent_rank_then_index"]),
    ("beam: keep-if-better ignored", "encode_beam", _keep_if_better_ignored,
     ["test_narrow_beam_never_beats_exhaustive_and_keep_if_better_keeps_optimum"]),
    ("losses: reconstruction scattered with perm, not its inverse", "reconstruct_error",
     _reconstruction_forward_perm, ["test_loss_full_two_routes_and_block_loss_matches_encode"]),
    ("Eq. (wa): diag(H) for diag(H^-1)", "hinv_diag", _hinv_is_diag_of_H,
     ["test_hinv_diag_closed_forms", "test_hinv_diag_equals_schur_complement"]),
    ("Eq. (wa): 1 / H_ii for [H^-1]_ii", "hinv_diag", _hinv_ignores_correlations,
     ["test_hinv_diag_closed_forms", "test_hinv_diag_equals_schur_complement"]),
    ("Eq. (wa): inverse diagonal multiplied, not divided", "importance", _eq_wa_multiplies,
     ["test_importance_eq_wa_is_app_a2_for_uncorrelated_channels"]),
    ("inference: inputs permuted with the inverse order", "lut_matvec", _lut_inverse_perm,
     ["test_lut_matvec_equals_the_reconstructed_matrix_times_the_input"]),
    ("inference: extended codebooks left out", "lut_matvec", _lut_base_only,
     ["test_lut_matvec_equals_the_reconstructed_matrix_times_the_input"]),
    ("coupled search: shift subtracted", "coupled_sweep", _coupled_variant(-1.0, True),
     ["test_coupled_sweep_never_raises_the_full_loss",
      "test_coupled_sweep_fixed_point_is_optimal_per_group_by_brute_force",
      "test_coupled_sweep_between_exhaustive_optimum_and_block_diagonal_start"]),
    ("coupled search: own block left in the coupling", "coupled_sweep",
     _coupled_variant(1.0, False),
     ["test_coupled_sweep_never_raises_the_full_loss",
      "test_coupled_sweep_fixed_point_is_optimal_per_group_by_brute_force",
      "test_coupled_sweep_between_exhaustive_optimum_and_block_diagonal_start"]),
    ("schedule: base codebook fitted on W, not the reordered W", "quantize_layer",
     _schedule_variant("base_on_W"), _SCHEDULE_PINS),
    ("schedule: base k-means warm-started from the prequantize codebook", "quantize_layer",
     _schedule_variant("warm_start"), _SCHEDULE_PINS),
    ("schedule: extended codebooks fitted without subtracting the base", "quantize_layer",
     _schedule_variant("ext_without_base"), _SCHEDULE_PINS),
    ("schedule: refinement updates the codebooks in reverse order", "quantize_layer",
     _schedule_variant("refine_reversed"), _SCHEDULE_PINS),
    ("schedule: second base codebook fitted on the reordered W, not the residual",
     "quantize_layer", _schedule_variant("base2_on_W_sorted"), _TWO_BASE_PINS),
    ("schedule: second base codebook on the critical groups only", "quantize_layer",
     _schedule_variant("base2_critical_only"), _TWO_BASE_PINS),
]


def _run_pin(spec):
    name, args = (spec, ()) if isinstance(spec, str) else spec
    getattr(pins, name)(*args)


def test_every_pin_named_here_passes_on_the_unmodified_oracle():
    for spec in sorted({p for *_, ps in MUTATIONS for p in ps}, key=str):
        _run_pin(spec)


@pytest.mark.parametrize("label,attr,plant,pin_names", MUTATIONS,
                         ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_fails_a_pin(monkeypatch, label, attr, plant, pin_names):
    monkeypatch.setattr(O, attr, plant(getattr(O, attr)))
    caught = []
    for spec in pin_names:
        try:
            _run_pin(spec)
        except AssertionError:  # a pin's own check, not an error of the planted code
            caught.append(spec)
    assert caught, f"no pin caught the planted mistake: {label}"
