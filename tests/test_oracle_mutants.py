"""The oracle's pins catch plausible mistakes.

Each mutant is a copy of oracle/olive_oracle.py with one planted mistake (an
off-by-one mask, a dropped term, a wrong sign, a missing factor, swapped
directions, a wrong denominator).  The pin checks below restate the pins of
test_oracle_pins.py as functions of the oracle module; all of them must hold
for the real oracle and at least one must fail for every mutant.  Everything
runs on the CPU.
"""

import json
import math
import os
import types

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

import oracle.olive_oracle as real

SRC = real.__file__
GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "splice_pack_small.json")
GOLDEN_TURNS = os.path.join(os.path.dirname(__file__), "golden", "splice_pack_turns.json")

MUTANTS = {
    "mask_includes_prefix_target": ("in_loss = i + 1 >= P\n", "in_loss = i + 1 >= P - 1\n"),
    "turn_flag_off_by_one": ("in_loss = bool(cont_loss[cont_off[s] + (i + 1 - P)])",
                             "in_loss = bool(cont_loss[cont_off[s] + (i - P)])"),
    "target_not_shifted": ("targets.append(seq[i + 1])", "targets.append(seq[i])"),
    "cut_at_prefix_start": ("cut.append(cu[-1] + P)", "cut.append(cu[-1])"),
    "lse_drops_log_sum": ("lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))", "lse = m"),
    "logits_skip_temperature": ("    z *= float(inv_tau)\n", "    z *= 1.0\n"),
    "grad_drops_onehot": ("        G[np.arange(len(rr)), targets[rr]] -= 1.0\n        G *= g * float(inv_tau)\n        dH[rr] = G @ W64",
                          "        G *= g * float(inv_tau)\n        dH[rr] = G @ W64"),
    "grad_wrong_sign": ("        G *= g * float(inv_tau)\n        dH[rr] = G @ W64",
                        "        G *= -g * float(inv_tau)\n        dH[rr] = G @ W64"),
    "grad_drops_inv_tau": ("        G *= g * float(inv_tau)\n        dH[rr] = G @ W64",
                           "        G *= g\n        dH[rr] = G @ W64"),
    "dW_transposed_pairing": ("        dW += G.T @ h\n", "        dW += G.T @ h[::-1]\n"),
    "mean_over_all_rows": ("        loss = loss / len(rows) if len(rows) else 0.0",
                           "        loss = loss / len(targets) if len(rows) else 0.0"),
    "kl_directions_swapped": ("            k = (ps * (lps - lpt)).sum(axis=1)",
                              "            k = (pt * (lpt - lps)).sum(axis=1)"),
    "kl_grad_drops_kl_term": ("                dz = ps * (lps - lpt - k[:, None])",
                              "                dz = ps * (lps - lpt)"),
    "kl_grad_forward_sign": ("                dz = ps - pt", "                dz = pt - ps"),
    "topk_grad_drops_mass_term": ("            G[k] = -ps[k] * (kl + P_S)", "            G[k] = -ps[k] * kl"),
    "topk_grad_drops_plus_one": ("(lps[k, S] - lpt[k, S] + 1.0)", "(lps[k, S] - lpt[k, S])"),
    "entropy_wrong_sign": ("H[rr] = -(np.exp(lp) * lp).sum(axis=1)", "H[rr] = (np.exp(lp) * lp).sum(axis=1)"),
    "topk_ties_by_descending_id": ("order = np.lexsort((ids, -lp[k]))[:K]",
                                   "order = np.lexsort((-ids, -lp[k]))[:K]"),
    "topk_takes_smallest": ("order = np.lexsort((ids, -lp[k]))[:K]", "order = np.lexsort((ids, lp[k]))[:K]"),
    "overlap_over_union": ("overlap[r] = len(set(S.tolist()) & set(Tk.tolist())) / K",
                           "overlap[r] = len(set(S.tolist()) & set(Tk.tolist())) / "
                           "len(set(S.tolist()) | set(Tk.tolist()))"),
    "topk_kl_renormalised": ("kl[r] = float((np.exp(lps[k, S]) * (lps[k, S] - lpt[k, S])).sum())",
                             "ls_ = lps[k, S] - np.logaddexp.reduce(lps[k, S]); "
                             "lt_ = lpt[k, S] - np.logaddexp.reduce(lpt[k, S]); "
                             "kl[r] = float((np.exp(ls_) * (ls_ - lt_)).sum())"),
}


def load_variant(name=None):
    with open(SRC) as f:
        text = f.read()
    if name is not None:
        old, new = MUTANTS[name]
        assert text.count(old) == 1, f"mutation site for {name} not unique"
        text = text.replace(old, new)
    mod = types.ModuleType(f"oracle_variant_{name}")
    exec(compile(text, SRC, "exec"), mod.__dict__)
    return mod


def _case(seed, T=10, d=12, V=41):
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((T, d))
    W = rng.standard_normal((V, d)) * 0.3
    targets = rng.integers(0, V, size=T)
    rows = np.sort(rng.choice(T, size=T // 2, replace=False))
    return h, W, targets, rows


# ----------------------------------------------------------------- pin checks
def pin_golden_splice(O):
    with open(GOLDEN) as f:
        g = json.load(f)
    out = O.splice_pack(g["prefix_ids"], g["prefix_off"], g["cont_ids"], g["cont_off"], g["V"])
    return all(list(map(int, np.atleast_1d(out[k]))) == (v if isinstance(v, list) else [v])
               for k, v in g["expect"].items())


def pin_turns_golden(O):
    with open(GOLDEN_TURNS) as f:
        g = json.load(f)
    out = O.splice_pack(g["prefix_ids"], g["prefix_off"], g["cont_ids"], g["cont_off"], g["V"],
                        cont_loss=g["cont_loss"])
    return all(list(map(int, np.atleast_1d(out[k]))) == (v if isinstance(v, list) else [v])
               for k, v in g["expect"].items())


def pin_uniform(O):
    h = np.random.default_rng(0).standard_normal((5, 8))
    logp, _, loss = O.token_logprob(h, np.zeros((64, 8)), np.arange(5), np.arange(5))
    return np.allclose(logp, -math.log(64), atol=1e-12) and abs(loss - 5 * math.log(64)) < 1e-9


def pin_scipy(O):
    h, W, t, r = _case(1)
    logp, lse, _ = O.token_logprob(h, W, t, r, inv_tau=1.3)
    z = 1.3 * h @ W.T
    ref = scipy.special.log_softmax(z, axis=1)
    return (np.allclose(logp[r], ref[r, t[r]], atol=1e-10)
            and np.allclose(lse[r], scipy.special.logsumexp(z, axis=1)[r], atol=1e-10))


def pin_torch_ce_and_autograd(O):
    ok = True
    for red in ("sum", "mean"):
        h, W, t, r = _case(2)
        _, _, loss = O.token_logprob(h, W, t, r, inv_tau=1.5, reduction=red)
        dH, dW = O.token_loss_bwd(h, W, t, r, inv_tau=1.5, reduction=red, grad_loss=0.7)
        ht = torch.from_numpy(h).requires_grad_(True)
        Wt = torch.from_numpy(W).requires_grad_(True)
        z = 1.5 * (ht[torch.from_numpy(r)] @ Wt.T)
        ref = F.cross_entropy(z, torch.from_numpy(t[r]), reduction=red)
        (0.7 * ref).backward()
        ok &= abs(loss - ref.item()) < 1e-9 * max(1.0, abs(ref.item()))
        ok &= np.allclose(dH, ht.grad.numpy(), atol=1e-12) and np.allclose(dW, Wt.grad.numpy(), atol=1e-12)
    return bool(ok)


def pin_kl(O):
    ok = True
    rng = np.random.default_rng(3)
    hs, Ws = rng.standard_normal((6, 7)), rng.standard_normal((30, 7)) * 0.5
    ht, Wt = rng.standard_normal((6, 9)), rng.standard_normal((30, 9)) * 0.5
    r = np.array([0, 2, 5])
    for direction in ("reverse", "forward"):
        kl, dHs = O.token_divergence(hs, Ws, ht, Wt, r, 1.1, direction, grad_kl=np.ones(6))
        hs_t = torch.from_numpy(hs).requires_grad_(True)
        lps = F.log_softmax(1.1 * (hs_t[torch.from_numpy(r)] @ torch.from_numpy(Ws).T), 1)
        lpt = F.log_softmax(1.1 * (torch.from_numpy(ht)[torch.from_numpy(r)] @ torch.from_numpy(Wt).T), 1)
        if direction == "reverse":
            ref = F.kl_div(lpt, lps, log_target=True, reduction="none").sum(1)
        else:
            ref = F.kl_div(lps, lpt, log_target=True, reduction="none").sum(1)
        ref.sum().backward()
        ok &= np.allclose(kl[r], ref.detach().numpy(), atol=1e-12)
        ok &= np.allclose(dHs, hs_t.grad.numpy(), atol=1e-12)
    return bool(ok)


def pin_topk_kl_grad(O):
    rng = np.random.default_rng(4)
    hs, Ws = rng.standard_normal((5, 6)), rng.standard_normal((25, 6)) * 0.6
    ht, Wt = rng.standard_normal((5, 8)), rng.standard_normal((25, 8)) * 0.6
    r = np.array([1, 2, 4])
    dH, dW = O.token_topk_kl_bwd(hs, Ws, ht, Wt, r, 5, inv_tau=0.9)
    hs_t = torch.from_numpy(hs).requires_grad_(True)
    Ws_t = torch.from_numpy(Ws).requires_grad_(True)
    rr = torch.from_numpy(r)
    lps = F.log_softmax(0.9 * (hs_t[rr] @ Ws_t.T), 1)
    lpt = F.log_softmax(0.9 * (torch.from_numpy(ht)[rr] @ torch.from_numpy(Wt).T), 1)
    S = torch.topk(lps.detach(), 5, dim=1).indices
    ls, lt = lps.gather(1, S), lpt.gather(1, S)
    (ls.exp() * (ls - lt)).sum().backward()
    return bool(np.allclose(dH, hs_t.grad.numpy(), atol=1e-12)
                and np.allclose(dW, Ws_t.grad.numpy(), atol=1e-12))


def pin_topk_closed_forms(O):
    """Uniform logits (entropy ln V, ties by ascending id) and a three-token row whose
    top-K overlap, truncated KL, top-K log-probs and entropy are worked out by hand."""
    V = 50
    h = np.random.default_rng(5).standard_normal((2, 3))
    _, H, tv, ti = O.token_topk(h, np.zeros((V, 3)), [0, 1], 4)
    ok = np.allclose(H, math.log(V), atol=1e-12) and np.array_equal(ti, np.tile(np.arange(4), (2, 1)))
    ok &= np.allclose(tv, -math.log(V), atol=1e-12)
    hs = np.ones((1, 1))
    Ws, Wt = np.array([[2.0], [1.0], [0.0]]), np.array([[0.0], [1.0], [2.0]])
    Z = math.e ** 2 + math.e + 1
    p0, p2 = math.e ** 2 / Z, 1 / Z
    for K, (ov_ref, kl_ref) in {1: (0.0, 2 * p0), 2: (0.5, 2 * p0), 3: (1.0, 2 * p0 - 2 * p2)}.items():
        ov, kl, _, _ = O.token_topk_compare(hs, Ws, hs, Wt, [0], K)
        ok &= ov[0] == ov_ref and abs(kl[0] - kl_ref) < 1e-12
    _, H3, tv3, ti3 = O.token_topk(hs, Ws, [0], 2)
    ok &= ti3[0].tolist() == [0, 1] and abs(tv3[0, 0] - (2 - math.log(Z))) < 1e-12
    ok &= abs(H3[0] - (math.log(Z) - (2 * math.e ** 2 + math.e) / Z)) < 1e-12
    return bool(ok)


PINS = [pin_golden_splice, pin_turns_golden, pin_uniform, pin_scipy, pin_torch_ce_and_autograd, pin_kl,
        pin_topk_kl_grad, pin_topk_closed_forms]


def test_real_oracle_passes_every_pin():
    O = load_variant(None)
    assert all(pin(O) for pin in PINS)


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_every_mutant_is_caught(name):
    O = load_variant(name)
    failed = []
    for pin in PINS:
        try:
            ok = pin(O)
        except Exception:  # a crash also counts as caught
            ok = False
        if not ok:
            failed.append(pin.__name__)
    assert failed, f"mutant {name} passed every pin"
