"""Mutation checks of the C oracle (CPU only): each test compiles a copy of oracle.c with
one plausible mistake planted (a dropped term, a wrong sign or comparison, a truncated
walk) and asserts that at least one of the oracle's pins then fails.  The unmutated
source passes them all (the pin files themselves)."""
import os

import pytest

import test_oracle_eff_pins as EP
import test_oracle_pins as CP
import test_oracle_tree_pins as TP

HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(os.path.dirname(HERE), "oracle", "oracle.c")

# name: (the exact source text, its mutated replacement)
MUTANTS = {
    "ancestor pairs compared": (
        "if (is_strict_ancestor(&G, i, j) || is_strict_ancestor(&G, j, i)) continue;",
        "if (0) continue;"),
    "strict threshold": (
        "if (cosine(&G, d, i, j) >= p->kappa)",
        "if (cosine(&G, d, i, j) > p->kappa)"),
    "pooling without w": (
        "S[i] = den > 0.0 ? (c_own[i] + p->w * oc) / den : 0.0;",
        "S[i] = den > 0.0 ? (c_own[i] + oc) / den : 0.0;"),
    "eta not clamped at 0": (
        "eta[i] = sim > 0.0 ? sim : 0.0;",
        "eta[i] = sim;"),
    "step reward sign": (
        "r[i] = (S[i] - S[u]) * (1.0 - eta[i]);",
        "r[i] = (S[u] - S[i]) * (1.0 - eta[i]);"),
    "step reward without the eta gate": (
        "r[i] = (S[i] - S[u]) * (1.0 - eta[i]);",
        "r[i] = (S[i] - S[u]);"),
    "one-edge groups standardised": (
        "if (K <= 1) continue;",
        "if (K <= 0) continue;"),
    "standardisation without eps": (
        "a_cor[tmp[k]] = (xs[k] - mean) / (sd + p->std_eps);",
        "a_cor[tmp[k]] = sd > 0.0 ? (xs[k] - mean) / sd : 0.0;"),
    "shallowest common ancestor": (
        "if (cnt[i] == Q && (aQ < 0 || G.depth[i] > G.depth[aQ])) aQ = i;",
        "if (cnt[i] == Q && (aQ < 0 || G.depth[i] < G.depth[aQ])) aQ = i;"),
    "efficiency sign": (
        "const double A = sbar * (xs[m - q0] - mean) / (sd + p->std_eps);",
        "const double A = sbar * (mean - xs[m - q0]) / (sd + p->std_eps);"),
    "route truncated to one edge": (
        "for (int x = v; x != aQ; x = G.parent[x]) {",
        "for (int x = v; x != aQ; x = aQ) {"),
    "graph reachability not propagated": (
        "if (G.label[i] == L && u > 0 && !reach[G.label[u]]) {",
        "if (0) {"),
    "tree reachability counts every step": (
        "if (c_own[i] > 0.0) good_tree += len;",
        "if (c_own[i] >= 0.0) good_tree += len;"),
    "same-depth rule ignored": (
        "if (p->merge_rule == 1 && G.depth[i] != G.depth[j]) continue;",
        "if (0) continue;"),
    "prompt embedding ignored": (
        "if (u > 0 || G.has_root_emb) sim = cosine(&G, d, u, i);",
        "if (u > 0) sim = cosine(&G, d, u, i);"),
    "root statistics not gathered": (
        "      c_own[G.parent[i]] += c_own[i];\n      t_own[G.parent[i]] += t_own[i];",
        "      if (G.parent[i] > 0) c_own[G.parent[i]] += c_own[i];\n"
        "      if (G.parent[i] > 0) t_own[G.parent[i]] += t_own[i];"),
    "terminal counts not propagated": (
        "t_own[G.parent[i]] += t_own[i];",
        "t_own[G.parent[i]] += 1.0;"),
    "every terminal correct": (
        "c_own[i] += (double)b->reward[G.rollout[i]];",
        "c_own[i] += 1.0;"),
    "pooling counts the state among the others": (
        "if (q == i) continue;",
        "if (0) continue;"),
    "correctness group of one member's children": (
        "for (int m = G.mem_off[L]; m < G.mem_off[L + 1]; ++m) {\n      const int q = G.mem_list[m];\n"
        "      for (int c = G.child_off[q]",
        "for (int m = G.mem_off[L]; m < G.mem_off[L] + 1; ++m) {\n      const int q = G.mem_list[m];\n"
        "      for (int c = G.child_off[q]"),
    "population std": (
        "return sqrt(s / (n - ddof));",
        "return sqrt(s / n);"),
    "class score summed, not averaged": (
        "sbar /= Q;",
        "sbar /= 1;"),
    "route contributions overwritten": (
        "e_eff[x] += A;",
        "e_eff[x] = A;"),
    "lambda ignored on tokens": (
        "      const double dual = a_cor[i] + p->lambda_eff * e_eff[i];\n      for (int k = 0;",
        "      const double dual = a_cor[i] + e_eff[i];\n      for (int k = 0;"),
    "lambda ignored on edges": (
        "    const double dual = a_cor[i] + p->lambda_eff * e_eff[i];\n    if (o->class_id)",
        "    const double dual = a_cor[i] + e_eff[i];\n    if (o->class_id)"),
    "graph reachability seeded by every terminal": (
        "if (G.terminal[i] && b->reward[G.rollout[i]] && !reach[G.label[i]]) {",
        "if (G.terminal[i] && !reach[G.label[i]]) {"),
    "cosine without the norms": (
        "return dot / (G->nrm[i] * G->nrm[j]);",
        "return dot;"),
    "leaves matched to rollouts in reverse": (
        "G.rollout[i] = G.terminal[i] ? r0 + k++ : -1;",
        "G.rollout[i] = G.terminal[i] ? r1 - 1 - k++ : -1;"),
    "mask only on the member's own edge": (
        "        emask[x] = 1;",
        "        emask[v] = 1;"),
}


def _pins(oracle_mod):
    return [
        lambda: CP.test_micro_worked_example(oracle_mod),
        lambda: CP.test_threshold_is_inclusive(oracle_mod),
        lambda: CP.test_classes_are_library_connected_components(oracle_mod, "tiny", 8, 0),
        lambda: CP.test_classes_are_library_connected_components(oracle_mod, "tiny", 8, 1),
        lambda: CP.test_micro_root_embedding_variant(oracle_mod),
        lambda: TP.test_tree_root_embedding_variant(oracle_mod),
        lambda: CP.test_group_invariants(oracle_mod, "tiny", 8),
        lambda: CP.test_routes_by_path_enumeration(oracle_mod),
        lambda: CP.test_two_edge_group_closed_form(oracle_mod),
        lambda: TP.test_tree_worked_example(oracle_mod),
        lambda: TP.test_tree_aQ_and_routes_by_path_enumeration(oracle_mod),
        lambda: TP.test_tree_eta_is_clamped_at_zero(oracle_mod),
        lambda: EP.test_eff_worked_example(oracle_mod),
        lambda: EP.test_eff_graph_by_library_reachability(oracle_mod, "tree"),
    ]


def _fails(pins):
    for pin in pins:
        try:
            pin()
        except AssertionError:
            return True
    return False


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_c_oracle_pins_catch_mutant(oracle_mod, tmp_path, name):
    old, new = MUTANTS[name]
    src = open(SOURCE).read()
    assert src.count(old) == 1, f"mutation site not found once: {old}"
    so = oracle_mod.compile_variant(src.replace(old, new), str(tmp_path))
    with oracle_mod.library(so):
        assert _fails(_pins(oracle_mod)), f"no pin catches the mutant: {name}"


def test_unmutated_c_oracle_passes_the_same_pins(oracle_mod):
    assert not _fails(_pins(oracle_mod))
