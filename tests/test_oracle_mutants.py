"""Planted mistakes in the oracle, each of which must fail one of its pins (CPU only).

Every case below changes one spot of `oracle/ptd_oracle.py` the way a plausible slip
would (a dropped term, an off-by-one, a wrong index or tie order), loads the changed source
as a separate module and runs the pins of `tests/test_oracle_pins.py` that cover that
function against it.  The oracle itself is never modified; the mutated copy exists only in
this process.  A mistake that no pin catches fails this test.
"""
import importlib.util
import os
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_SRC = os.path.join(ROOT, "oracle", "ptd_oracle.py")

ATTN = ["test_attention_worked_example", "test_star_tree_sees_context_root_self", "test_chain_tree_is_causal_chunk",
        "test_single_node_is_plain_decode", "test_gqa_matches_repeated_kv_heads",
        "test_identical_keys_give_mean_of_visible_values"]
TOPK = ["test_topk_worked_example", "test_topk_matches_lexsort_with_ties", "test_topk_brute_force_rank"]
VERIFY = ["test_verify_worked_examples", "test_verify_brute_force_exhaustive"]
COMPACT = ["test_compact_worked_example", "test_compact_matches_gather_and_keeps_prefix"]
SAMPLING = ["test_sampling_worked_examples", "test_sampling_one_hot_reduces_to_greedy", "test_sampling_invariants_on_random_trees",
            "test_sampling_leaf_root_bonus_is_P_and_temperature", "test_sampling_star_tree_emits_P"]
DRAFT = ["test_draft_update_worked_examples", "test_draft_update_identity_and_sliding_window",
         "test_draft_update_invariants", "test_draft_update_matches_trie_formulation"]
POOL = ["test_pool_worked_example", "test_pool_idempotent_and_chain", "test_pool_matches_path_set_formulation"]
ROPE = ["test_tree_positions_closed_forms", "test_rope_defining_properties"]

# (name, original text, planted text, pins that cover it)
MUTANTS = [
    # tree-masked attention (Sec. 3.1, 3.2)
    ("last-committed-slot-hidden", "vis[:, :ctx_len] = True", "vis[:, :max(ctx_len - 1, 0)] = True", ATTN),
    ("strict-ancestors-only", "            vis[i, ctx_len + a] = True", "            vis[i, ctx_len + a] = a != i or i == 0",
     ATTN),
    ("gqa-head-modulo", "        kv = h // G", "        kv = h % Hkv", ATTN),
    ("scale-one-over-d", "scale = 1.0 / math.sqrt(D)", "scale = 1.0 / D", ATTN),
    ("mask-dropped", "s = np.where(vis, s, -np.inf)", "s = np.where(vis, s, s)", ATTN),
    # top-k
    ("ties-higher-index-first", 'order = np.argsort(-x, kind="stable")[:k]',
     'order = (x.shape[0] - 1 - np.argsort(-x[::-1], kind="stable"))[:k]', TOPK),
    ("ascending", 'order = np.argsort(-x, kind="stable")[:k]', 'order = np.argsort(x, kind="stable")[:k]', TOPK),
    # greedy verification (Sec. 3.2)
    ("ties-to-largest-sequence", "path < best", "path > best", VERIFY),
    ("accept-len-without-root", "return best, len(best), int(target[best[-1]])",
     "return best, len(best) - 1, int(target[best[-1]])", VERIFY),
    ("bonus-of-the-parent", "return best, len(best), int(target[best[-1]])",
     "return best, len(best), int(target[best[-2] if len(best) > 1 else best[-1]])", VERIFY),
    ("edge-tests-child-target", "int(tokens[c]) == int(target[n])", "int(tokens[c]) == int(target[c])", VERIFY),
    # KV compaction (Alg. 1 step 6)
    ("new-ctx-off-by-one", "return new, ctx_len + len(path)", "return new, ctx_len + len(path) - 1", COMPACT),
    ("source-slot-without-prefix", "new[ctx_len + j] = snap[ctx_len + int(n)]", "new[ctx_len + j] = snap[int(n)]",
     COMPACT),
    # sampling verification (Alg. 2)
    ("no-renormalisation", "p_hat = P[t] / S if S > 0.0 else 0.0", "p_hat = P[t]", SAMPLING),
    ("rejected-token-kept", "            S -= P[t]\n            P[t] = 0.0\n", "            S -= P[t]\n", SAMPLING),
    ("bonus-from-full-P", "    target = float(u_bonus) * S\n    cdf = np.cumsum(P)",
     "    P = softmax_row(logits[v], temperature)\n    S = 1.0\n    target = float(u_bonus) * S\n    cdf = np.cumsum(P)",
     SAMPLING),
    ("last-child-never-tried", "        for n in sigma[v]:\n            t = int(tokens[n])",
     "        for n in sigma[v][:-1] if len(sigma[v]) > 1 else sigma[v]:\n            t = int(tokens[n])", SAMPLING),
    # draft tree update (Sec. 3.1 expansion, width and depth control)
    ("no-reuse-of-existing-child", "            if any(tok[i] == d for i in kids):\n                continue",
     "            pass", DRAFT),
    ("width-off-by-one", "if len(kids) >= width or", "if len(kids) > width or", DRAFT),
    ("latest-child-kept", "first_child = min(i for i in range(n) if par[i] == s)",
     "first_child = max(i for i in range(n) if par[i] == s)", DRAFT),
    ("depth-in-edges", "        if sub_depth <= max_depth:\n            continue",
     "        if sub_depth - 1 <= max_depth:\n            continue", DRAFT),
    ("new-nodes-expanded-too", "    for v in range(T):\n        for r in range(expand):",
     "    v = 0\n    while v < len(par):\n        v += 1\n        if v > len(par):\n            break\n"
     "        for r in range(expand):", DRAFT),
    ("new-seed-keeps-parent", "        new_par.append(-1 if (p == -1 or not keep[p]) else new_index[p])",
     "        new_par.append(-1 if p == -1 else (new_index[p] if keep[p] else p))", DRAFT),
    # candidate pool (Sec. 3.1 merging; Alg. 1 steps 1 and 4)
    ("new-child-without-subtree",
     "                pnode.children.append(match)\n            self._merge(match, parents, tokens, kids, c)",
     "                pnode.children.append(match)\n                continue\n"
     "            self._merge(match, parents, tokens, kids, c)", POOL),
    ("seeds-only", "        for v in range(len(parents)):\n            tok = int(tokens[v])",
     "        for v in [i for i in range(len(parents)) if parents[i] == -1]:\n            tok = int(tokens[v])", POOL),
    ("latest-children-retrieved", "                for c in node.children[:width]:",
     "                for c in node.children[::-1][:width]:", POOL),
    ("retrieval-depth-off-by-one", "        depth = 1\n        while frontier", "        depth = 0\n        while frontier",
     POOL),
    ("node-budget-off-by-one", "                    if len(tokens) >= max_nodes:\n                        break",
     "                    if len(tokens) > max_nodes:\n                        break", POOL),
    # tree positions and the rotary encoding
    ("position-without-minus-one", "[ctx_len + len(a) - 1 for a", "[ctx_len + len(a) for a", ROPE),
    ("interleaved-pairs",
     "    a, b = x[..., :half], x[..., half:]\n    return np.concatenate([a * c - b * s, a * s + b * c], axis=-1)",
     "    a, b = x[..., 0::2], x[..., 1::2]\n    out = np.empty_like(x)\n    out[..., 0::2] = a * c - b * s\n"
     "    out[..., 1::2] = a * s + b * c\n    return out", ROPE),
    ("negative-angle", "[a * c - b * s, a * s + b * c]", "[a * c + b * s, -a * s + b * c]", ROPE),
    ("frequency-exponent", "inv_freq = base ** (-2.0 * np.arange(half", "inv_freq = base ** (-1.0 * np.arange(half",
     ROPE),
]


@pytest.fixture(scope="module")
def pins():
    spec = importlib.util.spec_from_file_location("oracle_pins_under_mutation",
                                                  os.path.join(ROOT, "tests", "test_oracle_pins.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _mutant(original: str, planted: str) -> types.ModuleType:
    src = open(ORACLE_SRC).read()
    assert src.count(original) == 1, "the planted spot must occur exactly once"
    mod = types.ModuleType("oracle_mutant")
    mod.__file__ = ORACLE_SRC
    exec(compile(src.replace(original, planted), ORACLE_SRC + " (mutant)", "exec"), mod.__dict__)
    return mod


def _calls(fn):
    """Keyword arguments of every parametrised case of a pin (one case if none)."""
    combos = [{}]
    for m in getattr(fn, "pytestmark", []):
        if m.name != "parametrize":
            continue
        names = [n.strip() for n in m.args[0].split(",")]
        combos = [{**c, **dict(zip(names, v if len(names) > 1 else (v,)))} for c in combos for v in m.args[1]]
    return combos


def _first_failing_pin(pins_mod, oracle_mod, names):
    original = pins_mod.oracle
    pins_mod.oracle = oracle_mod
    try:
        for name in names:
            fn = getattr(pins_mod, name)
            for kw in _calls(fn):
                try:
                    fn(**kw)
                except Exception:   # an assertion, or the mistake breaking the function outright
                    return name, kw
        return None
    finally:
        pins_mod.oracle = original


def test_every_pin_named_here_exists(pins):
    for _, _, _, names in MUTANTS:
        for n in names:
            assert callable(getattr(pins, n, None)), n


def test_pins_pass_on_the_oracle_itself(pins):
    """Every pin used below passes on the unmodified source loaded the same way, so a pin
    that fails on a mutant fails because of the planted mistake."""
    src = open(ORACLE_SRC).read()
    mod = types.ModuleType("oracle_unmodified")
    exec(compile(src, ORACLE_SRC, "exec"), mod.__dict__)
    names = []
    for _, _, _, ns in MUTANTS:
        names += [n for n in ns if n not in names]
    assert _first_failing_pin(pins, mod, names) is None


@pytest.mark.parametrize("name,original,planted,names", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(pins, name, original, planted, names):
    caught = _first_failing_pin(pins, _mutant(original, planted), names)
    assert caught is not None, f"no pin catches the planted mistake '{name}'"
