"""The oracle's pins catch plausible mistakes: each case below plants one
mistake in a copy of an oracle module (a dropped term, a wrong sign, index,
comparison or operand), runs that module's pin tests against the copy, and
requires at least one of them to fail.  Nothing here touches the GPU path; the
mistakes live only in the in-memory copies.  (A change that cannot alter any
result -- e.g. reordering the tokens of one softmax, which is a sum over a
set -- is not a mistake and is not listed.)
"""
import importlib
import inspect
import sys
import types

import pytest

# (oracle module, pin-test module, name of the oracle module inside the pin-test module, [(old, new), ...])
MUTANTS = {
    # ---- decode attention (plain definition) ----------------------------------
    "attn_scale_dropped": ("attention", "test_oracle_attention", "attention",
                           [("s = scale * (K @ qf[r, j])", "s = (K @ qf[r, j])")]),
    "attn_head_map_interleaved": ("attention", "test_oracle_attention", "attention",
                                  [("for j in range(h * gq, (h + 1) * gq):", "for j in range(h, Hq, num_kv_heads):")]),
    "attn_lse_without_max": ("attention", "test_oracle_attention", "attention",
                             [("lse[r, j] = m + np.log(e.sum())", "lse[r, j] = np.log(e.sum())")]),
    "attn_not_normalised": ("attention", "test_oracle_attention", "attention",
                            [("o[r, j] = (e @ V) / e.sum()", "o[r, j] = (e @ V)")]),
    "attn_keys_for_values": ("attention", "test_oracle_attention", "attention",
                             [("vp = gather_tokens(v_pages,", "vp = gather_tokens(k_pages,")]),
    "attn_suffix_of_wrong_row": ("attention", "test_oracle_attention", "attention",
                                 [("ks = gather_tokens(k_pages, suffix_block_table[r], int(suffix_len[r])",
                                   "ks = gather_tokens(k_pages, suffix_block_table[g], int(suffix_len[g])"),
                                  ("vs = gather_tokens(v_pages, suffix_block_table[r], int(suffix_len[r])",
                                   "vs = gather_tokens(v_pages, suffix_block_table[g], int(suffix_len[g])")]),
    "attn_partial_page_tail": ("attention", "test_oracle_attention", "attention",
                               [("out[t:t + n] = bf16_bits_to_f32(pages[page, kv_head, :n, :])",
                                 "out[t:t + n] = bf16_bits_to_f32(pages[page, kv_head, page_size - n:, :])")]),
    "attn_first_page_only": ("attention", "test_oracle_attention", "attention",
                             [("page = int(table_row[t // page_size])", "page = int(table_row[0])")]),
    "attn_kv_head_of_query_head": ("attention", "test_oracle_attention", "attention",
                                   [("kp = gather_tokens(k_pages, prompt_block_table[g], int(prompt_len[g]), h,",
                                     "kp = gather_tokens(k_pages, prompt_block_table[g], int(prompt_len[g]), "
                                     "(h + 1) % num_kv_heads,")]),
    "attn_default_scale_1_over_d": ("attention", "test_oracle_attention", "attention",
                                    [("scale = 1.0 / np.sqrt(D)", "scale = 1.0 / D")]),
    # ---- sample head ------------------------------------------------------------
    "samp_cutoff_sign": ("sampling", "test_oracle_sampling", "sampling",
                         [("theta32 = np.float32(t * np.log(m))", "theta32 = np.float32(-t * np.log(m))")]),
    "samp_weights_ignore_temperature": ("sampling", "test_oracle_sampling", "sampling",
                                        [("w = np.exp((l[idx] - l.max()) / t)", "w = np.exp(l[idx] - l.max())")]),
    "samp_greedy_last_index": ("sampling", "test_oracle_sampling", "sampling",
                               [("return int(np.argmax(np.asarray(row, dtype=np.float64)))",
                                 "r = np.asarray(row, dtype=np.float64); return int(r.size - 1 - np.argmax(r[::-1]))")]),
    "samp_kept_strict": ("sampling", "test_oracle_sampling", "sampling",
                         [("return row32 >= c", "return row32 > c")]),
    "samp_bf16_shift": ("sampling", "test_oracle_sampling", "sampling",
                        [("<< np.uint32(16)", "<< np.uint32(15)")]),
    "samp_probe_uses_temperature": ("sampling", "test_oracle_sampling", "sampling",
                                    [("if is_probe or float(temperature) == 0.0:", "if float(temperature) == 0.0:")]),
    "samp_cdf_left": ("sampling", "test_oracle_sampling", "sampling",
                      [('k = int(np.searchsorted(cdf, target, side="right"))',
                        'k = int(np.searchsorted(cdf, target, side="left"))')]),
    "samp_inactive_rows_sampled": ("sampling", "test_oracle_sampling", "sampling",
                                   [("        if not active[r]:\n            continue\n", "")]),
    "samp_boundary_band_wide": ("sampling", "test_oracle_sampling", "sampling",
                                [("BOUNDARY_REL = 1e-6", "BOUNDARY_REL = 1e-3")]),
    # ---- Philox4x32-10 ----------------------------------------------------------
    "philox_product_halves_swapped": ("philox", "test_oracle_philox", "philox",
                                      [("return p >> 32, p & MASK32", "return p & MASK32, p >> 32")]),
    "philox_weyl_constant": ("philox", "test_oracle_philox", "philox",
                             [("PHILOX_W1 = 0xBB67AE85", "PHILOX_W1 = 0xBB67AE84")]),
    "philox_high_halves_swapped": ("philox", "test_oracle_philox", "philox",
                                   [("c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0",
                                     "c0, c1, c2, c3 = hi0 ^ c1 ^ k0, lo1, hi1 ^ c3 ^ k1, lo0")]),
    "philox_key_bumped_first": ("philox", "test_oracle_philox", "philox",
                                [("if r > 0:", "if r >= 0:")]),
    "philox_nine_rounds": ("philox", "test_oracle_philox", "philox", [("ROUNDS = 10", "ROUNDS = 9")]),
    "philox_uniform_word1": ("philox", "test_oracle_philox", "philox",
                             [("(seed & MASK32, seed >> 32))[0]", "(seed & MASK32, seed >> 32))[1]"),
                              ("x0 = philox4x32_10_np(ctr, key)[:, 0]", "x0 = philox4x32_10_np(ctr, key)[:, 1]")]),
    "philox_counter_halves_swapped": ("philox", "test_oracle_philox", "philox",
                                      [("(step & MASK32, step >> 32, 0, 0)", "(step >> 32, step & MASK32, 0, 0)"),
                                       ("ctr[:, 0] = step & MASK32\n    ctr[:, 1] = step >> 32",
                                        "ctr[:, 0] = step >> 32\n    ctr[:, 1] = step & MASK32")]),
    # ---- hard gate (compatibility predicate, Alg. 1) -----------------------------
    "gate_no_two_token_minimum": ("gate", "test_oracle_gate", "gate",
                                  [("        if len(pi) >= min_confirm and is_prefix(pi, q):\n",
                                    "        if is_prefix(pi, q):\n")]),
    "gate_prefix_strict": ("gate", "test_oracle_gate", "gate",
                           [("return len(a) <= len(b) and", "return len(a) < len(b) and")]),
    "gate_discard_step_late": ("gate", "test_oracle_gate", "gate",
                               [("        st.decision = NON_REFUSAL\n        st.decisive_step = step\n",
                                 "        st.decision = NON_REFUSAL\n        st.decisive_step = step + 1\n")]),
    "gate_cap_off_by_one": ("gate", "test_oracle_gate", "gate",
                            [("if len(st.q) >= max_len:", "if len(st.q) > max_len:")]),
    "gate_stop_outcome_flipped": ("gate", "test_oracle_gate", "gate",
                                  [("st.decision = REFUSAL if ok else NON_REFUSAL",
                                    "st.decision = NON_REFUSAL if ok else REFUSAL")]),
    "gate_mask_hits_probe": ("gate", "test_oracle_gate", "gate",
                             [("out[g * rows_per_group + 1:(g + 1) * rows_per_group] = 0",
                               "out[g * rows_per_group:(g + 1) * rows_per_group] = 0")]),
    "gate_stop_token_kept_in_q": ("gate", "test_oracle_gate", "gate",
                                  [("    if eos >= 0 and int(y) == eos:\n        st.done = True\n",
                                    "    if eos >= 0 and int(y) == eos:\n        st.q.append(int(y))\n"
                                    "        st.done = True\n")]),
    "gate_confirm_needs_three": ("gate", "test_oracle_gate", "gate",
                                 [("return any(len(pi) >= min_confirm and is_prefix(",
                                   "return any(len(pi) > min_confirm and is_prefix(")]),
    "gate_probe_row_left_on": ("gate", "test_oracle_gate", "gate",
                               [("        if st.done:\n            out[g * rows_per_group] = 0\n", "")]),
    # ---- soft gate (Alg. 2) ---------------------------------------------------------
    "soft_mass_of_whole_top_k": ("soft_gate", "test_oracle_soft_gate", "osg",
                                 [("m = float(sum(p[a] for a in a_ref))", "m = float(sum(p[a] for a in top_k(l, k)))")]),
    "soft_a_star_last": ("soft_gate", "test_oracle_soft_gate", "osg",
                         [("a_star = a_ref[0]", "a_star = a_ref[-1]")]),
    "soft_window_one_longer": ("soft_gate", "test_oracle_soft_gate", "osg",
                               [("in_window = st.steps < c", "in_window = st.steps <= c")]),
    "soft_stop_token_not_a_candidate": ("soft_gate", "test_oracle_soft_gate", "osg",
                                        [("if (eos >= 0 and int(a) == eos) or ogate.compatible",
                                          "if ogate.compatible")]),
    "soft_ties_to_higher_index": ("soft_gate", "test_oracle_soft_gate", "osg",
                                  [("order = np.lexsort((np.arange(l.size), -l))",
                                    "order = np.lexsort((-np.arange(l.size), -l))")]),
    "soft_mass_strict": ("soft_gate", "test_oracle_soft_gate", "osg",
                         [("if a_ref and m >= rho:", "if a_ref and m > rho:")]),
    "soft_empty_candidates_continue": ("soft_gate", "test_oracle_soft_gate", "osg",
                                       [("if a_ref and m >= rho:", "if m >= rho and (a_ref or [None]):"),
                                        ("a_star = a_ref[0]", "a_star = (a_ref or [int(np.argmax(l))])[0]")]),
    "soft_discard_step_late": ("soft_gate", "test_oracle_soft_gate", "osg",
                               [("st.decisive_step = st.steps\n", "st.decisive_step = st.steps + 1\n")]),
    "soft_softmax_unshifted_temperature": ("soft_gate", "test_oracle_soft_gate", "osg",
                                           [("e = np.exp(l - l.max())", "e = np.exp((l - l.max()) / 2.0)")]),
    # ---- residual-stream precheck (App. A) ----------------------------------------
    "pre_bias_sign": ("precheck", "test_oracle_precheck", "precheck",
                      [("return h64 @ w64 + float(b)", "return h64 @ w64 - float(b)")]),
    "pre_weights_reversed": ("precheck", "test_oracle_precheck", "precheck",
                             [("return h64 @ w64 + float(b)", "return h64 @ w64[::-1] + float(b)")]),
    "pre_sigmoid_sign": ("precheck", "test_oracle_precheck", "precheck",
                         [("out[pos] = 1.0 / (1.0 + np.exp(-z[pos]))", "out[pos] = 1.0 / (1.0 + np.exp(z[pos]))")]),
    "pre_skip_strict": ("precheck", "test_oracle_precheck", "precheck",
                        [("return z, p, p <= float(theta)", "return z, p, p < float(theta)")]),
    "pre_started_probes_skipped": ("precheck", "test_oracle_precheck", "precheck",
                                   [("st.steps == 0 and ", "")]),
    "pre_masks_a_sample_row": ("precheck", "test_oracle_precheck", "precheck",
                               [("out[g * rows_per_group] = 0", "out[g * rows_per_group + 1] = 0")]),
}


def _mutant_module(name: str, edits):
    """A fresh copy of ``oracle.<name>`` with the edits applied to its source."""
    real = importlib.import_module(f"oracle.{name}")
    src = inspect.getsource(real)
    for old, new in edits:
        assert src.count(old) >= 1, (name, old)
        src = src.replace(old, new)
    mod = types.ModuleType(f"oracle.{name}")
    mod.__dict__.update({"__package__": "oracle", "__file__": real.__file__})
    exec(compile(src, f"<mutant of oracle/{name}.py>", "exec"), mod.__dict__)
    return mod


def _pin_tests(test_mod):
    return [getattr(test_mod, n) for n in sorted(dir(test_mod))
            if n.startswith("test_") and callable(getattr(test_mod, n))]


@pytest.mark.parametrize("case", sorted(MUTANTS))
def test_pins_catch_the_planted_mistake(case):
    oname, tname, attr, edits = MUTANTS[case]
    tests_dir = __import__("os").path.dirname(__file__)
    if tests_dir not in sys.path:
        sys.path.insert(0, tests_dir)
    test_mod = importlib.import_module(tname)
    real = getattr(test_mod, attr)
    mutant = _mutant_module(oname, edits)
    failed = []
    setattr(test_mod, attr, mutant)
    try:
        for fn in _pin_tests(test_mod):
            try:
                fn()
            except Exception as e:  # a failed assertion, or the mistake breaking the computation
                failed.append((fn.__name__, type(e).__name__))
                break
    finally:
        setattr(test_mod, attr, real)
    assert failed, f"no pin of {tname} catches {case}"


def test_unmutated_copies_pass_every_pin():
    """The copying itself changes nothing: an unedited copy passes all pins."""
    tests_dir = __import__("os").path.dirname(__file__)
    if tests_dir not in sys.path:
        sys.path.insert(0, tests_dir)
    for oname, tname, attr in {(v[0], v[1], v[2]) for v in MUTANTS.values()}:
        test_mod = importlib.import_module(tname)
        real = getattr(test_mod, attr)
        setattr(test_mod, attr, _mutant_module(oname, []))
        try:
            for fn in _pin_tests(test_mod):
                fn()
        finally:
            setattr(test_mod, attr, real)
