"""Planted mistakes in a copy of the oracle must each fail a pin.

Each case rewrites one line of the oracle's C source into a plausible bug
(a dropped term, a wrong sign or index, a swapped operand), compiles the copy
into a temporary directory, swaps it in for the real library and runs one
pin from test_oracle_pins, expecting that pin to fail. CPU only.
"""
import ctypes
import os
import subprocess

import pytest

from oracle import oracle as orc
import test_oracle_pins as pins
import test_oracle_topk as topk_pins

MUTATIONS = [
    # (name, original text, planted mistake, pin expected to fail, args)
    ("hash_zero_is_set", "int bit = acc > 0.0f;", "int bit = acc >= 0.0f;",
     pins.test_sort_keys_hand_built_2d, ()),
    ("gray_rank_or", "k ^= c;", "k |= c;",
     pins.test_gray_rank_matches_reflected_gray_sequence, ()),
    ("unstable_merge", "if (key[perm[b]] < key[perm[a]])",
     "if (key[perm[b]] <= key[perm[a]])",
     pins.test_stable_argsort_matches_numpy_stable, (1000, 32)),
    ("missing_scale", "z[j] = s * scale;\n        if (z[j] > zmax) zmax = z[j];\n    }\n    int literal",
     "z[j] = s;\n        if (z[j] > zmax) zmax = z[j];\n    }\n    int literal",
     pins.test_single_block_is_dense_softmax_attention, (64, 16, 0)),
    ("dropped_eps_sparse", "o[e] /= (den + floor_);", "o[e] /= den;",
     pins.test_zero_sort_bits_is_block_diagonal_local_attention, (16,)),
    ("next_key_block",
     "key_window(pos[i] / b, nb, N / b, &lo, &hi);",
     "key_window((pos[i] / b + 1) % (N / b), nb, N / b, &lo, &hi);",
     pins.test_query_block_t_attends_exactly_key_block_t, ()),
    ("neighbour_window_too_wide",
     "*lo = blk - nb > 0 ? blk - nb : 0;",
     "*lo = blk - 2 * nb > 0 ? blk - 2 * nb : 0;",
     pins.test_neighbour_blocks_with_zero_sort_bits_are_banded, (16, 1)),
    ("upper_neighbours_dropped",
     "*hi = blk + nb < T - 1 ? blk + nb : T - 1;",
     "*hi = blk < T - 1 ? blk : T - 1;",
     pins.test_neighbour_blocks_with_zero_sort_bits_are_banded, (8, 2)),
    ("dropped_table_average", "den /= (double)L;", "",
     pins.test_race_beta_zero_closed_form, ()),
    ("phi_from_values", "race_phi(K + (size_t)j * d_h, d_h, w_l, gamma",
     "race_phi(V + (size_t)j * d_h, d_h, w_l, gamma",
     pins.test_race_matches_brute_force_kernel_matrix, (1.0,)),
    ("tanh_dropped", "u[bb] = tanh(a);", "u[bb] = a;",
     pins.test_race_feature_softmax_equals_product_identity, ()),
    ("lambda_dropped", "d_s[k] + lam[k] * d_lr[k] + eps", "d_s[k] + d_lr[k] + eps",
     pins.test_multiplier_direct_equals_log_domain_and_in_unit_interval, ()),
    ("gate_swapped", "g_lr[k] * O_lr[(size_t)k * d_h + e]",
     "g_s[k] * O_lr[(size_t)k * d_h + e]",
     pins.test_gates_select_branches_and_ablation_sets_m_to_one, ()),
    # top-k selector
    ("topk_tie_break_reversed",
     "(sc[x] == sc[a] && idx[x] < idx[a])",
     "(sc[x] == sc[a] && idx[x] > idx[a])",
     topk_pins.test_hand_worked_example, ()),
    ("topk_keeps_one_too_many", "keep[a] = beaten < k;",
     "keep[a] = beaten <= k;",
     topk_pins.test_integer_inputs_match_brute_force,
     (64, 4, 8, 2, 8, 2, 0)),
    ("topk_own_block_not_forced", "taken[t] = 1;", "taken[t] = 0;",
     topk_pins.test_integer_inputs_match_brute_force,
     (64, 4, 8, 3, 5, 1, 1)),
    ("topk_block_tie_higher_u",
     "if (!taken[u] && (best < 0 || s[u] > s[best])) best = u;",
     "if (!taken[u] && (best < 0 || s[u] >= s[best])) best = u;",
     topk_pins.test_hand_worked_example, ()),
    ("topk_block_sum_skips_last_row",
     "for (int p = t * b; p < (t + 1) * b; ++p)",
     "for (int p = t * b; p < (t + 1) * b - 1; ++p)",
     topk_pins.test_hand_worked_example, ()),
    ("topk_scores_keys_against_keys",
     "sc[m * b + o] = select_dot(qi, kx + (size_t)j * d_h, d_h);",
     "sc[m * b + o] = select_dot(kx + (size_t)i * d_h, kx + (size_t)j * d_h, d_h);",
     topk_pins.test_integer_inputs_match_brute_force,
     (96, 6, 16, 2, 20, 2, 2)),
]


@pytest.mark.parametrize("name,old,new,pin,args", MUTATIONS,
                         ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(tmp_path, name, old, new, pin, args):
    src = open(orc._SRC).read()
    assert src.count(old) == 1, name
    mutated = tmp_path / "mutant.c"
    mutated.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.check_call(["gcc", "-O1", "-ffp-contract=off", "-fPIC",
                           "-shared", "-std=c11", "-o", str(so),
                           str(mutated), "-lm"])
    saved = orc.lib()
    orc._lib = orc.configure(ctypes.CDLL(os.fspath(so)))
    try:
        with pytest.raises(AssertionError):
            pin(*args)
    finally:
        orc._lib = saved
