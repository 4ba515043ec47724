"""The pins catch plausible oracle mistakes.

Each mutant below is the oracle source with one plausible slip (a dropped
term, a wrong sign or index, a transposed operand, a flipped tie-break). Each
is compiled on the CPU and must fail at least one pin in pins.ALL_CHECKS.
"""

import os
import subprocess
import sys

import pytest

import oracle
from pins import ALL_CHECKS

SRC = os.path.join(os.path.dirname(oracle.__file__), "smetric_oracle.c")

MUTANTS = {
    "mix64_shift": ("z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;",
                    "z = (z ^ (z >> 31)) * 0xBF58476D1CE4E5B9ULL;"),
    "word_halves_swapped": ("return lo | (hi << 32);", "return hi | (lo << 32);"),
    "digest_start_drops_block_size": ("uint64_t d = oracle_mix64(seed ^ (uint64_t)B);",
                                      "uint64_t d = oracle_mix64(seed);"),
    "chain_drops_previous": ("h = oracle_mix64((h + ORACLE_GAMMA) ^ d);",
                             "h = oracle_mix64(ORACLE_GAMMA ^ d);"),
    "chain_xor_for_add": ("h = oracle_mix64((h + ORACLE_GAMMA) ^ d);",
                          "h = oracle_mix64((h ^ ORACLE_GAMMA) ^ d);"),
    "no_sentinel_remap": ("if (h < 2) h |= 2;", ""),
    "digest_fold_reversed": ("for (int32_t k = 0; k < B / 2; ++k) d = oracle_mix64(",
                             "for (int32_t k = B / 2 - 1; k >= 0; --k) d = oracle_mix64("),
    "digest_skips_word0": ("for (int32_t k = 0; k < B / 2; ++k) d = oracle_mix64(",
                           "for (int32_t k = 1; k < B / 2; ++k) d = oracle_mix64("),
    "digest_last_word_only": ("d = oracle_mix64(d ^ oracle_word(tokens, b * B + 2 * k));",
                              "d = oracle_mix64(oracle_mix64(seed ^ (uint64_t)B) ^ oracle_word(tokens, b * B + 2 * k));"),
    "word_index_off_by_one": ("oracle_word(tokens, b * B + 2 * k)",
                              "oracle_word(tokens, b * B + k)"),
    "session_key_index": ("session_key[r] = h[(n < S ? n : S) - 1];",
                          "session_key[r] = h[(n - 1 < S ? n - 1 : S)];"),
    "walk_counts_missing_block": ("if (!held) { c[i] = k; running--; }",
                                  "if (!held) { c[i] = k + 1; running--; }"),
    "global_walk_ignored": ("if (!held) { *g = k; running--; }",
                            "if (!held || 1) { *g = k; running--; }"),
    "miss_uses_local_hit": ("int64_t miss = L - (int64_t)B * gi;",
                            "int64_t miss = L - (int64_t)B * c[i];"),
    "fetch_sign": ("int64_t fetch = (int64_t)B * (gi - c[i]);",
                   "int64_t fetch = (int64_t)B * (c[i] - gi);"),
    "global_weight_dropped": ("+ w_glob * fetch;", ";"),
    "tie_to_highest": ("if (best < 0 || cost < best_cost)", "if (best < 0 || cost <= best_cost)"),
    "global_hit_reports_g": ("global_hit[r] = (int32_t)((int64_t)B * (gb - c[best]));",
                             "global_hit[r] = (int32_t)((int64_t)B * gb);"),
    "tail_block_hashed": ("int64_t n = L / B;\n  uint64_t h = oracle_mix64",
                          "int64_t n = (L + B - 1) / B;\n  uint64_t h = oracle_mix64"),
    "policy_drops_half_term": ("c_att * nn * (2 * L - nn)", "c_att * nn * (2 * L)"),
    "policy_drops_queue": ("est2[i] = 2 * queued[i] + ", "est2[i] = "),
    "policy_prev_highest_id": ("if (c[i] > c[prev]) prev = i;", "if (c[i] >= c[prev]) prev = i;"),
    "policy_cached_inclusive": ("hit_den > hit_num * est_hit[r];", "hit_den >= hit_num * est_hit[r];"),
    "policy_meets_strict": ("const int meets_prev = est2[prev] <= budget2;",
                            "const int meets_prev = est2[prev] < budget2;"),
    "policy_no_last_resort": ("(meets_prev || !any_meets)", "meets_prev"),
    "policy_ignores_turn": ("turn[r] != 0 && cached", "cached"),
    "policy_no_rotation": ("(int32_t)(((int64_t)rr_base + r) % N)", "0"),
    "policy_rotation_takes_last": ("if (est2[i] < est2[to]) to = i;", "if (est2[i] <= est2[to]) to = i;"),
    "coloc_no_tpot_filter": ("cand[i] = cost2[i] <= 2 * tpot_budget[i];", "cand[i] = 1;"),
    "coloc_filter_uses_load": ("cand[i] = cost2[i] <= 2 * tpot_budget[i];",
                               "cand[i] = est2[i] <= 2 * tpot_budget[i];"),
    "coloc_empty_filter_kept": ("for (int32_t i = 0; i < N; ++i) cand[i] = 1;", ";"),
    "coloc_last_resort": ("meets_prev && cand[prev];", "(meets_prev || 1) && cand[prev];"),
    "coloc_prev_not_checked": ("meets_prev && cand[prev];", "meets_prev;"),
    "coloc_sum_not_product": ("(unsigned __int128)(uint64_t)est2[i] * (uint64_t)num_requests[i];",
                              "(unsigned __int128)((uint64_t)est2[i] + (uint64_t)num_requests[i]);"),
    "link_earliest_parent": ("for (int32_t p = r - 1; p >= 0; --p) {", "for (int32_t p = 0; p < r; ++p) {"),
    "link_turn_ignored": ("|| (int64_t)turns[p] != (int64_t)turns[r] - 1) continue;", ") continue;"),
    "link_user_ignored": ("if (users[p] != users[r] || ", "if ("),
    "link_longer_parent": ("if (np > nr) continue;", ";"),
    "link_session_is_parent": ("session[r] = parent[r] < 0 ? r : session[parent[r]];",
                               "session[r] = parent[r] < 0 ? r : parent[r];"),
    "bailian_no_normalisation": ("(unsigned __int128)(uint64_t)((lam_den - lam_num) * batch[i]) * Lr : 0;",
                                 "(unsigned __int128)(uint64_t)((lam_den - lam_num) * batch[i]) * Lr * Lm : 0;"),
    "bailian_weights_swapped": ("(unsigned __int128)(uint64_t)((lam_den - lam_num) * batch[i]) * Lr : 0;",
                                "(unsigned __int128)(uint64_t)(lam_num * batch[i]) * Lr : 0;"),
    "bailian_hit_for_miss": ("(unsigned __int128)(uint64_t)lam_num * (L > 0 ? miss : 1) * Lm;",
                             "(unsigned __int128)(uint64_t)lam_num * (L > 0 ? (uint64_t)L - miss : 1) * Lm;"),
    "lmetric_sum": ("(unsigned __int128)(uint64_t)(queued[i] + L - (int64_t)B * c[i]) * (uint64_t)batch[i];",
                    "(unsigned __int128)(uint64_t)(queued[i] + L - (int64_t)B * c[i]) + (uint64_t)batch[i];"),
    "lmetric_drops_queue": ("(uint64_t)(queued[i] + L - (int64_t)B * c[i])", "(uint64_t)(L - (int64_t)B * c[i])"),
    "baseline_tie_to_highest": ("if (best < 0 || f < best_f) { best = i; best_f = f; }",
                                "if (best < 0 || f <= best_f) { best = i; best_f = f; }"),
    "sequential_no_update": ("q[best] += L - (int64_t)B * c[best];", ";"),
    "sequential_update_global": ("q[best] += L - (int64_t)B * c[best];", "q[best] += L - (int64_t)B * g;"),
    "reuse_latest_producer": ("for (int32_t p = 0; p < r && producer < 0; ++p)",
                              "for (int32_t p = r - 1; p >= 0 && producer < 0; --p)"),
    "reuse_system_off_by_one": ("if (b < sys_blocks[r]) sys[r]++;", "if (b <= sys_blocks[r]) sys[r]++;"),
    "reuse_self_hit": ("for (int32_t p = 0; p < r && producer < 0; ++p)",
                       "for (int32_t p = 0; p <= r && producer < 0; ++p)"),
    "reuse_system_by_session": ("if (b < sys_blocks[r]) sys[r]++;", "if (b < sys_blocks[r] && sessions[producer] != sessions[r]) sys[r]++;"),
    "imbalance_window_end_inclusive": ("const int64_t b = end[r] < hi ? end[r] : hi;",
                                       "const int64_t b = end[r] < hi + 1 ? end[r] : hi + 1;"),
    "imbalance_counts_request_length": ("if (b > a) s += b - a;", "if (b > a) s += end[r] - start[r];"),
    "imbalance_tie_to_highest": ("if (s > out_max[w]) {", "if (s >= out_max[w]) {"),
    "imbalance_window_origin": ("const int64_t lo = (int64_t)w * T, hi = lo + T;",
                                "const int64_t lo = (int64_t)w * T + 1, hi = lo + T;"),
    "coloc_product_64_bit": ("(unsigned __int128)(uint64_t)est2[i] * (uint64_t)num_requests[i];",
                             "(unsigned __int128)((uint64_t)est2[i] * (uint64_t)num_requests[i]);"),
}


def _build_mutant(name, tmp_path):
    src = open(SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) >= 1, name
    path_c = tmp_path / f"{name}.c"
    path_so = tmp_path / f"{name}.so"
    path_c.write_text(src.replace(old, new, 1))
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-w", "-fopenmp", "-shared", "-fPIC",
                           str(path_c), "-o", str(path_so)])
    return oracle.load_library(str(path_so))


_RUNNER = """
import sys
sys.path[:0] = [{root!r}, {tests!r}]
import oracle
from pins import ALL_CHECKS
L = oracle.load_library({so!r})
failed = []
for check in ALL_CHECKS:
    try:
        check(L)
    except Exception as e:
        failed.append(check.__name__)
print("FAILED_CHECKS", ",".join(failed))
"""


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, tmp_path):
    src = open(SRC).read()
    old, new = MUTANTS[name]
    assert src.count(old) >= 1, name
    path_c = tmp_path / f"{name}.c"
    path_so = tmp_path / f"{name}.so"
    path_c.write_text(src.replace(old, new, 1))
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-w", "-fopenmp", "-shared", "-fPIC",
                           str(path_c), "-o", str(path_so)])
    here = os.path.dirname(os.path.abspath(__file__))
    code = _RUNNER.format(root=os.path.dirname(here), tests=here, so=str(path_so))
    p = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, timeout=300)
    if p.returncode != 0:
        return  # the mutant crashed (e.g. read past its buffer): caught
    line = [x for x in p.stdout.splitlines() if x.startswith("FAILED_CHECKS")][-1]
    failed = line.split(" ", 1)[1].strip() if " " in line else ""
    assert failed, f"mutant {name} passed every pin"


# The LRU oracle (plain Python): each mutant restates the recency rule with
# one plausible slip and must fail pins.check_lru_recency.
def _lru_mutant(stamp_of=None, keep_first_touch=False, evict_largest=False):
    class Mutant(oracle.OracleLRU):
        def commit(self, n_blocks, instance, hashes, also_global):
            import numpy as np
            hashes = [int(x) for x in np.asarray(hashes, dtype=np.uint64)]
            pos = 0
            for r, (nb, i) in enumerate(zip(np.asarray(n_blocks).tolist(), np.asarray(instance).tolist())):
                keys = hashes[pos:pos + nb]
                pos += nb
                if i < 0:
                    continue
                for t in ([i, -1] if also_global else [i]):
                    if self.caps[t] <= 0:
                        continue
                    tier = self.stamp[t]
                    for b, key in enumerate(keys):
                        st = stamp_of(self.k, r, b) if stamp_of else (self.k, r, -b)
                        if key not in tier or (not keep_first_touch and tier[key] < st):
                            tier[key] = st
            self.k += 1
            ev_k, ev_t = [], []
            for t, tier in self.stamp.items():
                over = len(tier) - self.caps[t]
                if self.caps[t] > 0 and over > 0:
                    order = sorted(tier.items(), key=lambda kv: kv[1], reverse=evict_largest)
                    for key, _ in order[:over]:
                        del tier[key]
                        ev_k.append(key)
                        ev_t.append(t)
            return np.array(ev_k, dtype=np.uint64), np.array(ev_t, dtype=np.int32)
    return Mutant


LRU_MUTANTS = {
    "deepest_block_most_recent": _lru_mutant(stamp_of=lambda k, r, b: (k, r, b)),
    "earlier_request_more_recent": _lru_mutant(stamp_of=lambda k, r, b: (k, -r, -b)),
    "batch_order_ignored": _lru_mutant(stamp_of=lambda k, r, b: (r, -b)),
    "first_touch_kept": _lru_mutant(keep_first_touch=True),
    "most_recent_evicted": _lru_mutant(evict_largest=True),
}


@pytest.mark.parametrize("name", sorted(LRU_MUTANTS))
def test_lru_mutant_is_caught(name, monkeypatch):
    from pins import check_lru_recency
    monkeypatch.setattr(oracle, "OracleLRU", LRU_MUTANTS[name])
    with pytest.raises(AssertionError):
        check_lru_recency(None)
