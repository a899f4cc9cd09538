"""Plant plausible mistakes in copies of the oracle; each must fail a pin.

Every mutant is the oracle's C source with one textual change, compiled into a
temporary library. A mutant that passes every pin would mean the pins cannot
tell that mistake from the definition.
"""
import os

import pytest

import oracle
import oracle_pins as pins

MUTANTS = {
    # mask: verify pass loses the diagonal (a token not seeing itself)
    "verify_excludes_self": ("return j <= i;", "return j < i;"),
    # mask: the diffusion pass made causal
    "diffusion_causal": ("if (mode == 0) return 1;", "if (mode == 0) return j <= i;"),
    # mask: block slots indexed from the wrong origin
    "block_offset": ("long j = t - L;", "long j = t - L + 1;"),
    # mask: verify pass made anti-causal (row i sees later block slots)
    "verify_anticausal": ("return j <= i;", "return j >= i;"),
    # GQA head mapping interleaved instead of grouped
    "gqa_interleaved": ("const int g = h / G;", "const int g = h % Hkv;"),
    # softmax scale dropped
    "scale_dropped": ("s[t] = scale * dot;", "s[t] = dot;"),
    # lse without the max shift
    "lse_missing_max": ("*lse = m + log(l);", "*lse = log(l);"),
    # page slot from the wrong index (K side only)
    "slot_index": ("const uint16_t *krow = k + (((long)page * Hkv + g) * P + (t % P)) * (long)D;",
                   "const uint16_t *krow = k + (((long)page * Hkv + g) * P + (t / P) % P) * (long)D;"),
    # query layout transposed ([B, Hq, bl, D] instead of [B, bl, Hq, D])
    "q_layout": ("q + (((long)b * bl + i) * Hq + h) * (long)D;", "q + (((long)b * Hq + h) * bl + i) * (long)D;"),
    # combine forgets the partial weights
    "combine_unweighted": ("orow[d] += c * op[d];", "orow[d] += op[d];"),
    # combine: normaliser dropped
    "combine_no_norm": ("for (int d = 0; d < D; ++d) orow[d] /= csum;", ""),
    # accept counts the bonus token
    "accept_plus_bonus": ("accepted[b] = j;", "accepted[b] = j < n ? j + 1 : j;"),
    # accept counts all matches instead of the matching prefix
    "accept_counts_matches": ("while (j < n && draft[(long)b * n + j] == verify[(long)b * n + j]) ++j;",
                              "for (int t = 0; t < n; ++t) j += draft[(long)b * n + t] == verify[(long)b * n + t];"),
    # unmask tie-break reversed
    "unmask_tie_high_index": ("return a < b;", "return a > b;"),
    # unmask: -inf treated as eligible
    "unmask_neginf_eligible": ("if (!isnan(c[i]) && !(isinf(c[i]) && c[i] < 0)) idx[m++] = i;",
                               "if (!isnan(c[i])) idx[m++] = i;"),
    # threshold: "exceeds" taken as >=
    "threshold_ge": ("if (eligible(c[i]) && c[i] > threshold) pos[count++] = i;",
                     "if (eligible(c[i]) && c[i] >= threshold) pos[count++] = i;"),
    # threshold: no top-1 fallback
    "threshold_no_fallback": ("            if (best >= 0) pos[count++] = best;\n", ""),
    # fallback picks the lowest confidence
    "top1_lowest": ("if (eligible(c[i]) && (best < 0 || ranks_before(c[i], i, c[best], best))) best = i;",
                    "if (eligible(c[i]) && (best < 0 || ranks_before(c[best], best, c[i], i))) best = i;"),
    # fallback breaks ties towards the higher position
    "top1_tie_high": ("if (eligible(c[i]) && (best < 0 || ranks_before(c[i], i, c[best], best))) best = i;",
                      "if (eligible(c[i]) && (best < 0 || c[i] >= c[best])) best = i;"),
    # greedy commits matches at positions already unmasked
    "greedy_ignores_mask": ("if (eligible(c[j]) && p[j] == t[j]) pos[count++] = j;",
                            "if (p[j] == t[j]) pos[count++] = j;"),
    # greedy commits the mismatches
    "greedy_mismatch": ("if (eligible(c[j]) && p[j] == t[j]) pos[count++] = j;",
                        "if (eligible(c[j]) && p[j] != t[j]) pos[count++] = j;"),
    # nan confidence taken as still masked
    "eligible_nan": ("return !isnan(c) && !(isinf(c) && c < 0);", "return !(isinf(c) && c < 0);"),
    # logits: ties go to the last maximum
    "logits_argmax_last": ("if (l > m) { m = l; id = v; }", "if (l >= m) { m = l; id = v; }"),
    # logits: confidence without the max shift
    "logits_no_shift": ("for (int v = 0; v < vocab; ++v) sum += exp(bf16_to_f64(row[v]) - m);",
                        "for (int v = 0; v < vocab; ++v) sum += exp(bf16_to_f64(row[v]));"),
    # logits: the sum leaves out the maximum's own term
    "logits_sum_skips_max": ("for (int v = 0; v < vocab; ++v) sum += exp(bf16_to_f64(row[v]) - m);",
                             "for (int v = 0; v < vocab; ++v) if (v != id) sum += exp(bf16_to_f64(row[v]) - m);"),
    # logits: a row of -inf reads as certain
    "logits_empty_certain": ("if (m == -INFINITY) { conf[r] = 0.0; continue; }",
                             "if (m == -INFINITY) { conf[r] = 1.0; continue; }"),
    # commit: slot from the page index
    "commit_slot": ("const long slot = t % P;", "const long slot = (t / P) % P;"),
    # commit: the prefix advances by the whole block
    "commit_advance_bl": ("if (advance) prefix_lens[b] = (int32_t)(L + count);",
                          "if (advance) prefix_lens[b] = (int32_t)(L + bl);"),
    # commit: the bonus position's row committed as well
    "commit_plus_bonus": ("const int count = counts ? counts[b] : bl;",
                          "const int count = counts ? (counts[b] < bl ? counts[b] + 1 : bl) : bl;"),
    # commit: pool written as [page, slot, head] instead of [page, head, slot]
    "commit_layout": ("const long dst = ((page * Hkv + g) * P + slot) * D;",
                      "const long dst = ((page * P + slot) * Hkv + g) * D;"),
    # quadratic SS: the chain also sees mask slots
    "quadss_chain_sees_masks": ("vis = chain[j] && j <= i;", "vis = j <= i;"),
    # quadratic SS: a mask sees the masks of every group
    "quadss_all_groups": ("(!chain[j] && group[j] == group[i])", "(!chain[j])"),
    # quadratic SS: a mask sees the whole chain
    "quadss_whole_chain": ("(chain[j] && group[j] <= group[i])", "chain[j]"),
    # table mode ignores the table
    "masked_ignores_table": ("if (mode == 2) return (int)((bm[i] >> j) & 1u);", "if (mode == 2) return 1;"),
    # ensemble: the weights swapped
    "ensemble_lambda_swapped": ("const double p = lambda * pa[v] + (1.0 - lambda) * pb[v];",
                                "const double p = (1.0 - lambda) * pa[v] + lambda * pb[v];"),
    # ensemble: ties to the last index
    "ensemble_ties_last": ("if (p > best) { best = p; id = v; }", "if (p >= best) { best = p; id = v; }"),
    # ensemble: mixes unnormalised weights
    "ensemble_unnormalised": ("for (int v = 0; v < vocab; ++v) p[v] /= sum;", ""),
    # selected rows: the triple read as (b, h, i)
    "rows_triple_bhi": ("int b = rows[3 * r], i = rows[3 * r + 1], h = rows[3 * r + 2];",
                        "int b = rows[3 * r], h = rows[3 * r + 1], i = rows[3 * r + 2];"),
    # selected rows: each result written one list position later (wrapping, in bounds)
    "rows_out_shifted": ("s, use, out + r * (long)D, lse + r, NULL);",
                         "s, use, out + ((r + 1) % nsel) * (long)D, lse + (r + 1) % nsel, NULL);"),
    # selected rows: lse written in reverse list order
    "rows_lse_reversed": ("s, use, out + r * (long)D, lse + r, NULL);",
                          "s, use, out + r * (long)D, lse + (nsel - 1 - r), NULL);"),
    # unmask: ascending order
    "unmask_ascending": ("if (ca > cb) return 1;\n    if (ca < cb) return 0;",
                         "if (ca < cb) return 1;\n    if (ca > cb) return 0;"),
}


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_fails_a_pin(tmp_path, name):
    old, new = MUTANTS[name]
    src = open(oracle.SOURCE).read()
    assert src.count(old) == 1, f"mutation site for {name} not unique"
    path = tmp_path / "mutant.c"
    path.write_text(src.replace(old, new))
    lib = oracle.compile_oracle(str(path), str(tmp_path / "libmutant.so"), openmp=False)
    orc = oracle.load(lib)
    failed = []
    for pin in pins.ALL_PINS:
        try:
            pin(orc)
        except (AssertionError, ValueError):
            failed.append(pin.__name__)
    assert failed, f"mutant {name} passed every pin"
