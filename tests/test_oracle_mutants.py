"""Planted mistakes: each edit below is a plausible error in the oracle (a
dropped term, a wrong sign, a wrong index or group map, an off-by-one in the
causal mask, a transposed operand).  Each edited copy is compiled on the CPU
and at least one pin in test_oracle_pins.py must fail against it."""
from __future__ import annotations

import ctypes

import pytest

from oracle import oracle as orc
from tests import test_oracle_pins as pins

MUTANTS = {
    "rope_sin_sign": ("y[i1] = b * cs + a * sn;", "y[i1] = b * cs - a * sn;"),
    "rope_half_pairing": ("int i1 = style == 0 ? k + half : 2 * k + 1;",
                          "int i1 = style == 0 ? half - 1 - k + half : 2 * k + 1;"),
    "rope_frequency": ("pow(base, -2.0 * (double)k / (double)d_rope)", "pow(base, -1.0 * (double)k / (double)d_rope)"),
    "drop_positional_score": ("s[j] = d->sm_scale * (acc + accr);", "s[j] = d->sm_scale * (acc);"),
    "missing_scale": ("s[j] = d->sm_scale * (acc + accr);", "s[j] = (acc + accr);"),
    "group_map_modulo": ("for (int h = g * hpg; h < (g + 1) * hpg; ++h) {", "for (int h = g; h < H; h += G) {"),
    "query_position_off_by_one": ("int64_t p = kv - q_len + i; /* query position; keys 0..p visible */",
                                  "int64_t p = kv - q_len + i - 1;"),
    "w_uk_transposed": ("const uint16_t *w = w_uk + ((int64_t)g * dn + dd) * r;\n                    double acc = 0.0;\n                    for (int rho = 0; rho < r; ++rho) acc += orc_bf16_value(w[rho]) * cj[rho];",
                        "const uint16_t *w = w_uk + (int64_t)g * dn * r + dd;\n                    double acc = 0.0;\n                    for (int rho = 0; rho < r; ++rho) acc += orc_bf16_value(w[(rho * dn) % (dn * r)]) * cj[rho];"),
    "lse_missing_max": ("if (lse) lse[row] = m + log(z);", "if (lse) lse[row] = log(z);"),
    "value_uses_key_weights": ("const uint16_t *w = w_uv + ((int64_t)g * dv + e) * r;",
                               "const uint16_t *w = w_uk + ((int64_t)g * dv + e) * r;"),
    "append_position_shift": ("int64_t pos = (int64_t)start_pos[b] + k, co, ro;",
                              "int64_t pos = (int64_t)start_pos[b] + k + 1, co, ro;"),
    "page_slot": ("slot = t % c->page_size;", "slot = (t + 1) % c->page_size;"),
    "latent_projection_transposed": ("acc += orc_bf16_value(w_dkv[(int64_t)e * D + t]) * x[t];",
                                     "acc += orc_bf16_value(w_dkv[((int64_t)t * r + e) % ((int64_t)r * D)]) * x[t];"),
    "projected_key_unrotated": ("orc_rope(kr, kr, dr, pos, d->rope_base, d->rope_style);\n        for (int e = 0; e < dr; ++e) c->k_rope",
                                "orc_rope(kr, kr, dr, 0, d->rope_base, d->rope_style);\n        for (int e = 0; e < dr; ++e) c->k_rope"),
    "query_rows_head_interleaved": ("const uint16_t *w = w_q + ((int64_t)hd * dq + e) * D;",
                                    "const uint16_t *w = w_q + ((int64_t)e * H + hd) * D;"),
    "acceptance_max_for_min": ("acc += pd < pt ? pd : pt;", "acc += pd > pt ? pd : pt;"),
    "acceptance_target_normaliser": ("pt = exp(t[y] - mt) / zt;", "pt = exp(t[y] - mt) / zd;"),
    "argmax_last_of_ties": ("if (d[y] > d[ad]) ad = y;", "if (d[y] >= d[ad]) ad = y;"),
    "gqa_query_not_rotated": ("orc_rope(qr, qr, dk, p, d->rope_base, d->rope_style);",
                              "orc_rope(qr, qr, dk, 0, d->rope_base, d->rope_style);"),
    "gqa_group_of_head": ("const int g = h / hpg;\n        const int64_t p = (int64_t)kv_len[b] - q_len + i;",
                          "const int g = h % G;\n        const int64_t p = (int64_t)kv_len[b] - q_len + i;"),
    "gqa_value_block": ("tok_offsets(c, b * G + g, j, &co, &ro);\n                acc += exp",
                        "tok_offsets(c, b * G + (g + 1) % G, j, &co, &ro);\n                acc += exp"),
    "e2e_loss_counts_masked_rows": ("if (mask && !mask[t]) continue;", "if (mask && mask[t] > 1) continue;"),
    "e2e_loss_missing_hidden": ("*loss = den > 0.0 ? num / ((double)hidden * den) : 0.0;",
                                "*loss = den > 0.0 ? num / den : 0.0;"),
    "output_projection_index": ("acc += orc_bf16_value(w[h * dv + e]) * o[(row0 + h) * dv + e];",
                                "acc += orc_bf16_value(w[e * H + h]) * o[(row0 + h) * dv + e];"),
}

PINS = [getattr(pins, n) for n in dir(pins) if n.startswith("test_")]


def _run_pins():
    """Run every pin (all parametrisations); return how many failed."""
    failed = 0
    for fn in PINS:
        params = getattr(fn, "pytestmark", [])
        grids = [m for m in params if m.name == "parametrize"]
        cases = [{}]
        for g in grids:
            names = [n.strip() for n in g.args[0].split(",")]
            new = []
            for c in cases:
                for v in g.args[1]:
                    vals = v if len(names) > 1 else (v,)
                    new.append({**c, **dict(zip(names, vals))})
            cases = new
        for kw in cases:
            try:
                fn(**kw)
            except Exception:
                failed += 1
    return failed


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_planted_mistake_is_caught(name, tmp_path, monkeypatch):
    old, new = MUTANTS[name]
    src = orc.source()
    assert src.count(old) >= 1, f"mutation anchor for {name} not found"
    so = orc.compile_variant(src.replace(old, new), str(tmp_path / f"mut_{name}.so"))
    monkeypatch.setattr(orc, "_lib", orc.configure(ctypes.CDLL(so)))
    assert _run_pins() > 0, f"no pin caught the planted mistake {name}"


def test_unmutated_oracle_passes_all_pins(monkeypatch):
    monkeypatch.setattr(orc, "_lib", None)
    assert _run_pins() == 0
