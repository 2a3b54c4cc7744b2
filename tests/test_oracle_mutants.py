"""Plausible mistakes planted in a copy of the oracle are each caught by at
least one pin (CPU only; the planted copies are compiled into a temporary
directory and never touch the real oracle)."""
import os

import pytest

import oracle
from oracle_pins import ALL_PINS

SRC = os.path.join(os.path.dirname(oracle.__file__), "gbla_oracle.c")

# (id, text in the oracle, replacement) -- each a one-token slip
MUTANTS = [
    ("phi_drops_plus_one", "return x > 0.0 ? x + 1.0 : exp(x);", "return x > 0.0 ? x : exp(x);"),
    ("phi_wrong_branch", "return x > 0.0 ? x + 1.0 : exp(x);", "return x >= 1.0 ? x + 1.0 : exp(x);"),
    ("silu_sign", "return x / (1.0 + exp(-x));", "return x / (1.0 + exp(x));"),
    ("conv_taps_reversed", "acc += w[(long)c * W + i] * x[s * ldx + c];",
     "acc += w[(long)c * W + (W - 1 - i)] * x[s * ldx + c];"),
    ("conv_off_by_one", "long s = t - (W - 1) + i;", "long s = t - W + i;"),
    ("conv_not_causal", "long s = t - (W - 1) + i;", "long s = t + i;"),
    ("softmax_no_max", "g[j] = exp(a[j * lda] - m);", "g[j] = exp(a[j * lda]);"),
    ("softmax_not_normalised", "for (long j = 0; j < L; ++j) g[j] /= s;",
     "for (long j = 0; j < L; ++j) g[j] /= 1.0;"),
    ("state_wrong_v_index", "S[d * D + e] += pk[d] * vt[j * D + e];",
     "S[d * D + e] += pk[d] * vt[j * D + d];"),
    ("z_ungated", "z[d] += pk[d];", "z[d] += oracle_phi(kt[j * D + d]);"),
    ("state_gate_dropped",
     "for (int d = 0; d < D; ++d) pk[d] = g[j] * oracle_phi(kt[j * D + d]);",
     "for (int d = 0; d < D; ++d) pk[d] = oracle_phi(kt[j * D + d]);"),
    ("readout_transposed", "num += pq[d] * S[d * D + e];", "num += pq[d] * S[e * D + d];"),
    ("readout_no_phi_q", "pq[d] = oracle_phi(qt[i * D + d]);", "pq[d] = qt[i * D + d];"),
    ("rms_sum_not_mean", "ms /= (double)D;", "ms /= 1.0;"),
    ("rms_eps_outside", "double r = 1.0 / sqrt(ms + eps);", "double r = 1.0 / (sqrt(ms) + eps);"),
    ("norm_weight_dropped", "y[d] = O[d] * r * w[d] * oracle_silu(og[d]);",
     "y[d] = O[d] * r * oracle_silu(og[d]);"),
    ("gate_not_silu", "y[d] = O[d] * r * w[d] * oracle_silu(og[d]);",
     "y[d] = O[d] * r * w[d] * og[d];"),
    ("uniform_gate_wrong", "g[j] = 1.0 / (double)L;", "g[j] = 1.0;"),
    ("driver_conv_head_offset", "J->conv_w + ((1 * J->H + h) * D) * W",
     "J->conv_w + ((1 * J->H + 0) * D) * W"),
    ("driver_gate_stride", "J->gate + b * J->N * J->H + h, J->og + base, ld, J->H,",
     "J->gate + b * J->N * J->H + h, J->og + base, ld, 1,"),
    ("driver_norm_head", "J->norm_w + h * D", "J->norm_w"),
    ("driver_len_unclamped", "if (L > J->N) L = J->N;", "if (L > J->N) L = J->N + 0; L = J->N;"),
    ("quadratic_gate_on_query", "A[i * L + j] = g[j] * s;", "A[i * L + j] = g[i] * s;"),
    ("project_stream_interleaved", "const long s = f / HD, col = f % HD;",
     "const long s = f % 4, col = f / 4;"),
    ("project_gate_column", "gate[(b * N + t) * H + (f - 4 * HD)] = acc;",
     "gate[(b * N + t) * H + (f - 4 * HD + 1) % H] = acc;"),
    ("project_weight_transposed", "acc += xr[c] * wr[c];",
     "acc += xr[c] * w[(long)c * F + f];"),
    ("project_skips_conv", "const double *xr = xt + t * d;",
     "const double *xr = x + (b * N + t) * d;"),
    ("project_batch_offset", "oracle_conv1d(x + b * N * d, L, d, d, conv_x, W, xt);",
     "oracle_conv1d(x, L, d, d, conv_x, W, xt);"),
    ("project_writes_padding", "for (long t = 0; t < L; ++t) {\n      const double *xr",
     "for (long t = 0; t < N; ++t) {\n      const double *xr"),
    ("project_absdot_signed", "mag += fabs(xr[c] * wr[c]);", "mag += xr[c] * wr[c];"),
    ("sa_no_scale", "s[j] = dot * scale;", "s[j] = dot;"),
    ("sa_no_max", "s[j] = exp(s[j] - m);", "s[j] = exp(s[j]);"),
    ("sa_keys_from_tail", "sa_row(J->q + base + i * ld, J->k + base, J->v + base, L,",
     "sa_row(J->q + base + i * ld, J->k + base + (N - L) * ld, J->v + base, L,"),
    ("sa_key_head", "sa_row(J->q + base + i * ld, J->k + base, J->v + base",
     "sa_row(J->q + base + i * ld, J->k + b * N * H * D, J->v + base"),
    ("sa_not_normalised", "out[d] /= den;", "out[d] /= 1.0;"),
    ("sa_value_index", "out[d] += s[j] * vj[d];", "out[d] += s[j] * vj[0];"),
    ("sa_abs_unsigned", "absout[d] += s[j] * fabs(vj[d]);", "absout[d] += s[j] * vj[d];"),
    ("bwd_dden_sign", "const double dden = -dOO / den[i];", "const double dden = dOO / den[i];"),
    ("bwd_dS_transposed", "for (int e = 0; e < D; ++e) dS[d * D + e] += P[d] * dnum[e];",
     "for (int e = 0; e < D; ++e) dS[e * D + d] += P[d] * dnum[e];"),
    ("bwd_phi_prime_branch", "return x > 0.0 ? 1.0 : exp(x);", "return x > 0.0 ? 1.0 : 1.0;"),
    ("bwd_conv_transpose_causal", "long t = s + (W - 1) - i;", "long t = s - (W - 1) + i;"),
    ("bwd_norm_cube", "dOi[e] = r * u - (r * r * r / (double)D) * Oi[e] * uo;",
     "dOi[e] = r * u - (r * r / (double)D) * Oi[e] * uo;"),
    ("scale_state_signed", "Sa[d * D + e] += kh * fabs(vt[j * D + e]);",
     "Sa[d * D + e] += kh * vt[j * D + e];"),
    ("scale_conv_signed",
     "if (t < L) acc += fabs(taps[m][(long)c * W + i]) * src[m][t * D + c];",
     "if (t < L) acc += taps[m][(long)c * W + i] * src[m][t * D + c];"),
]


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(name, old, new, tmp_path):
    text = open(SRC).read()
    assert text.count(old) >= 1, f"mutation target for {name} not found in the oracle"
    src = tmp_path / "mutant.c"
    src.write_text(text.replace(old, new, 1))
    so = oracle.build(str(src), str(tmp_path / "libmutant.so"))
    lib = oracle.load(so)
    caught = []
    for pin in ALL_PINS:
        try:
            pin(lib)
        except AssertionError:
            caught.append(pin.__name__)
        except (ValueError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"no pin caught the planted mistake {name}"
