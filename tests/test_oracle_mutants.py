"""The oracle's pins catch plausible mistakes (no GPU).

Each case plants one mistake in the CPU oracle (a dropped term, a wrong sign, index or
normaliser, a transposed operand, a shared state) by editing the source of one oracle
function, and checks that the pins in ``test_oracle_pins.py`` named for it fail on the
mutant.  The mistakes are planted in the oracle only; nothing here touches the CUDA path.
"""
import importlib.util
import inspect
import os
import textwrap

import pytest

from oracle import cachedsearch_oracle as O

_spec = importlib.util.spec_from_file_location(
    "_oracle_pins_for_mutants", os.path.join(os.path.dirname(__file__), "test_oracle_pins.py"))
P = importlib.util.module_from_spec(_spec)
_spec.loader.exec_module(P)

WORKED = "test_cache_rule_worked_example"
HUGE_TAU = "test_huge_tau_skips_every_step_after_the_first_closed_form"
TAU0 = "test_tau_zero_is_uncached_sampling_bitwise"
WINDOWS = "test_warmup_cooldown_windows_force_compute"
X0 = "test_x0_estimate_score_on_last_step_is_final_latent_score"
X0_LINE = "test_x0_estimate_is_exact_for_a_constant_field"
BRUTE = "test_cached_search_brute_force_argmax"
TOPK = "test_topk_order_ties_and_nan"
BLOCK = "test_block_against_torch_functional_composition"
ZERO_BLOCKS = "test_dit_zero_blocks_reduce_to_head_of_embedding"
TEXT_PERM = "test_dit_text_token_permutation_invariance"
ATT_HAND = "test_attention_special_cases"
ATT_SDPA = "test_attention_rows_sum_to_one_and_match_torch_sdpa"
PRIMS = "test_layer_norm_gelu_linear_against_independent_routines"
PATCH = "test_patchify_layout_and_inverse"
SINUS = "test_timestep_sinusoid_values"
CFG = "test_cfg_guidance_one_is_conditional_and_tau_zero_is_uncached_guided_sampling"
BEAM = "test_beam_refill_layout_and_state_copy"
BEAM_DEGENERATE = "test_beam_and_pruned_search_degenerate_cases"
STEP = "test_search_step_equals_per_candidate_rollout"
STATIC = "test_static_schedule_hand_example_and_every_one_is_uncached"
MOD_CLOSED = "test_modulation_closed_form_through_identity_weights"
MOD_SINUS = "test_modulation_sinusoid_path_closed_form"
ADALN_ROLES = "test_adaln_vectors_play_their_roles_in_the_block"
HEAD_ROLES = "test_head_modulation_roles"
TEXT_CLOSED = "test_text_kv_closed_form_through_identity_weights"
COND_TORCH = "test_conditioning_against_torch_nn_composition"
ROWS = "test_row_subset_forms_equal_the_full_forward"

# (id, oracle function, text replaced, replacement, pins that must fail on the mutant)
MUTANTS = [
    # sampler (Sec. 2, Eq. euler)
    ("grid-denominator", "time_grid", "/ T", "/ (T + 1)", ["test_time_grid_endpoints_and_spacing"]),
    ("euler-sign", "euler", "x + (t_next", "x - (t_next",
     ["test_euler_linear_field_closed_form", "test_euler_constant_field_reaches_x1_minus_v", WORKED]),
    ("cached-velocity-at-next-time", "rollout", "velocity_fn_t(z, t[k - 1])", "velocity_fn_t(z, t[k])",
     [TAU0, HUGE_TAU]),
    ("uncached-velocity-at-next-time", "rollout_uncached", "velocity_fn_t(x, t[k - 1])",
     "velocity_fn_t(x, t[k])", [TAU0, CFG]),
    # indicator (Eq. indicator)
    ("drift-not-normalised", "relative_drift", " / np.sqrt(np.sum(x_ref ** 2))", "", [WORKED]),
    ("drift-normalised-by-x", "relative_drift", "np.sum(x_ref ** 2)", "np.sum(x ** 2)", [WORKED]),
    ("drift-squared-norm", "relative_drift", "np.sqrt(np.sum((x - x_ref) ** 2))",
     "np.sum((x - x_ref) ** 2)", [WORKED]),
    ("indicator-not-accumulated", "wrapper_call", "(st.a > tau)", "(drift > tau)", [WORKED]),
    ("indicator-not-reset", "wrapper_call", "st.a = 0.0\n", "pass\n", [WORKED]),
    # cache (Eq. delta, Eq. skip)
    ("delta-sign", "wrapper_call", "st.delta = v - x", "st.delta = x - v", [WORKED, HUGE_TAU]),
    ("skip-reuses-cached-output", "wrapper_call", "v = x + st.delta", "v = st.x_ref + st.delta",
     [WORKED, HUGE_TAU]),
    ("reference-not-refreshed", "wrapper_call", "st.x_ref = x.copy()",
     "st.x_ref = x.copy() if st.x_ref is None else st.x_ref", [WORKED]),
    ("warmup-off-by-one", "forced_compute", "return k <= K_w", "return k < K_w", [WINDOWS]),
    ("cooldown-off-by-one", "forced_compute", "or k > T - K_c or", "or k >= T - K_c or", [WINDOWS]),
    ("empty-cache-not-forced", "forced_compute", " or not has_ref", "", [WORKED, HUGE_TAU]),
    # batched step, scoring and selection (Algorithm 1)
    ("candidates-share-one-state", "search_step", "wrapper_call(st,", "wrapper_call(states[0],",
     [STEP]),
    ("x0-estimate-wrong-time", "search_step", "x0 = out - t[k] *", "x0 = out - t[k - 1] *", [X0, X0_LINE]),
    ("x0-estimate-is-next-latent", "search_step", "x0 = out - t[k] * np.stack(vs)", "x0 = out", [X0_LINE]),
    ("score-sign", "score", "return -float(", "return float(", [X0, BRUTE]),
    ("score-squared", "score", "np.sqrt(np.sum(", "(np.sum(", [X0, BRUTE]),
    ("topk-ascending", "topk", "(-key[i][0], i)", "(key[i][0], i)", [TOPK]),
    ("topk-ties-high-index-first", "topk", "(-key[i][0], i)", "(-key[i][0], -i)", [TOPK]),
    ("topk-nan-first", "topk", "-np.inf if np.isnan(v)", "np.inf if np.isnan(v)", [TOPK]),
    ("refill-drops-survivor", "beam_refill", "range(children + 1)", "range(children)", [BEAM]),
    ("refill-children-fresh-state", "beam_refill", "new_states.append(cp)",
     "new_states.append(cp if j == 0 else CacheState())", [BEAM, BEAM_DEGENERATE]),
    ("refill-resets-indicator", "beam_refill", "st.x_ref.copy(), st.a)", "st.x_ref.copy(), 0.0)", [BEAM]),
    ("static-phase", "static_schedule", "(k - K_w) % every", "(k - K_w - 1) % every", [STATIC]),
    ("cfg-base-branch", "cfg_combine", "v_uncond + w", "v_cond + w", [CFG]),
    ("cfg-branches-share-state", "search_step_cfg", "wrapper_call(states_u[i]", "wrapper_call(states_c[i]",
     [CFG]),
    # DiT primitives
    ("attention-scale", "attention", "/ np.sqrt(hd)", "/ hd", [ATT_HAND, ATT_SDPA]),
    ("softmax-axis", "softmax_rows", "e / e.sum(axis=-1", "e / e.sum(axis=0", [ATT_HAND, ATT_SDPA]),
    ("value-heads-strided", "multi_head_attention", "v[:, h * hd:(h + 1) * hd]", "v[:, h::heads]", [BLOCK]),
    ("layernorm-eps-outside-root", "layer_norm", "np.sqrt(var + eps)", "(np.sqrt(var) + eps)", [PRIMS]),
    ("layernorm-unbiased-variance", "layer_norm", "((x - mu) ** 2).mean(axis=-1, keepdims=True)",
     "((x - mu) ** 2).sum(axis=-1, keepdims=True) / (x.shape[-1] - 1)", [PRIMS]),
    ("gelu-without-cubic", "gelu_tanh", " + 0.044715 * x ** 3", "", [PRIMS]),
    ("linear-untransposed", "linear", "np.float64).T +", "np.float64) +", [PRIMS, BLOCK]),
    ("patch-subpixel-order", "patchify", ".transpose(1, 2, 4, 0, 3, 5)", ".transpose(1, 2, 4, 0, 5, 3)",
     [PATCH]),
    ("unpatch-axes", "unpatchify", ".transpose(3, 0, 1, 4, 2, 5)", ".transpose(3, 0, 2, 4, 1, 5)", [PATCH]),
    ("sinusoid-sin-cos", "timestep_sinusoid", "[np.cos(arg), np.sin(arg)]", "[np.sin(arg), np.cos(arg)]",
     [SINUS]),
    ("sinusoid-frequency", "timestep_sinusoid", "/ half)", "/ (half - 1))", [SINUS]),
    # DiT block and head
    ("block-gate-dropped", "DiT.block", "x + gate1 * linear(sa", "x + linear(sa", [BLOCK]),
    ("block-scale-without-one", "DiT.block", "* (1.0 + scale1)", "* scale1", [BLOCK]),
    ("block-cross-without-norm", "DiT.block", "h = layer_norm(x)\n", "h = x\n", [BLOCK]),
    ("block-q-k-swapped", "DiT.block", "multi_head_attention(qkv[:, :d], qkv[:, d:2 * d]",
     "multi_head_attention(qkv[:, d:2 * d], qkv[:, :d]", [BLOCK]),
    ("block-ffn-residual-dropped", "DiT.block", "return x + gate2 * f", "return gate2 * f",
     [BLOCK, ZERO_BLOCKS]),
    ("cross-k-v-swapped", "DiT.block", "multi_head_attention(qc, kv[0], kv[1], H)",
     "multi_head_attention(qc, kv[1], kv[0], H)", [BLOCK]),
    ("text-kv-rows-misaligned", "DiT.text_kv", "kv.append((y[:, :d], y[:, d:]))",
     "kv.append((y[:, :d], np.roll(y[:, d:], 1, axis=0)))", [TEXT_PERM]),
    ("head-shift-scale-swapped", "DiT.velocity", "(1.0 + hm[1]) + hm[0]", "(1.0 + hm[0]) + hm[1]",
     [ZERO_BLOCKS]),
    ("head-without-norm", "DiT.velocity", "layer_norm(tok) * (1.0", "tok * (1.0", [ZERO_BLOCKS]),
    ("block-shift-scale1-swapped", "DiT.block", "* (1.0 + scale1) + shift1", "* (1.0 + shift1) + scale1",
     [ADALN_ROLES]),
    ("block-shift-scale2-swapped", "DiT.block", "* (1.0 + scale2) + shift2", "* (1.0 + shift2) + scale2",
     [ADALN_ROLES]),
    ("block-gate2-dropped", "DiT.block", "x + gate2 * f", "x + f", [ADALN_ROLES]),
    # conditioning MLPs (timestep embedding -> adaLN vectors; text projection -> K/V)
    ("mod-silu-dropped", "DiT.modulation", 'linear(silu(e), p["mod_w"]', 'linear(e, p["mod_w"]',
     [MOD_CLOSED, COND_TORCH]),
    ("mod-shift-scale-swapped", "DiT.modulation", ".reshape(6, d)", ".reshape(6, d)[[1, 0, 2, 3, 4, 5]]",
     [MOD_CLOSED, COND_TORCH]),
    ("mod-offset-not-added", "DiT.modulation", 'm + p[f"blk{b}.mod_off"]', 'm + 0 * p[f"blk{b}.mod_off"]',
     [MOD_CLOSED, COND_TORCH]),
    ("mod-offset-of-block-0", "DiT.modulation", 'p[f"blk{b}.mod_off"]', 'p["blk0.mod_off"]',
     [MOD_CLOSED, COND_TORCH]),
    ("head-mod-silu-dropped", "DiT.modulation", "hm = linear(silu(e)", "hm = linear(e", [MOD_CLOSED, COND_TORCH]),
    ("head-mod-shift-scale-swapped", "DiT.modulation", ".reshape(2, d)", ".reshape(2, d)[::-1]",
     [MOD_CLOSED, HEAD_ROLES, COND_TORCH]),
    ("time-mlp-silu-dropped", "DiT.modulation", "e = linear(silu(linear(timestep_sinusoid",
     "e = linear((linear(timestep_sinusoid", [MOD_SINUS, COND_TORCH]),
    ("sinusoid-time-scale", "timestep_sinusoid", "arg = 1000.0 * float(t)", "arg = float(t)",
     [SINUS, MOD_SINUS, COND_TORCH]),
    ("text-gelu-dropped", "DiT.text_kv", "txt = linear(gelu_tanh(linear(", "txt = linear((linear(",
     [TEXT_CLOSED, COND_TORCH]),
    ("text-kv-split-swapped", "DiT.text_kv", "kv.append((y[:, :d], y[:, d:]))", "kv.append((y[:, d:], y[:, :d]))",
     [TEXT_CLOSED, COND_TORCH]),
    ("rows-keys-from-subset", "DiT.block_rows", "kv_self = linear(layer_norm(x) *", "kv_self = linear(layer_norm(x[rows]) *",
     [ROWS]),
    ("rows-value-heads-from-keys", "DiT.block_rows", "kv_self[:, :d], kv_self[:, d:], H)",
     "kv_self[:, :d], kv_self[:, :d], H)", [ROWS]),
    ("rows-head-scale-dropped", "DiT.velocity_rows", "* (1.0 + hm[1]) + hm[0]", "+ hm[0]", [ROWS]),
    ("text-kv-one-block", "DiT.text_kv", 'linear(txt, p[f"blk{b}.ckv_w"], p[f"blk{b}.ckv_b"])',
     'linear(txt, p["blk0.ckv_w"], p["blk0.ckv_b"])', [TEXT_CLOSED, COND_TORCH]),
]


def _plant(monkeypatch, qual, old, new):
    owner = O
    name = qual
    if "." in qual:
        cls, name = qual.split(".")
        owner = getattr(O, cls)
    src = textwrap.dedent(inspect.getsource(getattr(owner, name)))
    assert src.count(old) == 1, f"{qual}: the planted text must occur exactly once"
    ns = {}
    exec(compile(src.replace(old, new), f"<mutant of {qual}>", "exec"), vars(O), ns)
    monkeypatch.setattr(owner, name, ns[name])


def _fails(pin):
    try:
        getattr(P, pin)()
    except Exception:  # an assertion, or the mutant breaking a shape
        return True
    return False


@pytest.mark.parametrize("mid,qual,old,new,pins", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_planted_mistake(monkeypatch, mid, qual, old, new, pins):
    _plant(monkeypatch, qual, old, new)
    survived = [p for p in pins if not _fails(p)]
    assert not survived, f"mutant {mid} passes {survived}"


def test_unmutated_oracle_passes_the_same_pins():
    pins = sorted({p for m in MUTANTS for p in m[4]})
    assert not [p for p in pins if _fails(p)]
