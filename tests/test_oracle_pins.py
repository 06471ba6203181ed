"""The fp64 oracle against what the paper and mathematics fix (CPU only)."""
import oracle
import oracle_pins as P


def test_table1_recompute_column():
    P.pin_table1(oracle.recompute_pct)


def test_eq2_shape():
    P.pin_eq2_shape(oracle.recompute_pct)


def test_redecode_len_integer_ceil():
    P.pin_redecode_len(oracle.redecode_len, oracle.recompute_pct)


def test_rope_inv_freq():
    P.pin_rope_inv_freq(oracle.rope_inv_freq)


def test_rope_matches_complex_product():
    P.pin_rope_complex(oracle.rope_rotate)


def test_rope_2x2_rotation_matrix():
    P.pin_rope_2x2(oracle.rope_rotate)


def test_rope_group_properties():
    P.pin_rope_group(oracle.rope_rotate)


def test_rerotate_reanchors_and_delta0_is_bit_copy():
    P.pin_rerotate(oracle.rerotate, oracle.rope_rotate)


def test_splice_equals_prefill_of_spliced_sequence():
    P.pin_splice_closed_form(oracle.splice_sequence, oracle.rope_rotate)


def test_anchored_splice_byte_identical():
    P.pin_anchored_splice_exact(oracle.splice_sequence, oracle.rope_rotate)


def test_paged_gather_loops():
    P.pin_paged_gather(oracle.paged_gather)


def test_attention_matches_library_sdpa():
    P.pin_attention_library(oracle.attention)


def test_attention_special_cases():
    P.pin_attention_special(oracle.attention)


def test_attention_relative_position_invariance():
    P.pin_attention_shift(oracle.attention, oracle.rope_rotate)


def test_attention_chunk_merge():
    P.pin_attention_split(oracle.attention)


def test_bf16_widening():
    import numpy as np
    import torch
    x = torch.tensor([0.0, -0.0, 1.0, -2.5, 3.140625, float("inf"), 1e-38], dtype=torch.bfloat16)
    bits = x.view(torch.int16).numpy()
    got = oracle.bf16_bits_to_f64(bits)
    assert np.array_equal(got, x.to(torch.float64).numpy())
    assert np.signbit(got[1])


def test_attention_softcap():
    P.pin_attention_softcap(oracle.attention)


def test_qkv_recompute():
    P.pin_qkv_recompute(oracle.qkv_recompute, oracle.rope_rotate)


def test_common_prefix_len():
    P.pin_common_prefix_len(oracle.common_prefix_len)


def test_warm_match():
    P.pin_warm_match(oracle.warm_match, oracle.common_prefix_len)


def test_warm_arena():
    P.pin_warm_arena(oracle.WarmArenaModel)


def test_slb_quantize():
    P.pin_slb_quantize(oracle.slb_quantize)


def test_slb_scores():
    P.pin_slb_scores(oracle.slb_scores, oracle.slb_quantize)


def test_slb_route():
    P.pin_slb_route(oracle.slb_route)


def test_suffix_positions():
    P.pin_suffix_positions(oracle.suffix_positions)
