"""Float64 CPU oracle for JARQ refinement.

TEST INFRASTRUCTURE: only the tests, ``__graft_entry__.smoke()`` and the CPU
baseline of ``bench.py`` use this package.  The product path never imports it.
"""
from .jarq_oracle import (FP32_EPS, Options, Prepared, Result, babai_proposal, canonicalize,
                          code_sweep, dequantize, group_target, objective, prepare_hessian,
                          refine_layer, scale_system, solve_scales)
from .jarq_hessian import accumulate_hessian, augmented_hessian
from .jarq_qep import corrected_weights, mu_constant, refine_mu, target_energy
from .jarq_ablation import (coordinate_descent_scales, independent_scales, joint_scales,
                            multicode_probe, refine_fixed_grid, scale_fit_gaps)
from .jarq_format import (dequantize_cast, pack_codes, packed_words, round_to_bfloat16,
                          unpack_codes)

__all__ = ["FP32_EPS", "Options", "Prepared", "Result", "babai_proposal", "canonicalize",
           "code_sweep", "dequantize", "group_target", "objective", "prepare_hessian",
           "refine_layer", "scale_system", "solve_scales", "dequantize_cast", "pack_codes",
           "packed_words", "round_to_bfloat16", "unpack_codes", "accumulate_hessian",
           "augmented_hessian", "corrected_weights", "mu_constant", "refine_mu", "target_energy",
           "coordinate_descent_scales", "independent_scales", "joint_scales", "multicode_probe",
           "refine_fixed_grid", "scale_fit_gaps"]
