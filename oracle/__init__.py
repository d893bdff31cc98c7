"""CPU oracle of the LC-VQ linear layer (LC-QAT, arxiv 2606.10531).

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline / reference legs may import this package. The GPU library never
imports it and shares no code with it.

Pinned by tests/test_oracle_pins.py; every function has at least one pin that
does not re-derive it from its own formula (closed forms, brute force,
finite differences, hand-worked fixtures in tests/golden/).
"""
from .lcvq import (BITS, DGE_GRAD_MAX, DGE_K, ZMAX, SingularMatrix, activation_transform,  # noqa: F401
                   brute_nearest, decode, dge_f,
                   dge_fprime, dge_grad, encode, gemm_packed2b, gemm_packed2b_hadamard, hadamard_block,
                   hadamard_rotate, init_latent, ldl_block, ldlq, ldlq_latent_given_codes, proxy_loss,
                   init_codebook, inverse, latent, linear_bwd, linear_fwd, mse, near_boundary,
                   pack2b, quantize, round_clamp, unpack2b)
