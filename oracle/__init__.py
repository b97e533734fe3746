"""CPU oracle for PEFT-BD speculative decoding -- TEST INFRASTRUCTURE.

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline leg
may import this package.  The GPU product path never imports, links or runs it, and
it imports nothing from the GPU package: it takes plain numpy arrays (bf16 bit
patterns as uint16) and computes what the paper defines.
"""
from .model import (OracleModel, OracleCache, accept_length, draft_block, greedy_generate,  # noqa: F401
                    spec_generate, adapter_param_count, base_param_count, MASK_CAUSAL, MASK_BLOCK_DRAFT,
                    LINEAR_NAMES)
from .report import draft_cost_table, break_even_accept, predicted_tokens_per_s  # noqa: F401
