"""fp64 CPU oracle for the Qwen3-architecture decoder forward pass.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may import this package.  The
product path (``paper_2609_12471_gb300``) never imports it and shares no code
with it; the two meet only in the seeded inputs of ``synth``.
"""
from .qwen3 import *  # noqa: F401,F403
from .grpo import (group_advantages, grpo_coef, grpo_loss_mean, grpo_token_grad,  # noqa: F401
                   grpo_token_loss, kl_k3)
from .backward import policy_loss_and_grads, sft_loss, sft_loss_and_grads  # noqa: F401
from .sampling import (gumbel, mix64, rollout_sampled, sample_token, sample_uniforms,  # noqa: F401
                       splitmix64_at)
