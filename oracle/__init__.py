"""fp64 CPU oracle of the BOM step and update (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline legs of
``bench.py`` may import this package; the product path never does.
"""
from .bom_oracle import (  # noqa: F401
    OracleError, LabelError, EmptyError,
    gelu, gelu_prime, silu, silu_prime,
    forward, backward, supervised_set, softmax_rows, log_sum_exp_rows, residuals,
    batch_mean_residual, ema_update, cross_entropy, bom_step, bom_update,
    mix_numerator, bom_update_gh, mix_cotangent_rows, head_weight_grad_rows, head_input_grad_rows, mix_grad_rows,
    own_step_projection, own_step_moment, drift_statistics, cancellation_ratio,
    bom_update_blockshared, clip_factor, bom_update_clipped,
)
