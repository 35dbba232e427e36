"""GB300-native fused output stage of Matryoshka language-model suites.

For every nested sub-model the LM-head logits, the next-token cross-entropy
and the distillation term from the teacher sub-model (paper Eq. 2, Eq. 3),
forward and backward, in hand-written sm_103a kernels behind the C ABI of
include/mls.h.  ``binding`` is the Python face of that ABI.
"""
from .binding import (  # noqa: F401
    HeadLoss,
    MLSError,
    Problem,
    SpecVerify,
    mls_get_status,
    mls_head_loss_bwd,
    mls_head_loss_fwd,
    mls_head_pairwise,
    mls_junction_bwd,
    mls_junction_fwd,
    mls_spec_verify,
    mls_spec_workspace_size,
    mls_strerror,
    mls_workspace_size,
)
