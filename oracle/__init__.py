"""fp64 CPU oracle of the SA sketching step (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU baseline /
reference legs may import this package; the product path never does.
"""
from .sa_oracle import (affinity, proto_softmax, sa_backward, sa_backward_per_user,  # noqa: F401
                        sa_backward_tokenwise, sa_backward_x, sa_forward, sa_forward_per_user,
                        sa_forward_tokenwise, sa_forward_x, token_softmax)
