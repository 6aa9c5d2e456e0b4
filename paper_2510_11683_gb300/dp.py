"""The data-parallel exchange of a BGPO step (torch.distributed plumbing).

Every (sequence, MC sample) unit of the path is independent once the
advantages and the old policy's l are given (Linearity, Sec. 3), so ranks own
disjoint sequences of the batch (bgpo_problem.b_offset keys their draws by
the global sequence index) and run Algorithm 1's inner loops with no
communication. The one exchange is the sum of the accumulated LM-head gradient
dW over the ranks before the policy update (Algorithm 1 updates the policy
once per outer iteration, after the gradient accumulation of the inner loops).
dX stays with the rank that owns its sequences: it flows back into that
rank's own network.
"""


def allreduce_dw(dW, group=None):
    """Sums dW [V, H] over the ranks of `group` in place (one all-reduce per
    optimiser step; NCCL on GPU tensors, gloo on CPU ones). A single process,
    or a group of one, returns dW unchanged. Returns dW."""
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return dW
    if dist.get_world_size(group) == 1:
        return dW
    dist.all_reduce(dW, op=dist.ReduceOp.SUM, group=group)
    return dW
