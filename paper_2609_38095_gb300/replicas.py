"""Probe-parallel 1.5-SPSA step over R replicas (Sec. 4.3, Algorithm 1): the
host-side protocol around the single-GPU calls.

Every replica holds the whole parameter set. Probe k of a step belongs to
rank k mod R. A replica evaluates the loss triples (L+, L-, L0) of its own
probes only; then the replicas exchange the triples (a K x 3 fp64 table, the
only data that crosses ranks in a step) and every replica runs the same
preconditioner and fused update on the full table. Both are deterministic
functions of (seed, table, lr), so replicas whose parameters were
bit-identical before the step are bit-identical after it -- provided the
probe passes leave the parameters untouched, which the out-of-place pair
schedule (zo_perturb_pair) guarantees. That schedule needs no parameter
broadcast at all.

The in-place schedule (+eps, -2eps, +eps per probe) leaves each replica's
parameters with the rounding drift of the restores of its own probes, which
differ between ranks; there the parameters of rank 0 are broadcast after the
update, which is Algorithm 1's broadcast moved from the start of the next
step to the end of this one.

How this differs from Algorithm 1: no seed scatter (probe k is a function of
the step seed and k on every rank), the losses are all-gathered instead of
gathered at rank 0, and every rank applies the update instead of rank 0
alone.

The collectives go through torch.distributed (any backend: the tests run
gloo ranks on CPU); the probe passes, preconditioner and update are the
library's CUDA calls. Without an initialised process group a step runs as a
single replica.
"""
import torch
import torch.distributed as dist

from . import zo

SCHEDULES = ("pair", "inplace")


def probes_of_rank(K: int, rank: int, world: int) -> range:
    """The probes rank `rank` of `world` evaluates: k = rank, rank + world, ..."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside a world of {world}")
    if K < 0:
        raise ValueError("K must be >= 0")
    return range(rank, K, world)


def assemble_losses(parts, K: int, world: int) -> torch.Tensor:
    """Full (K, 3) table from the per-rank rows: parts[r] holds the rows of
    probes_of_rank(K, r, world) in increasing k (extra padding rows are
    ignored). Rows are copied, never combined, so the table is bit-exact."""
    if len(parts) != world:
        raise ValueError(f"{len(parts)} parts for a world of {world}")
    ref = parts[0]
    table = torch.empty(K, 3, dtype=ref.dtype, device=ref.device)
    for r, part in enumerate(parts):
        n = len(probes_of_rank(K, r, world))
        if part.dim() != 2 or part.shape[1] != 3 or part.shape[0] < n:
            raise ValueError(f"rank {r} sent {tuple(part.shape)} rows for its {n} probes")
        table[r::world] = part[:n]
    return table


def _tensors(x):
    return x.tensors if isinstance(x, zo.ParamList) else list(x)


def _world(group):
    if dist.is_available() and dist.is_initialized():
        return dist.get_rank(group), dist.get_world_size(group)
    return 0, 1


def all_gather_losses(own: torch.Tensor, K: int, group=None) -> torch.Tensor:
    """Exchange the rows of this rank's probes; every rank gets the full
    (K, 3) table. `own` lives where the group's backend wants it (CPU for
    gloo, the rank's GPU for nccl)."""
    rank, world = _world(group)
    n_own = len(probes_of_rank(K, rank, world))
    if own.dim() != 2 or own.shape != (n_own, 3):
        raise ValueError(f"rank {rank} holds {tuple(own.shape)} rows, expected ({n_own}, 3)")
    if world == 1:
        return own.clone()
    m = -(-K // world)                    # the most probes any rank owns
    buf = torch.zeros(m, 3, dtype=own.dtype, device=own.device)
    buf[:n_own] = own
    parts = [torch.empty_like(buf) for _ in range(world)]
    dist.all_gather(parts, buf, group=group)
    return assemble_losses(parts, K, world)


def broadcast_params(params, src: int = 0, group=None):
    """Copy rank `src`'s parameters to every rank (in place)."""
    _, world = _world(group)
    if world == 1:
        return
    for t in _tensors(params):
        if t.numel():
            dist.broadcast(t, src=src, group=group)


def pair_probe_losses(params, plus, minus, seed: int, K: int, eps: float, rank: int, world: int, loss_into,
                      l0: torch.Tensor) -> torch.Tensor:
    """Rows (L+, L-, L0) of this rank's probes with the out-of-place pair
    schedule: per probe one zo_perturb_pair pass writes theta +- eps z_k to
    plus / minus, and loss_into(tensors, out) writes the loss of a tensor
    list into the one-element fp64 tensor out. theta is not written."""
    mine = probes_of_rank(K, rank, world)
    rows = torch.empty(len(mine), 3, dtype=torch.float64, device=l0.device)
    rows[:, 2] = l0
    for i, k in enumerate(mine):
        zo.perturb_pair(params, plus, minus, seed, k, eps)
        loss_into(_tensors(plus), rows[i, 0:1])
        loss_into(_tensors(minus), rows[i, 1:2])
    return rows


def inplace_probe_losses(params, seed: int, K: int, eps: float, rank: int, world: int, loss_into,
                         l0: torch.Tensor):
    """Rows of this rank's probes with Algorithm 1's in-place sequence, the
    restore of each probe fused with the next probe's +eps (zo_perturb2).
    Returns (rows, pending): pending = (probe, +eps) is the last restore,
    left for the update to apply in its own pass, or None."""
    mine = list(probes_of_rank(K, rank, world))
    rows = torch.empty(len(mine), 3, dtype=torch.float64, device=l0.device)
    rows[:, 2] = l0
    if not mine:
        return rows, None
    tensors = _tensors(params)
    zo.perturb(params, seed, mine[0], eps)
    for i, k in enumerate(mine):
        loss_into(tensors, rows[i, 0:1])
        zo.perturb(params, seed, k, -2.0 * eps)
        loss_into(tensors, rows[i, 1:2])
        if i + 1 < len(mine):
            zo.perturb2(params, seed, k, eps, mine[i + 1], eps)
    return rows, (mine[-1], eps)


def finish_step(params, table: torch.Tensor, seed: int, eps: float, lr=None, alpha: float = 0.1,
                lambda_reg: float = 1.0, pending=None):
    """The part every replica runs on the full (K, 3) table: preconditioner
    and fused update (with the pending restore of the in-place schedule, if
    any). Returns (c, status)."""
    c, status = zo.precondition(table, eps, alpha=alpha, lambda_reg=lambda_reg)
    zo.update(params, seed, c, eps if lr is None else lr, status=status, pre=pending)
    return c, status


def step(params, seed: int, K: int, eps: float, loss_into, lr=None, alpha: float = 0.1, lambda_reg: float = 1.0,
         schedule: str = "pair", plus=None, minus=None, group=None):
    """One probe-parallel 1.5-SPSA step on this rank; returns (table, c,
    status) as device tensors.

    params: this replica's parameters (a ParamList or a list of CUDA
    tensors); plus / minus: two lists shaped like params (pair schedule
    only). loss_into(tensors, out) writes the loss of a list of tensors into
    the one-element fp64 tensor out. lr defaults to eps (Algorithm 1). The
    loss rows are exchanged with all_gather_losses over `group` (nccl for
    CUDA rows)."""
    if schedule not in SCHEDULES:
        raise ValueError(f"schedule must be one of {SCHEDULES}")
    if schedule == "pair" and (plus is None or minus is None):
        raise ValueError("the pair schedule needs plus and minus buffers")
    rank, world = _world(group)
    plist = params if isinstance(params, zo.ParamList) else zo.ParamList(list(params))
    dev = plist.device
    l0 = torch.empty(1, dtype=torch.float64, device=dev)
    loss_into(plist.tensors, l0)
    if schedule == "pair":
        own = pair_probe_losses(plist, plus, minus, seed, K, eps, rank, world, loss_into, l0)
        pending = None
    else:
        own, pending = inplace_probe_losses(plist, seed, K, eps, rank, world, loss_into, l0)
    table = all_gather_losses(own, K, group=group)
    c, status = finish_step(plist, table, seed, eps, lr=lr, alpha=alpha, lambda_reg=lambda_reg, pending=pending)
    if schedule == "inplace":
        broadcast_params(plist, src=0, group=group)
    return table, c, status
