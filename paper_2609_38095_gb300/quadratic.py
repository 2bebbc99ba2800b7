"""One full 1.5-SPSA step on the small synthetic workload, on the device.

Algorithm 1 with the quadratic f(theta) = 1/2 sum_i a_i theta_i^2 standing in
for the model's forward pass (an ill-conditioned quadratic of the stiff
paraboloid family, Sec. 5.3): the clean loss L0 once, then per probe k the
loss at theta + eps z_k and at theta - eps z_k, the preconditioner on the
K x 3 loss table (Eqs. 3-5) and the fused update (Eq. 6). Every step of it is
a call of the C ABI; the only other device work is the copy of L0 into the
table's third column (K doubles).

Schedules (the weights at every forward point and after the step are the
same bits in all three):
  onepass  the fused schedule with every perturbation pass and the loss that
           follows it in one launch (zo_perturb_quadratic_loss): 2K + 1
           launches for the forward points, then the preconditioner and the
           update
  fused    the restore of probe k and the +eps of probe k+1 in one pass
           (zo_perturb2), the last restore inside the update pass
           (zo_update_ex); each loss a call of zo_quadratic_loss
  alg1     Algorithm 1's +eps, -2 eps, +eps passes per probe, then the update
The losses of onepass differ from the other two by rounding only (each loss
term carried in fp32 pairs instead of fp64).
"""
import torch

from . import zo

SCHEDULES = ("onepass", "fused", "alg1")


class QuadraticStep:
    """The device buffers of the workload's step: theta (fp32, updated in
    place), the curvatures a (fp32), the loss table, coefficients, status and
    the loss workspace. Nothing is allocated per step."""

    def __init__(self, theta: torch.Tensor, a: torch.Tensor, K: int, eps: float, lr: float, schedule="fused"):
        if schedule not in SCHEDULES:
            raise ValueError(f"schedule must be one of {SCHEDULES}")
        if theta.dtype != torch.float32 or a.dtype != torch.float32 or theta.numel() != a.numel():
            raise ValueError("theta and a must be fp32 tensors of one size")
        if theta.device != a.device:
            raise ValueError("theta and a must live on one device")
        self.theta, self.a, self.K, self.eps, self.lr, self.schedule = theta, a, int(K), float(eps), float(lr), schedule
        dev = theta.device
        self.plist = zo.ParamList([theta])
        self.losses = torch.empty(self.K, 3, dtype=torch.float64, device=dev)
        self.c = torch.empty(self.K, dtype=torch.float64, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.ws = torch.empty(zo.quadratic_loss_workspace_size(theta.numel()), dtype=torch.uint8, device=dev)
        # the loss with its arguments checked once, and the table cells it writes
        self.loss = zo.QuadraticLoss(theta, a, self.ws)
        self.onepass = zo.QuadraticPass(theta, a) if schedule == "onepass" else None
        row = self.losses.stride(0) * self.losses.element_size()
        base = self.loss.out_address(self.losses)
        self._lp = [base + k * row for k in range(self.K)]                  # L+ of probe k
        self._lm = [base + k * row + 8 for k in range(self.K)]              # L- of probe k
        self._l0 = base + 16                                                # L0, row 0
        self._l0_rows = (self.losses[1:, 2], self.losses[0:1, 2].expand(self.K - 1)) if self.K > 1 else None

    def step(self, seed: int):
        """Enqueue one step on the current stream (nothing waits)."""
        K, eps = self.K, self.eps
        if self.onepass is not None:
            q = self.onepass
            q(seed, (), self._l0, copies=K, stride=3)              # clean loss L0 into every row
            q(seed, ((0, eps),), self._lp[0])                      # L+ of probe 0
            for k in range(K):
                q(seed, ((k, -2 * eps),), self._lm[k])             # L- at theta - eps z_k
                if k + 1 < K:                                      # restore k, +eps of k + 1, L+ of k + 1
                    q(seed, ((k, eps), (k + 1, eps)), self._lp[k + 1])
            zo.precondition(self.losses, eps, out=(self.c, self.status))
            zo.update(self.plist, seed, self.c, self.lr, status=self.status, pre=(K - 1, eps))
            return
        self.loss(self._l0)                                    # clean loss L0 (Algorithm 1)
        if self._l0_rows is not None:
            self._l0_rows[0].copy_(self._l0_rows[1])           # into every row's third column
        fused = self.schedule == "fused"
        if fused:
            zo.perturb(self.plist, seed, 0, eps)
        for k in range(K):
            if not fused:
                zo.perturb(self.plist, seed, k, eps)
            self.loss(self._lp[k])                             # L+ at theta + eps z_k
            zo.perturb(self.plist, seed, k, -2 * eps)
            self.loss(self._lm[k])                             # L- at theta - eps z_k
            if not fused:
                zo.perturb(self.plist, seed, k, eps)           # restore
            elif k + 1 < K:
                zo.perturb2(self.plist, seed, k, eps, k + 1, eps)
        zo.precondition(self.losses, eps, out=(self.c, self.status))
        zo.update(self.plist, seed, self.c, self.lr, status=self.status, pre=(K - 1, eps) if fused else None)

    def library_launches_per_step(self) -> int:
        """Kernels of this library one step launches (with zo_quadratic_loss
        the loss is two: partial sums, then their fold)."""
        K = self.K
        if self.schedule == "onepass":
            return 2 * K + 1 + 2
        losses = 2 * (2 * K + 1)
        passes = 2 * K if self.schedule == "fused" else 3 * K
        return losses + passes + 2
