"""torch.optim front end of the library's R-iKFAD step.

``RIKFADOptimizer(params, lr, alpha, mu, gamma=0.0, eps_stab=1e-16)`` steps every
parameter of a group in one ``rikfad_step`` call: 2-D parameters by the rank-1
friction rule, every other shape element-wise (Section 2 of the paper; ``lr`` is
the step size h).  It is argument marshalling only: a group's handle is created
at its first step, the momentum buffers live in ``self.state[p]["momentum"]`` in
the library's stored form, and ``materialize()`` turns them into the paper's P.
``state_dict()`` also carries each group's library state image, so a checkpoint
resumes the exact trajectory.
Parameters and their gradients must be contiguous float32 CUDA tensors of one
device (autograd gives a float32 parameter a float32 gradient; bfloat16
gradients are for the pointer API, ``rikfad.RIKFAD``).  A parameter without a
gradient at a step takes a zero gradient, since the handle steps a fixed list.
"""
import torch

from . import rikfad


class RIKFADOptimizer(torch.optim.Optimizer):
    def __init__(self, params, lr, alpha, mu, gamma=0.0, eps_stab=1e-16):
        if not lr > 0:
            raise ValueError("lr (the step size h) must be > 0")
        defaults = dict(lr=lr, alpha=alpha, mu=mu, gamma=gamma, eps_stab=eps_stab)
        super().__init__(params, defaults)
        self._groups = {}     # group index -> (handle, parameter list, zero gradients)

    @staticmethod
    def _shape(p):
        return (p.shape[0], p.shape[1]) if p.dim() == 2 else (p.numel(), 0)

    def _group_handle(self, i, group):
        params = group["params"]
        entry = self._groups.get(i)
        if entry is not None and len(entry[1]) == len(params) and all(a is b for a, b in zip(entry[1], params)):
            return entry
        if entry is not None:
            entry[0].close()
        for p in params:
            if not (p.is_cuda and p.dtype == torch.float32 and p.is_contiguous()):
                raise ValueError("parameters must be contiguous float32 CUDA tensors")
            if p.device != params[0].device:
                raise ValueError("parameters of a group must share one device")
        handle = rikfad.RIKFAD([self._shape(p) for p in params], group["alpha"], group["mu"],
                               group["gamma"], group["eps_stab"], grad_dtype="f32")
        entry = (handle, list(params), [torch.zeros_like(p) for p in params])
        self._groups[i] = entry
        return entry

    def _momenta(self, params):
        out = []
        for p in params:
            st = self.state[p]
            if "momentum" not in st:
                st["momentum"] = torch.zeros_like(p)
            out.append(st["momentum"])
        return out

    @torch.no_grad()
    def step(self, closure=None):
        loss = None
        if closure is not None:
            with torch.enable_grad():
                loss = closure()
        for i, group in enumerate(self.param_groups):
            if not group["params"]:
                continue
            handle, params, zeros = self._group_handle(i, group)
            grads = []
            for p, z in zip(params, zeros):
                g = p.grad
                if g is not None and not (g.dtype == torch.float32 and g.is_contiguous()):
                    raise ValueError("gradients must be contiguous float32 tensors")
                grads.append(z if g is None else g)
            handle.step(group["lr"], params, grads, self._momenta(params),
                        stream=torch.cuda.current_stream(params[0].device))
        return loss

    @torch.no_grad()
    def materialize(self):
        """Turn every momentum buffer into the paper's P_{n+1} (in place)."""
        for handle, params, _ in self._groups.values():
            handle.materialize(self._momenta(params), stream=torch.cuda.current_stream(params[0].device))

    def state_dict(self):
        """torch's state (the momentum buffers, in the stored form) plus each
        group's library state image (factors, element-wise friction and the
        pending step size; rikfad_export_state) as a CPU byte tensor."""
        sd = super().state_dict()
        images = {}
        for i, group in enumerate(self.param_groups):
            entry = self._groups.get(i)
            if entry is not None:
                handle, params, _ = entry
                img = torch.empty(handle.state_image_bytes(), dtype=torch.uint8, device=params[0].device)
                handle.export_state(img, stream=torch.cuda.current_stream(params[0].device))
                images[i] = img.cpu()
        sd["rikfad_images"] = images
        return sd

    def load_state_dict(self, state_dict):
        sd = dict(state_dict)
        images = sd.pop("rikfad_images", {})
        self.close()          # the groups are replaced; handles are made again below or at the next step
        super().load_state_dict(sd)
        for i, group in enumerate(self.param_groups):
            if i in images:
                handle, params, _ = self._group_handle(i, group)
                img = images[i].to(params[0].device)
                handle.import_state(img, stream=torch.cuda.current_stream(params[0].device))

    def check_finite(self):
        """Raise rikfad.RikfadError(ERR_NONFINITE) if a step produced a
        non-finite factor, friction or denominator (see rikfad_check_finite)."""
        for handle, params, _ in self._groups.values():
            handle.check_finite(torch.cuda.current_stream(params[0].device))

    def close(self):
        for handle, _, _ in self._groups.values():
            handle.close()
        self._groups.clear()
