"""Device-memory plumbing for libmoara: torch tensors that back one module's
buffers, and a small driver that owns a context.  Every computation happens in
the library's kernels; torch only allocates and holds memory.
"""

from __future__ import annotations

import torch

from . import binding as B


def _bf16_bits(t):
    return t.to(torch.bfloat16).view(torch.int16)


class ModuleBuffers:
    """Caller-owned buffers of one registered weight (layouts of moara.h)."""

    def __init__(self, m, n, r, block_size, grad_dtype="bf16", device="cuda",
                 W0=None, with_bf16=True, state_dtype="f32", right=False):
        self.m, self.n, self.r, self.block_size = m, n, r, block_size
        self.kb = -(-n // block_size)
        self.grad_dtype = grad_dtype
        dev = torch.device(device)
        f32 = dict(dtype=torch.float32, device=dev)
        # W and the direction moments in fp32, or bf16 (hparams.state_dtype)
        st = dict(dtype=torch.bfloat16 if state_dtype == "bf16" else torch.float32, device=dev)
        if W0 is None:
            self.W = torch.zeros(m, n, **st)
        else:
            self.W = torch.as_tensor(W0).to(**st).contiguous().clone()
        # left projector P (m x r) with r x n moments, or a right projector
        # Q (n x r) with m x r moments
        self.right = right
        pr = n if right else m
        mom = (m, r) if right else (r, n)
        self.P = torch.zeros(pr, r, **f32)
        self.P_bf16 = torch.zeros(pr, r, dtype=torch.int16, device=dev) if with_bf16 else None
        self.exp_avg = torch.zeros(*mom, **st)
        self.exp_avg_sq = torch.zeros(*mom, **st)
        self.mag_avg = torch.zeros(m, self.kb, **f32)
        self.mag_avg_sq = torch.zeros(m, self.kb, **f32)
        nbytes = B.moara_workspace_bytes(m, n, r, block_size)
        self.workspace = torch.zeros(nbytes, dtype=torch.uint8, device=dev)

    def desc(self):
        d = B.moara_module_desc()
        d.m, d.n, d.r = self.m, self.n, self.r
        d.grad_dtype = B.MOARA_DTYPE_BF16 if self.grad_dtype == "bf16" else B.MOARA_DTYPE_F32
        d.W = self.W.data_ptr()
        d.P = self.P.data_ptr()
        d.P_bf16 = self.P_bf16.data_ptr() if self.P_bf16 is not None else None
        d.exp_avg = self.exp_avg.data_ptr()
        d.exp_avg_sq = self.exp_avg_sq.data_ptr()
        d.mag_avg = self.mag_avg.data_ptr()
        d.mag_avg_sq = self.mag_avg_sq.data_ptr()
        d.workspace = self.workspace.data_ptr()
        d.workspace_bytes = self.workspace.numel()
        return d

    def state_tensors(self):
        return {"W": self.W, "P": self.P, "exp_avg": self.exp_avg,
                "exp_avg_sq": self.exp_avg_sq, "mag_avg": self.mag_avg,
                "mag_avg_sq": self.mag_avg_sq}

    def state_dict(self):
        sd = {k: v.detach().clone() for k, v in self.state_tensors().items()}
        if self.P_bf16 is not None:
            sd["P_bf16"] = self.P_bf16.clone()
        return sd

    def load_state_dict(self, sd):
        for k, v in self.state_tensors().items():
            v.copy_(sd[k])
        if self.P_bf16 is not None and "P_bf16" in sd:
            self.P_bf16.copy_(sd["P_bf16"])


def _device_floats(ptr, n, device):
    """A float32 tensor over n floats of library-owned device memory (no copy);
    valid while the owning context lives."""
    class _Iface:
        __cuda_array_interface__ = {"shape": (n,), "typestr": "<f4", "data": (ptr, False), "version": 2}
    with torch.cuda.device(device):
        return torch.as_tensor(_Iface(), device=f"cuda:{device}")


class MoaraGroup:
    """A context plus the modules registered in it."""

    def __init__(self, hp=None, device=0, refresh_workspace_bytes=None, **overrides):
        self.hp = hp if hp is not None else B.moara_default_hparams()
        for k, v in overrides.items():
            setattr(self.hp, k, v)
        self.device = device
        self.ctx = B.moara_create(self.hp, device)
        self.modules = []
        self.ids = []
        self._refresh_ws = None
        self._refresh_ws_request = refresh_workspace_bytes
        self._clip_extra = None
        self._clip_view = _device_floats(B.moara_clip_state(self.ctx), 2, self.device)

    def add(self, m, n, r, grad_dtype="bf16", W0=None):
        buf = ModuleBuffers(m, n, r, self.hp.block_size, grad_dtype,
                            f"cuda:{self.device}", W0=W0,
                            with_bf16=True,
                            state_dtype="bf16" if self.hp.state_dtype == B.MOARA_DTYPE_BF16 else "f32",
                            right=self.hp.proj_rule == B.MOARA_PROJ_SMALLER and m > n)
        mid = B.moara_init_module(self.ctx, buf.desc())
        self.modules.append(buf)
        self.ids.append(mid)
        return mid

    def ensure_refresh_workspace(self):
        need = max(B.moara_refresh_workspace_bytes(self.ctx, b.m, b.n, b.r) for b in self.modules)
        want = max(need, self._refresh_ws_request or 0)
        if self._refresh_ws is None or self._refresh_ws.numel() < want:
            self._refresh_ws = torch.empty(want, dtype=torch.uint8,
                                           device=f"cuda:{self.device}")
            B.moara_set_refresh_workspace(self.ctx, self._refresh_ws.data_ptr(), want)

    def load_projector(self, mid, P, stream=0):
        src = torch.as_tensor(P, dtype=torch.float32).to(f"cuda:{self.device}").contiguous()
        B.moara_load_projector(self.ctx, mid, src.data_ptr(), stream)
        torch.cuda.current_stream(self.device).synchronize() if stream == 0 else None

    def refresh(self, grads, ids=None, stream=0):
        self.ensure_refresh_workspace()
        ids = self.ids if ids is None else ids
        B.moara_refresh_projector(self.ctx, ids, [g.data_ptr() for g in grads], stream)

    def clip_state(self):
        """{total norm, coefficient} of the last clipped step (a 2-float tensor
        view of the context's device array)."""
        return self._clip_view

    def set_clip_extra(self, extra_sq):
        """extra_sq: a one-element float32 device tensor (kept alive here), or None."""
        self._clip_extra = extra_sq
        B.moara_set_clip_extra(self.ctx, 0 if extra_sq is None else extra_sq.data_ptr())

    def alignment(self, grads, ids=None, stream=0):
        """S(W, t) of each module (a float32 tensor on the group's device)."""
        ids = self.ids if ids is None else ids
        out = torch.empty(len(ids), dtype=torch.float32, device=self.device)
        B.moara_alignment(self.ctx, ids, [g.data_ptr() for g in grads], out.data_ptr(), stream)
        return out

    def step(self, grads, t, lr, auto_refresh=False, ids=None, stream=0):
        ids = self.ids if ids is None else ids
        if auto_refresh:
            self.ensure_refresh_workspace()
        B.moara_step_grouped(self.ctx, ids, [g.data_ptr() for g in grads], t, lr,
                             auto_refresh, stream)

    def step_host(self, host_grads, t, lr, auto_refresh=False, ids=None, chunk_bytes=256 << 20,
                  stream=0):
        """Step with gradients in page-locked host tensors (see
        moara_step_grouped_host)."""
        ids = self.ids if ids is None else ids
        if auto_refresh:
            self.ensure_refresh_workspace()
        B.moara_step_grouped_host(self.ctx, ids, [g.data_ptr() for g in host_grads], t, lr,
                                  auto_refresh, chunk_bytes, stream)

    def status(self, stream=0):
        return B.moara_get_device_status(self.ctx, stream)

    def close(self):
        if self.ctx:
            B.moara_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
