"""ZO steps of the synthetic workloads, chained from libzoact C-ABI calls.

One ZO step (Algorithm 2 with one two-sided query) is

    for every adapted linear, in graph order:  zoact_lowrank_proj + zoact_pair_forward (+ glue)
    zoact_loss_pair   -> L+, L-, D, a  (device memory)
    zoact_adam_step   -> C, m, v updated with g = a * Z over all layers

With ``n_queries = q`` the step is the paper's own one-sided form: every
linear is evaluated at q + 1 points in one launch (zoact_multi_forward: the
unperturbed C, then C + mu Z^(j) with mu = eps), zoact_loss_multi gives
L_0..L_q and a_j = (L_j - L_0) / mu, and zoact_adam_step_multi updates C with
g = (1/q) sum_j a_j Z^(j).

with no host synchronisation.  This module only allocates buffers and issues
the calls; every arithmetic step runs in libzoact's kernels.  Layers that read
the same input with the same basis (q/k/v, gate/up after a calibration pass)
share one projection P = X U; a stacked decoder's q, k and v, whose weights
share one buffer, run as one pair forward (zoact_pair_forward_group_rs).

Graph wiring (names follow synth.Workload):
  toy        h = GELU(l1 x) (shared input, GELU fused in the epilogue); y = l2 h
  llama_mlp  h = silu(gate x) * up x  (one gated call, shared input); y = down h
  llama/opt  per decoder layer on input h:
               a = rms(h); q, k, v = Q a, K a, V a
               o = O rms(q + rep(k) + rep(v));  b = rms(o)
               llama: h' = down rms(silu(gate b) * up b)
               opt:   h' = fc2 rms(relu(fc1 b))
             the first layer's q, k, v see the same input for both signs;
             after it, q, k, v are one launch and the mixer reads column views.

Hooks: `capture(name, X)` is called with each linear's input (the + half)
before its pair forward -- Algorithm 1's calibration pass uses it to take the
bases; `on_decoder(L, h)` with the input of decoder L of a stack ([T, d] for
the first, the stacked [n_blocks T, d] after it; the buffer is reused later,
so a hook that keeps it clones it); `flops`, when a list, receives the
algorithmic FLOP count (2 rows d_in d_out, gated x2) of every pair-forward
call, with no events or synchronisation.
"""
import torch

from . import _lib as Z

_TORCH = {"fp32": torch.float32, "bf16": torch.bfloat16, "fp16": torch.float16}


class AdaptedLinear:
    def __init__(self, name, W, U, layer_id, offset, r, w_scales=None, wtype=None, d_in=None):
        self.name = name
        self.W = W
        self.U = U
        self.w_scales = w_scales
        self.layer_id = int(layer_id)
        self.offset = int(offset)
        self.r = int(r)
        self.wtype = Z.TORCH_DT[W.dtype] if wtype is None else wtype
        self.d_out = W.shape[0]
        self.d_in = int(d_in) if d_in is not None else W.shape[1]
        self.layer = None

    def bind(self, C):
        view = C[self.offset:self.offset + self.d_out * self.r]
        self.layer = Z.make_layer(self.W, self.U, view, self.layer_id, w_scales=self.w_scales, wtype=self.wtype,
                                  d_in=self.d_in)


class ZOStep:
    """Holds frozen weights/bases, the coefficient arenas and activation buffers."""

    def __init__(self, ctx, kind, linears, T, act_dtype, eps=1e-3, lr=1e-4, beta1=0.9, beta2=0.999,
                 adam_eps=1e-8, n_heads=32, n_kv_heads=8, head_dim=128, n_queries=None):
        self.ctx = ctx
        self.kind = kind
        self.T = int(T)
        self.dtype = _TORCH[act_dtype] if isinstance(act_dtype, str) else act_dtype
        self.eps, self.lr, self.beta1, self.beta2, self.adam_eps = eps, lr, beta1, beta2, adam_eps
        self.n_rep = n_heads // n_kv_heads if kind == "llama" else 1
        self.head_dim = head_dim
        self.linears = linears                      # list of AdaptedLinear, forward order
        self.by_name = {l.name: l for l in linears}
        # stacks: each decoder's q, k and v read one input; their weights share one buffer so that, on stacked
        # rows, one launch can run all three (zoact_pair_forward_group_rs)
        self.groups = ([[f"{L}.q", f"{L}.k", f"{L}.v"] for L in range(len(linears) // (7 if kind == "llama" else 6))]
                       if kind in ("llama", "opt") else [])
        self._nogroup = set()
        colocate_weights([[self.by_name[n] for n in g] for g in self.groups])
        dev = linears[0].W.device
        n = max(l.offset + l.d_out * l.r for l in linears)
        n = (n + 3) // 4 * 4
        self.C = torch.zeros(n, dtype=torch.float32, device=dev)
        self.m = torch.zeros_like(self.C)
        self.v = torch.zeros_like(self.C)
        for l in linears:
            l.bind(self.C)
        self.blocks = [(l.offset, l.d_out, l.r, l.layer_id) for l in linears]
        self.n_queries = n_queries                  # None: two-sided pair; q: one-sided with q queries
        self.nb = 2 if n_queries is None else int(n_queries) + 1
        # two loss vectors, alternated by loss(): a step's result can be read back (on another stream) while
        # the next step writes the other one
        n_loss = 4 if n_queries is None else 2 * self.nb - 1
        self._loss_bufs = [torch.zeros(n_loss, dtype=torch.float64, device=dev) for _ in range(2)]
        self._loss_i = 0
        self._bufs = {}
        self._pcache = {}
        self.device = dev
        self.capture = None
        self.on_decoder = None
        self.flops = None
        # forward_loss fuses the loss pair into the last linear when set; off by default: the fused epilogue
        # lengthens the Llama-3-8B down launch by more than the separate loss launch takes
        self.fuse_loss = False
        # stacks: RMS normalisations as row scales of the pair forwards where the library applies them
        self.row_scales = True
        self._utc = {}
        self.prepare_bases()

    def prepare_bases(self):
        """The frozen bases in the tensor-core projection's operand form, once per distinct U
        (16-bit activations only).  Call again after changing a U in place."""
        self._utc = {}
        if self.dtype not in (torch.bfloat16, torch.float16):
            return
        for l in self.linears:
            key = l.U.data_ptr()
            if key in self._utc:
                continue
            t = torch.empty(Z.zoact_basis_prepared_bytes(l.d_in, l.r), dtype=torch.uint8, device=self.device)
            Z.zoact_basis_prepare(self.ctx, l.U, Z.TORCH_DT[self.dtype], t)
            self._utc[key] = t

    # ---- buffers ----
    def buf(self, key, rows, cols, dtype=None):
        dtype = self.dtype if dtype is None else dtype
        t = self._bufs.get(key)
        if t is None or t.shape != (rows, cols) or t.dtype != dtype:
            t = torch.empty(rows, cols, dtype=dtype, device=self.device)
            self._bufs[key] = t
        return t

    def _wrote(self, t):
        """A buffer was rewritten: projections of it are stale."""
        for slot in [s for s, (key, _) in self._pcache.items() if key[0] == t.data_ptr()]:
            del self._pcache[slot]

    def _proj(self, lin, X, slot):
        key = (X.data_ptr(), X.shape[0], lin.U.data_ptr())
        hit = self._pcache.get(slot)
        if hit is not None and hit[0] == key:
            return hit[1]
        for s, (k, P) in self._pcache.items():      # same input and basis already projected
            if k == key:
                self._pcache[slot] = (key, P)
                return P
        P = self.buf(f"P{slot}", X.shape[0], lin.r, torch.float32)
        utc = self._utc.get(lin.U.data_ptr())
        if utc is not None and X.dtype == self.dtype:
            Z.zoact_lowrank_proj_prepared(self.ctx, X, utc, lin.r, P)
        else:
            Z.zoact_lowrank_proj(self.ctx, X, lin.U, P)
        self._pcache[slot] = (key, P)
        return P

    def _counted(self, fn, flops):
        fn()
        if self.flops is not None:
            self.flops.append(flops)

    def query_ids(self, query):
        """The q Philox query ids of one one-sided step."""
        return [int(query) * self.n_queries + j for j in range(self.n_queries)]

    def points(self, query):
        return Z.one_sided_blocks(self.eps, self.query_ids(query))

    def _sums(self, key, d_out, rows):
        """The out_sumsq array of a pair forward with row scales, and the 1/rms vector made from it."""
        return (self.buf(f"ss_{key}", Z.rowscale_parts(d_out), rows, torch.float32),
                self.buf(f"inv_{key}", 1, rows, torch.float32).view(rows))

    def pair(self, name, X, shared, seed, query, out_key, act=Z.ACT_NONE, fused=None, in_scale=None, sums=False):
        """fused = (target, out): the last linear with the loss pair fused (zoact_pair_forward_loss); returns None
        when that ran, else (the launch does not qualify) the output as without it.

        Row scales (stacked rows): in_scale [rows] is 1/rms of X's rows, applied to the output rows
        (X is the unnormalised input).  sums=True returns (Y, 1/rms of Y's rows) from the partial sums of squares
        the launch writes, or (Y, None) where the launch cannot write them (the caller then normalises Y)."""
        l = self.by_name[name]
        if self.capture is not None:
            self.capture(name, X[:self.T])
        P = self._proj(l, X, 0)
        flops = 2.0 * X.shape[0] * l.d_in * l.d_out
        if in_scale is not None or sums:
            Y = self.buf(out_key, self.nb * self.T, l.d_out)
            ss, inv = self._sums(out_key, l.d_out, Y.shape[0]) if sums else (None, None)
            if self.n_queries is None:
                fn = lambda: Z.zoact_pair_forward_rs(self.ctx, l.layer, X, self.T, shared, self.eps, seed, query, Y,
                                                     P=P, act=act, in_scale=in_scale, out_sumsq=ss)
            else:
                fn = lambda: Z.zoact_multi_forward_rs(self.ctx, l.layer, X, self.T, shared, self.points(query), seed,
                                                      Y, P=P, act=act, in_scale=in_scale, out_sumsq=ss)
            try:
                self._counted(fn, flops)
            except Z.ZoactError as e:
                if e.status != Z.ZOACT_ERR_UNSUPPORTED or in_scale is not None:
                    raise
                Y = self.pair(name, X, shared, seed, query, out_key, act)
                return (Y, None) if sums else Y
            self._wrote(Y)
            if sums:
                Z.zoact_rms_scale(self.ctx, ss, l.d_out, inv)
                return Y, inv
            return Y
        if fused is not None and self.n_queries is None and not shared:
            target, out = fused
            try:
                self._counted(lambda: Z.zoact_pair_forward_loss(self.ctx, l.layer, X, self.T, self.eps, seed, query,
                                                                Z.TORCH_DT[self.dtype], out, target=target, P=P,
                                                                act=act), flops)
                return None
            except Z.ZoactError as e:
                if e.status != Z.ZOACT_ERR_UNSUPPORTED:
                    raise
        Y = self.buf(out_key, self.nb * self.T, l.d_out)
        if self.n_queries is None:
            fn = lambda: Z.zoact_pair_forward(self.ctx, l.layer, X, self.T, shared, self.eps, seed, query, Y, P=P,
                                              act=act)
        else:
            fn = lambda: Z.zoact_multi_forward(self.ctx, l.layer, X, self.T, shared, self.points(query), seed, Y,
                                               P=P, act=act)
        self._counted(fn, flops)
        self._wrote(Y)
        return Y

    def gated(self, gname, uname, X, shared, seed, query, out_key, in_scale=None, sums=False):
        """silu(gate X) * up X; row scales as in pair()."""
        g, u = self.by_name[gname], self.by_name[uname]
        if self.capture is not None:
            self.capture(gname, X[:self.T])
            self.capture(uname, X[:self.T])
        Pg = self._proj(g, X, 0)
        Pu = self._proj(u, X, 1)
        H = self.buf(out_key, self.nb * self.T, g.d_out)
        flops = 2.0 * X.shape[0] * g.d_in * g.d_out * 2
        if in_scale is not None or sums:
            ss, inv = self._sums(out_key, g.d_out, H.shape[0]) if sums else (None, None)
            if self.n_queries is None:
                fn = lambda: Z.zoact_pair_forward_gated_rs(self.ctx, g.layer, u.layer, X, self.T, shared, self.eps,
                                                           seed, query, H, P_gate=Pg, P_up=Pu, in_scale=in_scale,
                                                           out_sumsq=ss)
            else:
                fn = lambda: Z.zoact_multi_forward_gated_rs(self.ctx, g.layer, u.layer, X, self.T, shared,
                                                            self.points(query), seed, H, P_gate=Pg, P_up=Pu,
                                                            in_scale=in_scale, out_sumsq=ss)
            try:
                self._counted(fn, flops)
            except Z.ZoactError as e:
                if e.status != Z.ZOACT_ERR_UNSUPPORTED or in_scale is not None:
                    raise
                H = self.gated(gname, uname, X, shared, seed, query, out_key)
                return (H, None) if sums else H
            self._wrote(H)
            if sums:
                Z.zoact_rms_scale(self.ctx, ss, g.d_out, inv)
                return H, inv
            return H
        if self.n_queries is None:
            fn = lambda: Z.zoact_pair_forward_gated(self.ctx, g.layer, u.layer, X, self.T, shared, self.eps, seed,
                                                    query, H, P_gate=Pg, P_up=Pu)
        else:
            fn = lambda: Z.zoact_multi_forward_gated(self.ctx, g.layer, u.layer, X, self.T, shared,
                                                     self.points(query), seed, H, P_gate=Pg, P_up=Pu)
        self._counted(fn, flops)
        self._wrote(H)
        return H

    def _groupable(self, ls):
        """Whether the library may run these linears as one launch: one basis, one weight type and width, and
        weight (and INT4 scale) rows that follow one another in memory."""
        l0 = ls[0]
        if self.dtype not in (torch.bfloat16, torch.float16):
            return False
        if any(l.U.data_ptr() != l0.U.data_ptr() or l.d_in != l0.d_in or l.r != l0.r or l.wtype != l0.wtype
               for l in ls):
            return False
        rows = 0
        for l in ls:
            if l.W.data_ptr() != l0.W.data_ptr() + rows * l0.W.stride(0) * l0.W.element_size():
                return False
            if l.w_scales is not None and (l0.w_scales is None or l.w_scales.data_ptr() != l0.w_scales.data_ptr() +
                                           rows * l0.w_scales.stride(0) * l0.w_scales.element_size()):
                return False
            rows += l.d_out
        return True

    def pair_group(self, names, X, seed, query, out_key, in_scale=None):
        """Linears that read X (stacked rows) as one pair forward (zoact_pair_forward_group_rs /
        zoact_multi_forward_group_rs).  Returns their outputs, column views of one [rows, sum d_out] buffer, or
        None where the library cannot run them as one launch (it then launched nothing; the caller runs them one
        by one)."""
        key = tuple(names)
        ls = [self.by_name[n] for n in names]
        if key in self._nogroup or not self._groupable(ls):
            self._nogroup.add(key)
            return None
        P = self._proj(ls[0], X, 0)
        dsum = sum(l.d_out for l in ls)
        Y = self.buf(out_key, self.nb * self.T, dsum)
        layers = [l.layer for l in ls]
        if self.n_queries is None:
            fn = lambda: Z.zoact_pair_forward_group_rs(self.ctx, layers, X, self.T, self.eps, seed, query, Y, P=P,
                                                       in_scale=in_scale)
        else:
            fn = lambda: Z.zoact_multi_forward_group_rs(self.ctx, layers, X, self.T, self.points(query), seed, Y, P=P,
                                                        in_scale=in_scale)
        try:
            self._counted(fn, 2.0 * X.shape[0] * ls[0].d_in * dsum)
        except Z.ZoactError as e:
            if e.status != Z.ZOACT_ERR_UNSUPPORTED:
                raise
            self._nogroup.add(key)
            return None
        self._wrote(Y)
        outs, c = [], 0
        for l in ls:
            outs.append(Y[:, c:c + l.d_out])
            c += l.d_out
        return outs

    def _glue_rms(self, X, key):
        Y = self.buf(key, X.shape[0], X.shape[1])
        Z.zoact_rms_norm(self.ctx, X, Y)
        self._wrote(Y)
        return Y

    # ---- forward graphs ----
    def forward(self, x, seed, query, fused=None):
        """The graph's output; with fused = (target, out) the last linear writes the loss pair into out instead
        where it can (then None is returned)."""
        self._pcache = {}
        if self.kind == "toy":
            h = self.pair("l1", x, True, seed, query, "h", act=Z.ACT_GELU)
            return self.pair("l2", h, False, seed, query, "y", fused=fused)
        if self.kind == "llama_mlp":
            H = self.gated("gate", "up", x, True, seed, query, "h")
            return self.pair("down", H, False, seed, query, "y", fused=fused)
        return self._stack(x, seed, query, fused)

    def forward_loss(self, x, target, seed, query):
        """forward() and then loss(); with fuse_loss set, the last linear's pair forward and the loss pair run
        as one launch (zoact_pair_forward_loss, two-sided only) when it qualifies.  Returns the device loss
        vector."""
        if self.n_queries is not None or not self.fuse_loss:
            return self.loss(self.forward(x, seed, query), target)
        self._loss_i ^= 1
        Y = self.forward(x, seed, query, fused=(target, self.loss_out))
        if Y is not None:                  # not fused: the separate loss pair (which takes the same vector)
            self._loss_i ^= 1
            self.loss(Y, target)
        return self.loss_out

    def _stack(self, x, seed, query, fused=None):
        """The stack's decoders.  With row scales (outside calibration, where the library applies them) the RMS normalisations of o, of the MLP hidden and of each decoder's output are not separate passes:
        the producing pair forward writes per-row sums of squares, zoact_rms_scale turns them into 1/rms, and the
        consuming pair forward scales its rows (include/zoact.h, row scales).  Otherwise, and wherever a launch
        cannot apply them, the normalised tensor is written by zoact_rms_norm first."""
        T = self.T
        n_dec = len(self.linears) // (7 if self.kind == "llama" else 6)
        rs = self.row_scales and self.capture is None
        h, inv_h = x, None
        shared = True
        for L in range(n_dec):
            if self.on_decoder is not None:
                self.on_decoder(L, h)
            last = L == n_dec - 1
            rows = T if shared else self.nb * T
            if inv_h is None:
                a = self._glue_rms(h, f"a{rows}")
                q = self.pair(f"{L}.q", a, shared, seed, query, "q")
                k = self.pair(f"{L}.k", a, shared, seed, query, "k")
                v = self.pair(f"{L}.v", a, shared, seed, query, "v")
            else:
                qkv = self.pair_group([f"{L}.q", f"{L}.k", f"{L}.v"], h, seed, query, "qkv", in_scale=inv_h)
                if qkv is not None:
                    q, k, v = qkv
                else:
                    q = self.pair(f"{L}.q", h, False, seed, query, "q", in_scale=inv_h)
                    k = self.pair(f"{L}.k", h, False, seed, query, "k", in_scale=inv_h)
                    v = self.pair(f"{L}.v", h, False, seed, query, "v", in_scale=inv_h)
            shared = False
            mix = self.buf("mix", self.nb * T, q.shape[1])
            Z.zoact_mix_rms(self.ctx, q, k, v, mix, self.n_rep if self.kind == "llama" else 1, self.head_dim)
            self._wrote(mix)
            inv_o = None
            if rs:
                o, inv_o = self.pair(f"{L}.o", mix, False, seed, query, "o", sums=True)
            else:
                o = self.pair(f"{L}.o", mix, False, seed, query, "o")
            b, sb = (o, inv_o) if inv_o is not None else (self._glue_rms(o, "b"), None)
            out_key = "h" if L % 2 == 0 else "h2"
            if self.kind == "llama":
                inv_m = None
                if sb is not None:
                    H, inv_m = self.gated(f"{L}.gate", f"{L}.up", b, False, seed, query, "hmlp", in_scale=sb, sums=True)
                else:
                    H = self.gated(f"{L}.gate", f"{L}.up", b, False, seed, query, "hmlp")
                m, sm, lname = (H, inv_m, f"{L}.down") if inv_m is not None else (self._glue_rms(H, "hmlp_n"), None,
                                                                                  f"{L}.down")
            else:
                inv_f = None
                if sb is not None:
                    f, inv_f = self.pair(f"{L}.fc1", b, False, seed, query, "f", act=Z.ACT_RELU, in_scale=sb, sums=True)
                else:
                    f = self.pair(f"{L}.fc1", b, False, seed, query, "f", act=Z.ACT_RELU)
                m, sm, lname = (f, inv_f, f"{L}.fc2") if inv_f is not None else (self._glue_rms(f, "f_n"), None,
                                                                                 f"{L}.fc2")
            inv_h = None
            if sm is not None and last and fused is not None:
                # the fused loss pair takes a normalised input: normalise it explicitly for that launch
                m, sm = self._glue_rms(m, "hmlp_n" if self.kind == "llama" else "f_n"), None
            if sm is not None:
                if last:
                    h = self.pair(lname, m, False, seed, query, out_key, in_scale=sm)
                else:
                    h, inv_h = self.pair(lname, m, False, seed, query, out_key, in_scale=sm, sums=True)
            else:
                h = self.pair(lname, m, False, seed, query, out_key, fused=fused if last else None)
        return h

    # ---- loss and update ----
    @property
    def loss_out(self):
        """The device loss vector of the latest loss() call (update() reads it)."""
        return self._loss_bufs[self._loss_i]

    def loss(self, Y, target):
        """Two-sided: [L+, L-, D, a].  One-sided: [L_0 .. L_q, a_1 .. a_q].  Each call writes the loss vector
        the previous call did not, so the previous step's vector stays valid until the call after next."""
        self._loss_i ^= 1
        if self.n_queries is None:
            Z.zoact_loss_pair(self.ctx, Y, self.T, self.eps, self.loss_out, target=target)
        else:
            Z.zoact_loss_multi(self.ctx, Y, self.T, self.nb, self.eps, self.loss_out, target=target)
        return self.loss_out

    def update(self, step, seed, query, lr=None):
        lr = self.lr if lr is None else lr
        if self.n_queries is None:
            Z.zoact_adam_step(self.ctx, self.C, self.m, self.v, self.blocks, self.loss_out, lr, self.beta1,
                              self.beta2, self.adam_eps, step, seed, query)
        else:
            Z.zoact_adam_step_multi(self.ctx, self.C, self.m, self.v, self.blocks, self.loss_out[self.nb:],
                                    self.query_ids(query), lr, self.beta1, self.beta2, self.adam_eps, step, seed)

    def step(self, x, target, step, seed, query, lr=None):
        """One ZO step: pair forwards, loss pair, Adam.  Returns the device loss tensor [L+, L-, D, a]."""
        Y = self.forward(x, seed, query)
        self.loss(Y, target)
        self.update(step, seed, query, lr)
        return self.loss_out


class HostFeeder:
    """Runs ZO steps on batches of PINNED host tensors, overlapping each batch's host-to-device copy (on a
    side stream, into one of two device buffer sets) with the previous step's compute.

    The device buffers, the side stream and the events are made once, here, for batches shaped like
    `example` (a tuple of host tensors, e.g. (x, target) or (x,)); run() then only issues copies, waits and
    steps, so a timed region around run() holds no allocation or stream creation.
    """

    def __init__(self, example, device=None):
        self.main = torch.cuda.current_stream(device)
        self.side = torch.cuda.Stream(device=self.main.device)
        self.shapes = [(h.shape, h.dtype) for h in example]
        self.bufs = [[torch.empty(sh, dtype=dt, device=self.main.device) for sh, dt in self.shapes]
                     for _ in range(2)]
        self.copied = [torch.cuda.Event(), torch.cuda.Event()]
        self.free = [torch.cuda.Event(), torch.cuda.Event()]
        self.read = [torch.cuda.Event(), torch.cuda.Event()]   # loss vector of step i read back (parity i % 2)

    def run(self, batches, step_fn, out_host):
        """One ZO step per batch.  step_fn(device_tensors, i) issues step i on the feeder's main stream (torch's
        current stream when the feeder was made) and returns its device loss vector, which is copied into
        out_host[i] (pinned) on the side stream once step i has finished, so no copy sits between two steps'
        kernels.  That needs consecutive steps to return different loss vectors (ZOStep.loss alternates two;
        step i + 2 rewrites step i's only after its read-back): a step function that returns the same vector
        twice in a row raises ValueError.  Returns after issuing all work (no synchronisation)."""
        if not batches:
            return
        for b in batches:
            if [(h.shape, h.dtype) for h in b] != self.shapes:
                raise ValueError("HostFeeder.run: every batch must match the feeder's shapes and dtypes")
        main, side, bufs = self.main, self.side, self.bufs
        copied, free, read = self.copied, self.free, self.read
        prev_ptr = None

        def fetch(i):
            b = i % 2
            side.wait_stream(main) if i < 2 else side.wait_event(free[b])   # buffer b no longer read
            with torch.cuda.stream(side):
                for d, h in zip(bufs[b], batches[i]):
                    d.copy_(h, non_blocking=True)
                copied[b].record(side)

        fetch(0)
        for i in range(len(batches)):
            if i + 1 < len(batches):
                fetch(i + 1)
            b = i % 2
            main.wait_event(copied[b])
            if i >= 2:
                main.wait_event(read[b])                 # step i - 2's loss vector, which step i rewrites, is read
            with torch.cuda.stream(main):
                out = step_fn(bufs[b], i)
            if out.data_ptr() == prev_ptr:
                raise ValueError("run_from_host: consecutive steps must return different loss vectors")
            prev_ptr = out.data_ptr()
            free[b].record(main)
            side.wait_event(free[b])
            with torch.cuda.stream(side):
                out_host[i].copy_(out, non_blocking=True)
                read[b].record(side)


def run_from_host(batches, step_fn, out_host):
    """HostFeeder(batches[0]).run(batches, step_fn, out_host): the feeder's buffers are made on every call;
    keep a HostFeeder to reuse them."""
    if not batches:
        return
    HostFeeder(batches[0]).run(batches, step_fn, out_host)


def coefficient_offsets(specs, r):
    """Offsets (multiples of 4) of each layer's [d_out, r] block in the flat arena."""
    offs, cur = [], 0
    for s in specs:
        offs.append(cur)
        cur += (s.d_out * r + 3) // 4 * 4
    return offs


def colocate_weights(groups):
    """Put the weights of each group of AdaptedLinears (linears that read one input, e.g. a decoder's q, k and
    v) in one buffer, rows in group order, so that the library can run the group as one launch; INT4 scales
    likewise.  Values are unchanged; a group already laid out so is left alone.  Call before binding."""
    for ls in groups:
        if len(ls) < 2:
            continue
        rows, ok = 0, True
        for l in ls:
            ok = ok and l.W.data_ptr() == ls[0].W.data_ptr() + rows * ls[0].W.stride(0) * ls[0].W.element_size()
            rows += l.d_out
        if ok:
            continue
        W = torch.cat([l.W for l in ls])
        S = torch.cat([l.w_scales for l in ls]) if ls[0].w_scales is not None else None
        c = 0
        for l in ls:
            l.W = W[c:c + l.d_out]
            if S is not None:
                l.w_scales = S[c:c + l.d_out]
            c += l.d_out


def calibrate_bases(ctx, step_cal, x_cal, r, oversample=16, n_iter=8, seed=0):
    """Algorithm 1: one calibration forward pass of the base model (C = 0, eps = 0) on x_cal,
    and each layer's basis U = top-r right singular vectors of its input, written in place.

    step_cal is a ZOStep over the same AdaptedLinear objects with T = len(x_cal); layers whose
    inputs are the same tensor (q/k/v, gate/up) have the same basis by definition: they get one
    basis computation and share its tensor, so later steps project their common input once (and a
    gated pair sees one projection).  ZOSteps built after this call bind the shared tensors.
    """
    last = {}

    def cap(name, X):
        lin = step_cal.by_name[name]
        key = (X.data_ptr(), X.shape[0])
        if last.get("key") == key:
            lin.U = last["U"]
            lin.bind(step_cal.C)
            return
        Z.zoact_basis_init(ctx, X.contiguous(), r, lin.U, oversample=oversample, n_iter=n_iter,
                           seed=seed + lin.layer_id)
        last["key"], last["U"] = key, lin.U

    step_cal.capture = cap
    step_cal.C.zero_()
    eps = step_cal.eps
    step_cal.eps = 0.0
    step_cal.forward(x_cal, 0, 0)
    step_cal.eps = eps
    step_cal.capture = None
