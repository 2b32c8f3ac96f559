"""One OrderMoE MoE layer on the GPU: device buffers from torch, every step
through the C ABI (route_select -> dispatch -> expert_ffn -> combine)."""
import torch

from . import binding as B


class MoELayer:
    """Holds a layer's weights, tables and scratch for up to T_max tokens."""

    def __init__(self, W_r, W1, W3, W2, tables, k, T_max, renorm=1, device=None):
        self.device = device or W1.device
        self.W_r, self.W1, self.W3, self.W2 = W_r, W1, W3, W2
        self.E, self.dff, self.d = W1.shape
        self.k, self.renorm, self.tables = k, renorm, tables
        self.T_max = T_max
        R = T_max * k
        dev = self.device
        self.logits = torch.empty(T_max, self.E, dtype=torch.float32, device=dev)
        self.topk_idx = torch.empty(T_max, k, dtype=torch.int32, device=dev)
        self.topk_w = torch.empty(T_max, k, dtype=torch.float32, device=dev)
        self.chosen = torch.empty(T_max, k, dtype=torch.int32, device=dev)
        self.server = torch.empty(T_max, k, dtype=torch.uint8, device=dev)
        self.kind = torch.empty(T_max, k, dtype=torch.uint8, device=dev)
        self.counters = torch.zeros(4, dtype=torch.int32, device=dev)
        self.offsets = torch.empty(self.E + 1, dtype=torch.int32, device=dev)
        self.row_token = torch.empty(R, dtype=torch.int32, device=dev)
        self.row_of = torch.empty(T_max, k, dtype=torch.int32, device=dev)
        self.X_perm = torch.empty(R, self.d, dtype=torch.bfloat16, device=dev)
        self.H = torch.empty(R, self.dff, dtype=torch.bfloat16, device=dev)
        self.Y_perm = torch.empty(R, self.d, dtype=torch.bfloat16, device=dev)
        ws = B.ordermoe_dispatch_workspace_bytes(T_max, k, self.E)
        self.ws = torch.empty(ws, dtype=torch.uint8, device=dev)

    def forward(self, X, home, loc, qhat, y, T=None, logits_in=None, stream=None):
        """y[:T] = MoE(X[:T]); loc/qhat are updated in place (Eq. 44)."""
        T = X.shape[0] if T is None else T
        assert T <= self.T_max
        R = T * self.k
        B.ordermoe_route_select(X, self.W_r, logits_in, T, self.E, self.d, self.k, self.renorm,
                                self.tables, home, loc, qhat, self.logits, self.topk_idx,
                                self.topk_w, self.chosen, self.server, self.kind, self.counters,
                                stream)
        B.ordermoe_dispatch(self.chosen, X, T, self.k, self.E, self.d, self.offsets,
                            self.row_token, self.row_of, self.X_perm, self.ws, stream)
        B.ordermoe_expert_ffn(self.X_perm, self.offsets, R, self.W1, self.W3, self.W2, self.E,
                              self.d, self.dff, self.H, self.Y_perm, stream)
        B.ordermoe_combine(self.Y_perm, self.row_of, self.topk_w, T, self.k, self.d, y, stream)
        return y

    def forward_residual(self, x, h, home, loc, qhat, h_out, x_out, T=None, eps=B.NORM_EPS,
                         stream=None):
        """One layer of a stack on the residual map: the layer runs on x
        (= RMSNorm(h)), then h_out = h + y and x_out = RMSNorm(h_out), the next
        layer's inputs. Router logits, decisions and the permutation stay in
        this object's buffers."""
        T = x.shape[0] if T is None else T
        assert T <= self.T_max
        R = T * self.k
        B.ordermoe_route_select(x, self.W_r, None, T, self.E, self.d, self.k, self.renorm,
                                self.tables, home, loc, qhat, self.logits, self.topk_idx,
                                self.topk_w, self.chosen, self.server, self.kind, self.counters,
                                stream)
        B.ordermoe_dispatch(self.chosen, x, T, self.k, self.E, self.d, self.offsets,
                            self.row_token, self.row_of, self.X_perm, self.ws, stream)
        B.ordermoe_expert_ffn(self.X_perm, self.offsets, R, self.W1, self.W3, self.W2, self.E,
                              self.d, self.dff, self.H, self.Y_perm, stream)
        B.ordermoe_combine_residual_norm(self.Y_perm, self.row_of, self.topk_w, h, T, self.k,
                                         self.d, eps, h_out, x_out, stream)
        return h_out, x_out


def build_tables(sim, group, placement, theta, qbar, sp, device, out=None):
    """Device tables for one layer from host arrays (sim, group, placement) and
    server parameters sp (synth.ServerParams); written into `out` (a uint8
    device tensor, e.g. one slice of a stack of layers' tables) when given."""
    E = sim.shape[0]; M = placement.shape[0]
    t = out if out is not None else torch.zeros(B.ordermoe_tables_bytes(E, M), dtype=torch.uint8,
                                                device=device)
    f = lambda a, dt: torch.as_tensor(a).to(device=device, dtype=dt).contiguous()
    B.ordermoe_build_tables(f(sim, torch.float32), f(group, torch.int32), f(placement, torch.uint8),
                            theta, qbar, f(sp.F, torch.float64), f(sp.B, torch.float64),
                            f(sp.tau, torch.float64), sp.z, sp.c, sp.omega_T, sp.omega_Q, t)
    return t


class LayerStack:
    """L MoE layers run through ordermoe_layer_forward with the token state
    (location, accumulated loss; Eqs. 36 and 44) carried from layer to layer."""

    def __init__(self, layers, tables, k, T_max, device, H=1, stride=0, P=None):
        """layers: dicts with W_r, W1, W3, W2 (device bf16). tables: a list of
        per-layer device buffers, or (for look-ahead, H > 1) one device buffer
        holding all layers' tables `stride` bytes apart; P [L-1, E, E] the
        transition matrices. Layer l looks min(H, L - l) - 1 layers ahead."""
        E, dff, d = layers[0]["W1"].shape
        L = len(layers)
        self.scratch = torch.empty(B.ordermoe_layer_scratch_bytes(T_max, E, d, dff, k),
                                   dtype=torch.uint8, device=device)
        self.descs = []
        for l, lay in enumerate(layers):
            if isinstance(tables, torch.Tensor):
                t = tables[l * stride:]
                Hl = min(H, L - l)
                Pl = P[l:l + Hl - 1].contiguous() if Hl > 1 else None
            else:
                t, Hl, Pl = tables[l], 1, None
            self.descs.append(B.make_layer_desc(T_max, lay["W_r"], lay["W1"], lay["W3"], lay["W2"],
                                                t, k, self.scratch, lookahead_H=Hl,
                                                tables_stride=stride, P=Pl))
        self.d, self.T_max = d, T_max

    def step(self, X_layers, home, loc, qhat, y_layers, counters=None, stream=None):
        """Layer l reads X_layers[l] and writes y_layers[l]; loc/qhat carry the
        trajectory (set loc = home, qhat = 0 before the first layer)."""
        T = X_layers[0].shape[0]
        for desc, X, y in zip(self.descs, X_layers, y_layers):
            B.ordermoe_layer_forward(desc, T, X, home, loc, qhat, y, counters, 0, stream)

    def step_residual(self, hs, xs, home, loc, qhat, counters=None, logits=None,
                      eps=B.NORM_EPS, stream=None):
        """One pass over the stack on the residual map: xs[0] = RMSNorm(hs[0]),
        then layer l runs on xs[l] and writes hs[l + 1] = hs[l] + y_l and
        xs[l + 1] = RMSNorm(hs[l + 1]). hs, xs: L + 1 device buffers [T, d]
        bf16 (hs[0] is the input); logits: optional [L, T, E] f32 receiving each
        layer's router logits (layer-major)."""
        T = hs[0].shape[0]
        B.ordermoe_rmsnorm(hs[0], T, self.d, eps, xs[0], stream)
        for l, desc in enumerate(self.descs):
            B.ordermoe_layer_forward_residual(desc, T, xs[l], hs[l], home, loc, qhat, eps,
                                              hs[l + 1], xs[l + 1],
                                              None if logits is None else logits[l], counters,
                                              stream)

    def capture(self, X_layers, home, loc, qhat, y_layers, counters=None, prologue=None):
        """Records one step (every layer's kernels, after the optional prologue,
        e.g. resetting loc and qhat) as a CUDA graph over these buffers, so a
        step is one graph launch. Returns the torch.cuda.CUDAGraph; replay()
        runs the step on the buffers' current contents."""
        return self._capture(lambda s: self.step(X_layers, home, loc, qhat, y_layers, counters,
                                                 stream=s), prologue)

    def capture_residual(self, hs, xs, home, loc, qhat, counters=None, prologue=None,
                         eps=B.NORM_EPS):
        """capture() of step_residual over these buffers."""
        return self._capture(lambda s: self.step_residual(hs, xs, home, loc, qhat, counters,
                                                          eps=eps, stream=s), prologue)

    def _capture(self, body, prologue):
        s = torch.cuda.Stream(device=self.scratch.device)
        s.wait_stream(torch.cuda.current_stream(self.scratch.device))
        with torch.cuda.stream(s):  # one eager step first: per-device set-up outside the capture
            if prologue is not None:
                prologue()
            body(s)
        torch.cuda.current_stream(self.scratch.device).wait_stream(s)
        torch.cuda.synchronize(self.scratch.device)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            if prologue is not None:
                prologue()
            body(s)
        return g


def exact_tables(E, M, device):
    """Selection tables that keep every routed expert (no substitutes: the
    threshold 2 exceeds any cosine; every expert on every server): the
    unmodified model, which a stack's calibration pass runs."""
    sim = torch.eye(E, dtype=torch.float32, device=device)
    group = torch.arange(E, dtype=torch.int32, device=device)
    x = torch.ones(M, E, dtype=torch.uint8, device=device)
    t = torch.zeros(B.ordermoe_tables_bytes(E, M), dtype=torch.uint8, device=device)
    f64 = lambda *sh: torch.ones(*sh, dtype=torch.float64, device=device)
    B.ordermoe_build_tables(sim, group, x, 2.0, 1.0, f64(M), f64(M, M), f64(M, M) * 0, 1.0, 1.0,
                            0.5, 0.5, t)
    return t


def calibrate_stack(layers, h_cal, k_freq, M, eps=B.NORM_EPS):
    """Offline statistics of a stack on the residual map (Section III-B on the
    representations each layer actually sees): the calibration tokens h_cal
    [N, d] pass through the unmodified stack (every routed expert kept), and
    layer l's similarity and counts (Eqs. 3-5) are taken over its own inputs
    x_l = RMSNorm(h_l), its transitions (Eq. 41) between the router logits of
    consecutive layers along the same pass. Returns a dict: sim [L, E, E],
    counts [L, E], P [L-1, E, E], tcount [L-1, E, E], logits [L, N, E] (f32
    device), hs and xs (the L + 1 residual states and normalised inputs)."""
    dev = h_cal.device
    N, d = h_cal.shape
    L = len(layers)
    E = layers[0]["W1"].shape[0]
    tab = exact_tables(E, M, dev)
    stack = LayerStack(layers, [tab] * L, k_freq, N, dev)
    hs = [h_cal] + [torch.empty_like(h_cal) for _ in range(L)]
    xs = [torch.empty_like(h_cal) for _ in range(L + 1)]
    home = torch.zeros(N, dtype=torch.uint8, device=dev)
    logits = torch.empty(L, N, E, dtype=torch.float32, device=dev)
    stack.step_residual(hs, xs, home, None, None, logits=logits, eps=eps)
    sim = torch.empty(L, E, E, dtype=torch.float32, device=dev)
    counts = torch.empty(L, E, dtype=torch.int32, device=dev)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(1, E, N), dtype=torch.uint8, device=dev)
    for l in range(L):
        B.ordermoe_similarity_no_logits(layers[l]["W_r"], xs[l], 1, E, d, N, k_freq, sim[l],
                                        counts[l], ws)
    P = torch.empty(max(L - 1, 1), E, E, dtype=torch.float32, device=dev)
    tcount = torch.empty(max(L - 1, 1), E, E, dtype=torch.int32, device=dev)
    if L >= 2:
        B.ordermoe_transitions_strided(logits, N, L, E, k_freq, E, N * E, tcount, P)
    return {"sim": sim, "counts": counts, "P": P[:L - 1], "tcount": tcount[:L - 1],
            "logits": logits, "xs": xs, "hs": hs}
