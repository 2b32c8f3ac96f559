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

    def capture(self, X_layers, home, loc, qhat, y_layers, counters=None, prologue=None):
        """Records one step (every layer's kernels, after the optional prologue,
        e.g. resetting loc and qhat) as a CUDA graph over these buffers, so a
        step is one graph launch. Returns the torch.cuda.CUDAGraph; replay()
        runs the step on the buffers' current contents."""
        s = torch.cuda.Stream(device=self.scratch.device)
        s.wait_stream(torch.cuda.current_stream(self.scratch.device))
        with torch.cuda.stream(s):  # one eager step first: per-device set-up outside the capture
            if prologue is not None:
                prologue()
            self.step(X_layers, home, loc, qhat, y_layers, counters, stream=s)
        torch.cuda.current_stream(self.scratch.device).wait_stream(s)
        torch.cuda.synchronize(self.scratch.device)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            if prologue is not None:
                prologue()
            self.step(X_layers, home, loc, qhat, y_layers, counters, stream=s)
        return g
