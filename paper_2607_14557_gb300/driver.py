"""One-GPU driver of the Seer hot path (argument marshalling and buffers only).

The driver owns the device buffers of one batch and enqueues the library's
entry points on one CUDA stream:

* ``SeerPath.step`` -- the step-0 detector (Sec. 3.2-3.3), routing +
  device-resident compaction (Sec. 3.4-3.5) and one truncated layer
  (Sec. 3.6), all enqueued back to back with no host synchronisation: every
  kernel reads the packed row count from device memory, so the layer can be
  queued before the host has seen the route.  The host reads the route later
  from the pinned control word (``SeerPath.route``), i.e. the latency of the
  decision is hidden behind the GPU work ("latency shadowing").
* ``SeerPath.padded_forward`` -- the same layer kernels over the untruncated
  window (the comparator of the speedup).
* ``SeerStack`` -- the multi-layer, multi-step denoising loop: one full
  step-0 pass (counts fused into the detection layer's gate/up epilogue),
  boundary scan and compaction, then the remaining steps over the packed
  sequences, replayed from a CUDA graph captured per graph capacity.

Every computation happens in libseer's CUDA kernels; this module never
touches tensor values on the host.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np
import torch

from . import seer as S


def _dev():
    return torch.device("cuda", torch.cuda.current_device())


def f16_copy(t: torch.Tensor) -> torch.Tensor:
    """f16 copy of a bf16 device tensor made by the library's converter."""
    dst = torch.empty(t.shape, dtype=torch.float16, device=t.device)
    S.seer_convert(t, "bf16", dst, "f16", t.numel())
    return dst


@dataclasses.dataclass
class LayerWeights:
    """Device weights of one block.  ``model`` holds the model-dtype tensors
    (the detector reads gate/up from here); ``run`` the tensors the layer
    kernels read (f16 copies for a bf16 model)."""
    model: Dict[str, torch.Tensor]
    run: Dict[str, torch.Tensor]

    @staticmethod
    def from_host(w: Dict[str, np.ndarray], dtype: str, device=None) -> "LayerWeights":
        device = device or _dev()
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        up = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device=device, dtype=tdt)
        model = {"w_qkv": up(np.concatenate([w["wq"], w["wk"], w["wv"]], axis=0)), "w_o": up(w["wo"]),
                 "w_gate": up(w["wg"]), "w_up": up(w["wu"]), "w_down": up(w["wd"]), "g_attn": up(w["g_attn"]),
                 "g_mlp": up(w["g_mlp"])}
        run = model if dtype == "f32" else {k: f16_copy(v) for k, v in model.items()}
        return LayerWeights(model, run)

    @staticmethod
    def from_bf16_bits(bits: Dict[str, np.ndarray], device=None, keep_model=()) -> "LayerWeights":
        """Upload bf16 bit patterns ({name: uint16 array}, as produced for a
        stack) and make the f16 copies the kernels run on; keep only the
        model-dtype tensors named in ``keep_model``."""
        device = device or _dev()
        up = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16).to(device)
        model = {"w_qkv": up(np.concatenate([bits["wq"], bits["wk"], bits["wv"]], axis=0)), "w_o": up(bits["wo"]),
                 "w_gate": up(bits["wg"]), "w_up": up(bits["wu"]), "w_down": up(bits["wd"]),
                 "g_attn": up(bits["g_attn"]), "g_mlp": up(bits["g_mlp"])}
        run = {k: f16_copy(v) for k, v in model.items()}
        return LayerWeights({k: v for k, v in model.items() if k in keep_model}, run)

    def struct(self) -> S.seer_layer_weights:
        r = self.run
        return S.make_weights(r["w_qkv"], r["w_o"], r["w_gate"], r["w_up"], r["w_down"], r["g_attn"], r["g_mlp"])

    def drop_model_copy(self, keep=("w_gate", "w_up")):
        """Free the model-dtype tensors the kernels no longer need."""
        if self.model is self.run:
            return
        self.model = {k: v for k, v in self.model.items() if k in keep}


class SeerPath:
    """Buffers and launches of one batch through detect -> pack -> layer."""

    def __init__(self, dims: S.seer_dims, dtype: str, B: int, N: int, T_full: int, params: S.seer_params,
                 device=None):
        self.dims, self.dtype, self.B, self.N, self.T_full, self.params = dims, dtype, B, N, T_full, params
        dev = self.device = device or _dev()
        tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
        d = dims.d_model
        i32 = dict(dtype=torch.int32, device=dev)
        self.counts = torch.empty(B * N, **i32)
        self.L_star = torch.empty(B, **i32)
        self.i_star = torch.empty(B, **i32)
        self.cu = torch.empty(B + 1, **i32)
        self.kv = torch.empty(B, **i32)
        self.meta = torch.empty(S.CTRL_WORDS, **i32)
        self.host_ctrl = torch.zeros(S.CTRL_WORDS, dtype=torch.int32).pin_memory()
        self.ctrl = torch.zeros(S.CTRL_WORDS, dtype=torch.int32)
        self.x_packed = torch.zeros((T_full, d), dtype=tdt, device=dev)
        self.y = torch.empty((T_full, d), dtype=tdt, device=dev)
        self.ws_bytes = S.seer_layer_workspace_size(dims, dtype, T_full, B)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=dev)
        self.epoch = 0

    def detect(self, x_full, resp_start, w: LayerWeights, stream=None):
        S.seer_detect_boundary(x_full, self.dtype, x_full.shape[0], resp_start, self.B, self.N, w.model["w_gate"],
                               w.model["w_up"], self.dims, self.params, self.counts, self.L_star, self.i_star,
                               stream=stream)

    def detect_multi(self, x_full, resp_start, taps: List[LayerWeights], stream=None):
        """Boundary from a multi-layer sparsity tap (Sec. 4.5 / Table 12): the
        near-zero counts of the response rows under each tapped layer's gate/up
        weights are summed (a count out of len(taps) * F) and scanned once."""
        for i, w in enumerate(taps):
            S.seer_sparsity_counts(x_full, self.dtype, x_full.shape[0], resp_start, self.B, self.N, w.model["w_gate"],
                                   w.model["w_up"], self.dims, self.params.act_eps, self.counts, accumulate=i > 0,
                                   stream=stream)
        S.seer_snr_scan(self.counts, self.B, self.N, len(taps) * self.dims.d_ff, self.params, self.L_star, self.i_star,
                        stream=stream)

    def pack(self, x_full, cu_full, ctx_len, stream=None):
        self.epoch += 1
        S.seer_pack_ragged(x_full, self.dtype, cu_full, ctx_len, self.L_star, self.B, self.dims.d_model, self.N,
                           self.T_full, self.params, self.x_packed, self.cu, self.kv, self.meta, self.host_ctrl,
                           self.epoch, stream=stream)

    def layer(self, w: LayerWeights, x=None, y=None, cu=None, kv=None, T_cap=None, stream=None):
        x = self.x_packed if x is None else x
        y = self.y if y is None else y
        S.seer_layer_forward(w.struct(), self.dims, self.dtype, x, y, self.cu if cu is None else cu,
                             self.kv if cu is None else kv, self.B, self.T_full if T_cap is None else T_cap, None, 0,
                             0.0, None, self.ws, self.ws_bytes, stream=stream)

    def step(self, x_full, cu_full, resp_start, ctx_len, w: LayerWeights, stream=None):
        """Detect, route + pack and run the truncated layer; nothing waits on the host."""
        self.detect(x_full, resp_start, w, stream)
        self.pack(x_full, cu_full, ctx_len, stream)
        self.layer(w, stream=stream)

    def run_from_host(self, x_host, cu_full, resp_start, ctx_len, w: LayerWeights, y_host, L_host, steps: int,
                      stream=None, copy_stream=None) -> Dict[str, object]:
        """``steps`` end-to-end steps from pinned host memory: every step copies
        its full-window input host -> device, runs detect -> route/pack ->
        truncated layer, and copies the packed output rows and L* device ->
        host.  Copies run on ``copy_stream`` with double-buffered device
        inputs and outputs, so step i+1's upload and step i-1's download
        overlap step i's compute.  Returns the route of the last step; all
        copies have completed on return."""
        dev = self.device
        stream = stream or torch.cuda.current_stream(dev)
        copy_stream = copy_stream or torch.cuda.Stream(dev)
        if getattr(self, "_x_in", None) is None or self._x_in[0].shape != x_host.shape:
            self._x_in = [torch.empty(x_host.shape, dtype=x_host.dtype, device=dev) for _ in range(2)]
            self._y_out = [self.y, torch.empty_like(self.y)]
            self._L_out = [torch.empty_like(self.L_star) for _ in range(2)]
        x_in, y_out, L_out = self._x_in, self._y_out, self._L_out
        loaded = [torch.cuda.Event() for _ in range(2)]      # input buffer holds its step's data
        consumed = [torch.cuda.Event() for _ in range(2)]    # compute no longer reads the input buffer
        computed = [torch.cuda.Event() for _ in range(2)]    # output buffer holds its step's result
        drained = [torch.cuda.Event() for _ in range(2)]     # output buffer copied to the host
        for e in consumed + drained:
            e.record(stream)

        def upload(i):
            b = i % 2
            copy_stream.wait_event(consumed[b])
            with torch.cuda.stream(copy_stream):
                x_in[b].copy_(x_host, non_blocking=True)
            loaded[b].record(copy_stream)

        route = None
        upload(0)
        for i in range(steps):
            b = i % 2
            if i + 1 < steps:
                upload(i + 1)
            stream.wait_event(loaded[b])
            stream.wait_event(drained[b])
            self.detect(x_in[b], resp_start, w, stream)
            self.pack(x_in[b], cu_full, ctx_len, stream)
            consumed[b].record(stream)
            self.layer(w, y=y_out[b], stream=stream)
            L_out[b].copy_(self.L_star, non_blocking=True)
            computed[b].record(stream)
            route = self.route()                 # host learns the packed total while the layer runs
            copy_stream.wait_event(computed[b])
            with torch.cuda.stream(copy_stream):
                y_host[:route["total"]].copy_(y_out[b][:route["total"]], non_blocking=True)
                L_host.copy_(L_out[b], non_blocking=True)
            drained[b].record(copy_stream)
        copy_stream.synchronize()
        stream.synchronize()
        return route

    def route(self, timeout_us: int = 10_000_000) -> Dict[str, object]:
        """Read the route of the last pack from the pinned control word."""
        S.seer_poll_ctrl(self.host_ctrl, self.epoch, timeout_us, self.ctrl)
        c = self.ctrl.numpy()
        groups = [{"bucket": int(c[8 + 4 * g]), "members": int(c[9 + 4 * g]), "path": int(c[10 + 4 * g]),
                   "rho": c[11 + 4 * g] / 1e6} for g in range(int(c[4]))]
        return {"total": int(c[1]), "max_seqlen": int(c[2]), "capacity": int(c[3]), "path_mask": int(c[5]),
                "pad_rows": int(c[6]), "groups": groups}

    def naive_pad_inputs(self, x_full, cu_full, ctx_len, stream=None):
        """Inputs of the naive-pad comparator (the batch-max padding that Sec. 3.4
        improves on, Eq. 3): every sequence keeps ``ctx_b + max_b L*_b`` rows,
        rows past ``ctx_b + L*_b`` are computed as queries and masked as keys.

        Built once after a step has produced ``L_star`` (reads it on the host);
        the rows are gathered by the library's pack kernel with the static path
        switched off (``tau_pad < 0``), so every segment keeps exactly its rows.
        Returns ``(x, cu, kv_len, T)``.
        """
        B, dev = self.B, self.device
        L = self.L_star.cpu().numpy().astype(np.int64)
        ctx = ctx_len.cpu().numpy().astype(np.int64)
        L_max = int(L.max())
        T = int(ctx.sum() + B * L_max)
        i32 = dict(dtype=torch.int32, device=dev)
        L_pad = torch.full((B,), L_max, **i32)
        x = torch.zeros((max(T, 1), self.dims.d_model), dtype=self.x_packed.dtype, device=dev)
        cu = torch.empty(B + 1, **i32)
        kv_all = torch.empty(B, **i32)
        meta = torch.empty(S.CTRL_WORDS, **i32)
        p = self.params
        no_static = S.make_params(p.act_eps, p.tau_jump, p.gamma, p.window, -1.0, p.eager_max_bucket, p.bucket_min)
        S.seer_pack_ragged(x_full, self.dtype, cu_full, ctx_len, L_pad, B, self.dims.d_model, self.N, T, no_static, x,
                           cu, kv_all, meta, None, 0, stream=stream)
        kv = torch.as_tensor((ctx + L).astype(np.int32)).to(dev)
        return x, cu, kv, T

    def varlen_only_inputs(self, x_full, cu_full, ctx_len, stream=None):
        """The last step's batch packed with the static path switched off
        (``tau_pad < 0``): every segment keeps exactly ``ctx_b + L*_b`` rows, so
        no bucket padding is computed.  Compared with the routed layout it
        prices the rows the static-graph groups pad (Sec. 3.4, Eq. 4).
        Returns ``(x, cu, kv_len, T_capacity)``."""
        B, dev = self.B, self.device
        i32 = dict(dtype=torch.int32, device=dev)
        x = torch.zeros_like(self.x_packed)
        cu = torch.empty(B + 1, **i32)
        kv = torch.empty(B, **i32)
        meta = torch.empty(S.CTRL_WORDS, **i32)
        p = self.params
        no_static = S.make_params(p.act_eps, p.tau_jump, p.gamma, p.window, -1.0, p.eager_max_bucket, p.bucket_min)
        S.seer_pack_ragged(x_full, self.dtype, cu_full, ctx_len, self.L_star, B, self.dims.d_model, self.N,
                           self.T_full, no_static, x, cu, kv, meta, None, 0, stream=stream)
        return x, cu, kv, self.T_full

    def padded_forward(self, x_full, cu_full, w: LayerWeights, y_full, stream=None):
        """The same layer over the untruncated windows (every key kept)."""
        S.seer_layer_forward(w.struct(), self.dims, self.dtype, x_full, y_full, cu_full, None, self.B, self.T_full,
                             None, 0, 0.0, None, self.ws, self.ws_bytes, stream=stream)


class SeerStack:
    """Denoising loop over a stack of layers (one GPU).

    Step 0 runs every layer over the full windows; the detection layer's
    gate/up epilogue counts near-zero activations of the response rows
    (``hook_counts``).  The boundaries that drive truncation come from the
    detector applied to the step-0 input rows with the detection layer's
    gate/up weights (random-init weights carry no semantic signal after a
    normalised stack, so the planted input stands in for a trained model);
    the route/pack kernel then compacts the step-0 input, and steps 1..T-1 run
    every layer over the packed sequences.  Step bodies are captured into CUDA
    graphs: the kernels read the packed row count from device memory, so one
    graph per capacity serves any total up to it.
    """

    def __init__(self, dims, dtype, B, N, T_full, params, layers: List[LayerWeights], detect_layer: int = 3,
                 device=None):
        self.path = SeerPath(dims, dtype, B, N, T_full, params, device)
        self.layers = layers
        self.detect_layer = detect_layer
        dev = self.path.device
        tdt = self.path.x_packed.dtype
        d = dims.d_model
        self.buf = [torch.empty((T_full, d), dtype=tdt, device=dev) for _ in range(2)]
        self.hook_counts = torch.zeros(B * N, dtype=torch.int32, device=dev)
        self.graphs: Dict[object, torch.cuda.CUDAGraph] = {}
        self.h_packed: Optional[torch.Tensor] = None
        self.kv_cache: Optional[List[torch.Tensor]] = None
        self.ctx_len: Optional[torch.Tensor] = None

    def _run_layers(self, x, cu, kv, T_cap, resp_start=None, stream=None, n_layers=None, start=0):
        p = self.path
        cur = x
        stop = len(self.layers) if n_layers is None else n_layers
        for li in range(start, stop):
            w = self.layers[li]
            out = self.buf[li % 2] if cur is not self.buf[li % 2] else self.buf[(li + 1) % 2]
            count = resp_start is not None and li == self.detect_layer
            S.seer_layer_forward(w.struct(), p.dims, p.dtype, cur, out, cu, kv, p.B, T_cap,
                                 resp_start if count else None, p.N if count else 0,
                                 p.params.act_eps if count else 0.0, self.hook_counts if count else None, p.ws,
                                 p.ws_bytes, stream=stream)
            cur = out
        return cur

    def step0(self, x_full, cu_full, resp_start, ctx_len, stream=None):
        """Full-window step with the fused count hook, then detect + route/pack."""
        p = self.path
        self.ctx_len = ctx_len
        out = self._run_layers(x_full, cu_full, None, p.T_full, resp_start=resp_start, stream=stream)
        p.detect(x_full, resp_start, self.layers[self.detect_layer], stream)
        p.pack(x_full, cu_full, ctx_len, stream)
        return out

    def step0_truncating(self, x_full, cu_full, resp_start, ctx_len, stream=None):
        """Step 0 truncated inside the step (Sec. 3.1: the layers after detection
        run on the retained tokens only): layers ``0..detect_layer`` over the
        full windows with the count hook, detection and route/pack, then the
        detection layer's output is compacted with the same layout and the
        remaining layers run over the packed sequences.  The step-0 input is
        packed too (input of the later steps).  Returns the last layer's output
        in the packed layout."""
        p = self.path
        self.ctx_len = ctx_len
        h = self._run_layers(x_full, cu_full, None, p.T_full, resp_start=resp_start, stream=stream,
                             n_layers=self.detect_layer + 1)
        p.detect(x_full, resp_start, self.layers[self.detect_layer], stream)
        p.pack(x_full, cu_full, ctx_len, stream)
        if self.h_packed is None:
            self.h_packed = torch.empty_like(p.x_packed)
        S.seer_pack_ragged(h, p.dtype, cu_full, ctx_len, p.L_star, p.B, p.dims.d_model, p.N, p.T_full, p.params,
                           self.h_packed, p.cu, p.kv, p.meta, None, 0, stream=stream)
        return self._run_layers(self.h_packed, p.cu, p.kv, p.T_full, stream=stream, start=self.detect_layer + 1)

    def truncated_step(self, T_cap=None, stream=None):
        p = self.path
        return self._run_layers(p.x_packed, p.cu, p.kv, T_cap or p.T_full, stream=stream)

    def padded_step(self, x_full, cu_full, stream=None):
        return self._run_layers(x_full, cu_full, None, self.path.T_full, stream=stream)

    def capture(self, key, fn):
        """Capture ``fn(stream=...)`` (one step body) into a CUDA graph under ``key``."""
        if key in self.graphs:
            return self.graphs[key]
        S.seer_profile_enable(False)
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            fn(stream=s)                       # warm-up outside capture
        torch.cuda.current_stream().wait_stream(s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            fn(stream=torch.cuda.current_stream())
        self.graphs[key] = g
        return g

    # ------------------------------------------------------------ prefix K/V cache
    def _cache_buffers(self):
        """Per-layer K/V caches [T_full, 2*H*dh] in the layers' intermediate
        type (packed truncated layout) and the response-row buffers."""
        p = self.path
        if self.kv_cache is None:
            dev = p.device
            it = torch.float32 if p.dtype == "f32" else torch.float16
            D = p.dims.n_heads * p.dims.head_dim
            self.kv_cache = [torch.empty((p.T_full, 2 * D), dtype=it, device=dev) for _ in self.layers]
            self.resp = [torch.empty_like(p.x_packed) for _ in range(3)]
            self.cu_resp = torch.empty(p.B + 1, dtype=torch.int32, device=dev)
        return self.kv_cache

    def prefill_step(self, stream=None):
        """A truncated step that also fills every layer's prefix K/V cache from
        that layer's input (the visual + prompt rows of each packed segment)."""
        p = self.path
        caches = self._cache_buffers()
        cur = p.x_packed
        for li, w in enumerate(self.layers):
            S.seer_kv_prefill(w.struct(), p.dims, p.dtype, cur, p.cu, self.ctx_len, p.B, p.T_full, caches[li], p.cu,
                              p.T_full, p.ws, p.ws_bytes, stream=stream)
            out = self.buf[li % 2] if cur is not self.buf[li % 2] else self.buf[(li + 1) % 2]
            S.seer_layer_forward(w.struct(), p.dims, p.dtype, cur, out, p.cu, p.kv, p.B, p.T_full, None, 0, 0.0, None,
                                 p.ws, p.ws_bytes, stream=stream)
            cur = out
        return cur

    def cached_step(self, resp_cap=None, stream=None):
        """A step over the response rows only: prefix keys/values come from the
        caches (Table 7: truncation composes with prefix KV caching).  Launches
        are sized for ``resp_cap`` response rows (default: the whole buffer);
        the kernels read the true count from ``cu_resp[B]``.  Returns the last
        layer's output rows in the response layout (``cu_resp``)."""
        p = self.path
        caches = self._cache_buffers()
        cap = p.T_full if resp_cap is None else min(int(resp_cap), p.T_full)
        S.seer_gather_response(p.x_packed, p.dtype, p.cu, self.ctx_len, p.B, p.dims.d_model, p.T_full, self.resp[0],
                               self.cu_resp, stream=stream)
        cur = self.resp[0]
        for li, w in enumerate(self.layers):
            out = self.resp[1] if cur is not self.resp[1] else self.resp[2]
            S.seer_layer_forward_cached(w.struct(), p.dims, p.dtype, cur, out, self.cu_resp, self.ctx_len, p.B, cap,
                                        caches[li], p.cu, p.kv, p.T_full, p.ws, p.ws_bytes, stream=stream)
            cur = out
        return cur

    def cached_graph(self, resp_cap: int):
        """Graph of one cached step sized for ``resp_cap`` response rows."""
        cap = min(int(resp_cap), self.path.T_full)
        self._cache_buffers()
        return self.capture(("cached", cap), lambda stream: self.cached_step(cap, stream=stream))

    def truncated_graph(self, capacity: int):
        """Graph of one truncated step sized for ``capacity`` packed rows."""
        cap = min(int(capacity), self.path.T_full)
        return self.capture(("trunc", cap), lambda stream: self.truncated_step(cap, stream=stream))
