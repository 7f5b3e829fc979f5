"""Device-resident layer stacks for ifq_forward (buffer management and marshalling only).

A DeviceStack takes a layer table (paper_1911_08076_gb300.synth) and its float
parameters, folds every quantized substructure with ifq_fold_layer, packs and
prepares the filters on the device with ifq_pack_signs / ifq_pack_weights,
allocates every output buffer with torch, and fills the ifq_layer records that
ifq_forward and ifq_graph_create consume.  All compute is in libifq.so.
"""
from __future__ import annotations

from typing import Dict, List, Optional

import numpy as np
import torch

from . import ifq


class DeviceStack:
    def __init__(self, workload, params, batch: Optional[int] = None, device: str = "cuda", path: int = 0,
                 kbits: Optional[int] = None):
        self.wl = workload
        kbits = getattr(workload, "kbits", 2) if kbits is None else kbits
        self.kbits = kbits
        fb = 2 if kbits == 2 else 4          # bits of a code's storage field
        self.batch = workload.batch if batch is None else batch
        self.device = torch.device(device)
        self.thr: Dict[int, torch.Tensor] = {}
        self.sign: Dict[int, torch.Tensor] = {}
        self.w_prep: Dict[int, torch.Tensor] = {}
        self.y_codes: Dict[int, torch.Tensor] = {}
        self.y_acc: Dict[int, torch.Tensor] = {}
        self.layers: List[ifq.Layer] = []
        self.host_thr: Dict[int, np.ndarray] = {}
        self.host_sign: Dict[int, np.ndarray] = {}
        self.fx: Dict[int, tuple] = {}
        B = self.batch
        kinds = {"conv": ifq.IFQ_LAYER_CONV, "pool": ifq.IFQ_LAYER_POOL, "fixed": ifq.IFQ_LAYER_FIXED}
        # The outputs of the leaf layers (the stack's results) share one contiguous block, so that a
        # caller reads every result back with one copy.
        leaves = set(self.leaf_layers())
        specs = []
        for li in sorted(leaves):
            for shape, dtype in self._out_specs(li, B, fb):
                specs.append((li, shape, dtype))
        offs, total = [], 0
        for _, shape, dtype in specs:
            offs.append(total)
            nbytes = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
            total += (nbytes + 255) // 256 * 256
        self.leaf_block = torch.empty(max(total, 1), dtype=torch.uint8, device=self.device)
        self._leaf_out = {}
        for (li, shape, dtype), off in zip(specs, offs):
            nbytes = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
            self._leaf_out.setdefault(li, []).append(self.leaf_block[off:off + nbytes].view(dtype).view(shape))

        def out(li, shape, dtype):
            if li in self._leaf_out:
                t = self._leaf_out[li].pop(0)
                assert tuple(t.shape) == tuple(shape) and t.dtype == dtype, (li, t.shape, shape)
                return t
            return torch.empty(shape, dtype=dtype, device=self.device)

        for li, l in enumerate(workload.layers):
            rec = ifq.Layer()
            rec.kind = kinds[l.kind]
            rec.src = l.src
            if l.kind == "conv":
                p = params[li]
                mode = {"codes": ifq.IFQ_OUT_CODES, "acc": ifq.IFQ_OUT_ACC, "both": ifq.IFQ_OUT_BOTH}[l.out]
                d = ifq.conv_desc(B, l.h, l.w, l.cin, l.cout, l.k, l.stride, l.pad, mode, path, pool=l.pool,
                                  kbits=kbits, in_bits=l.in_bits)
                K = l.k * l.k * l.cin
                # a layer on 8-bit input values has |A| <= 255 K: its fold clamps at L K_fold >= 255 K
                K_fold = -(-255 * K // ((1 << kbits) - 1)) if l.in_bits == 8 else K
                T, s = ifq.ifq_fold_layer(K_fold, p.alpha, p.gamma, p.beta, p.mean, p.var, p.delta_in, p.bias,
                                          p.eps, p.q_base, p.q_offset, kbits)
                self.host_thr[li], self.host_sign[li] = T, s
                self.thr[li] = torch.from_numpy(T).to(self.device)
                self.sign[li] = torch.from_numpy(s).to(self.device)
                w = torch.from_numpy(np.ascontiguousarray(p.w.reshape(l.cout, K))).to(self.device)
                kwords = (K + 31) // 32
                bits = torch.empty((l.cout, kwords), dtype=torch.int32, device=self.device)
                ifq.ifq_pack_signs(w, bits, l.cout, K)
                prep = torch.empty(ifq.ifq_weights_prep_bytes(d), dtype=torch.uint8, device=self.device)
                ifq.ifq_pack_weights(d, bits, prep)
                self.w_prep[li] = prep
                ho, wo = ifq.ifq_conv_out_shape(d)   # after the fused pool, if any
                assert (ho, wo) == (l.out_h, l.out_w), (l.name, ho, wo)
                if mode & ifq.IFQ_OUT_CODES:
                    self.y_codes[li] = out(li, (B, ho, wo, l.cout * fb // 8), torch.uint8)
                if mode & ifq.IFQ_OUT_ACC:
                    self.y_acc[li] = out(li, (B, ho, wo, l.cout), torch.int32)
                rec.conv = d
                rec.w_prep = prep.data_ptr()
                rec.thr = self.thr[li].data_ptr()
                rec.sign = self.sign[li].data_ptr()
                rec.y_codes = self.y_codes[li].data_ptr() if li in self.y_codes else None
                rec.y_acc = self.y_acc[li].data_ptr() if li in self.y_acc else None
            elif l.kind == "fixed":
                sl, sp = workload.layers[l.src], params[l.src]
                mul, add = ifq.ifq_fold_output_separated(l.m, sp.alpha, sp.delta_in, sp.bias)
                self.fx[li] = (torch.from_numpy(mul).to(self.device), torch.from_numpy(add).to(self.device))
                self.y_acc[li] = out(li, (B, sl.out_h, sl.out_w, sl.cout), torch.int32)
                rec.fixed = ifq.FixedDesc(l.m)
                rec.fx_mul = self.fx[li][0].data_ptr()
                rec.fx_add = self.fx[li][1].data_ptr()
                rec.y_acc = self.y_acc[li].data_ptr()
            else:
                d = ifq.pool_desc(B, l.h, l.w, l.c, l.k, l.stride, l.pad, kbits)
                ho, wo = ifq.ifq_pool_out_shape(d)
                assert (ho, wo) == (l.ho, l.wo), (l.name, ho, wo)
                self.y_codes[li] = out(li, (B, ho, wo, l.c * fb // 8), torch.uint8)
                rec.pool = d
                rec.sign = self.sign[l.src].data_ptr() if l.signed else None
                rec.y_codes = self.y_codes[li].data_ptr()
            self.layers.append(rec)
        self.ws_bytes = ifq.ifq_forward_workspace_bytes(self.layers)
        self.ws = torch.empty(max(self.ws_bytes, 1), dtype=torch.uint8, device=self.device)
        self._graph = None

    def _out_specs(self, li: int, B: int, fb: int):
        """(shape, dtype) of each output buffer of layer li, in the order the constructor makes them."""
        l = self.wl.layers[li]
        if l.kind == "conv":
            specs = []
            if l.out in ("codes", "both"):
                specs.append(((B, l.out_h, l.out_w, l.cout * fb // 8), torch.uint8))
            if l.out in ("acc", "both"):
                specs.append(((B, l.out_h, l.out_w, l.cout), torch.int32))
            return specs
        if l.kind == "fixed":
            sl = self.wl.layers[l.src]
            return [((B, sl.out_h, sl.out_w, sl.cout), torch.int32)]
        return [((B, l.ho, l.wo, l.c * fb // 8), torch.uint8)]

    def input_buffer(self) -> torch.Tensor:
        wl = self.wl
        fb = 8 if getattr(wl, "in_bits", 0) == 8 else (2 if self.kbits == 2 else 4)
        return torch.empty((self.batch, wl.h, wl.w, wl.c * fb // 8), dtype=torch.uint8, device=self.device)

    def forward(self, x: torch.Tensor, stream=None):
        ifq.ifq_forward(self.layers, x, self.ws, self.ws_bytes, stream)

    def forward_layers(self, x: torch.Tensor, before=None, after=None, stream=None):
        """ifq_forward's launches issued one ifq_conv2bit / ifq_maxpool2bit call at a time, with
        optional callbacks before and after each layer (for per-launch CUDA events)."""
        for li, rec in enumerate(self.layers):
            src = x if rec.src < 0 else self.y_codes.get(rec.src)
            if before:
                before(li)
            if rec.kind == ifq.IFQ_LAYER_CONV:
                ifq.ifq_conv2bit(rec.conv, src, rec.w_prep, rec.thr, rec.sign, rec.y_codes, rec.y_acc, self.ws,
                                 self.ws_bytes, stream)
            elif rec.kind == ifq.IFQ_LAYER_FIXED:
                sl = self.wl.layers[rec.src]
                ifq.ifq_fixed_output(self.y_acc[rec.src], self.batch * sl.out_h * sl.out_w, sl.cout,
                                     self.fx[li][0], self.fx[li][1], rec.fixed.m, self.y_acc[li], stream)
            else:
                ifq.ifq_maxpool2bit(rec.pool, src, rec.sign, rec.y_codes, stream)
            if after:
                after(li)

    def capture(self, x: torch.Tensor, stream=None) -> int:
        """Capture ifq_forward on input buffer x into a CUDA graph (replaced on each call)."""
        self.release()
        self._graph = ifq.ifq_graph_create(self.layers, x, self.ws, self.ws_bytes, stream)
        return self._graph

    def leaf_spans(self):
        """(byte offset, bytes) of every leaf output buffer within leaf_block (the block pads each
        buffer to 256 bytes; the padding is not part of any result)."""
        base = self.leaf_block.data_ptr()
        spans = []
        for li in self.leaf_layers():
            for t in (self.y_codes.get(li), self.y_acc.get(li)):
                if t is not None:
                    spans.append((t.data_ptr() - base, t.numel() * t.element_size()))
        return spans

    def leaf_results_equal(self, leaf_host: torch.Tensor, other: Optional[torch.Tensor] = None) -> bool:
        """Whether the host copy of the leaf block holds the same results as this stack's device block
        (or as `other`, a block of the same layout), buffer by buffer."""
        dev = (self.leaf_block if other is None else other).cpu()
        return all(torch.equal(leaf_host[o:o + n], dev[o:o + n]) for o, n in self.leaf_spans())

    def capture_io(self, x: torch.Tensor, x_host: torch.Tensor, leaf_host: torch.Tensor, stream=None) -> int:
        """Capture ifq_forward on input buffer x into a CUDA graph that also copies x_host (pinned)
        into x first and every leaf layer's outputs into leaf_host (pinned, the size of leaf_block,
        the same layout) right after that layer (replaced on each call)."""
        assert leaf_host.numel() * leaf_host.element_size() == self.leaf_block.numel()
        base_d, base_h = self.leaf_block.data_ptr(), leaf_host.data_ptr()
        n = len(self.layers)
        codes_dst, acc_dst = [None] * n, [None] * n
        for li in self.leaf_layers():
            if li in self.y_codes:
                codes_dst[li] = base_h + (self.y_codes[li].data_ptr() - base_d)
            if li in self.y_acc:
                acc_dst[li] = base_h + (self.y_acc[li].data_ptr() - base_d)
        self.release()
        self._graph = ifq.ifq_graph_create_io(self.layers, x, self.ws, self.ws_bytes, x_host,
                                              x_host.numel() * x_host.element_size(), codes_dst, acc_dst, stream)
        return self._graph

    def replay(self, stream=None):
        ifq.ifq_graph_launch(self._graph, stream)

    def release(self):
        if self._graph is not None:
            ifq.ifq_graph_destroy(self._graph)
            self._graph = None

    def __del__(self):
        try:
            self.release()
        except Exception:
            pass

    def leaf_layers(self) -> List[int]:
        """Layers whose output no other layer consumes (the stack's results)."""
        used = {l.src for l in self.wl.layers}
        return [i for i in range(len(self.wl.layers)) if i not in used]

    def output(self, li: int):
        """Host copy of layer li's output: codes (packed uint8) and/or int32 accumulators."""
        out = {}
        if li in self.y_codes:
            out["codes"] = self.y_codes[li].cpu().numpy()
        if li in self.y_acc:
            out["acc"] = self.y_acc[li].cpu().numpy()
        return out
