"""Layer stacking by the static per-layer profile mask (Sec. layer-wise
Hadamard strategy selection; Table integer_transitions): a chain of prepared
layers run through hatq_layer, one call per layer.

Each layer's epilogue emits either the next layer's INT8 operand directly
(the next layer is WH, or its DH input transform is fused into this epilogue
with hb_next) or original-basis INT8 codes that the next layer's hatq_layer
call transforms and requantizes first. No arithmetic happens here.
"""
from __future__ import annotations

from . import hatq


class Chain:
    def __init__(self, layers, params, scales, plan, out_f32_last=False, device="cuda", f16_operands=()):
        """layers: objects with c_in, c_out, k, stride, pad, form, hb_in, hb_out, act;
        params: [(w_ohwi float32, bias float32)]; scales: [{'s_x', 's_out'}, plus 's_z' and
        's_u' for a SiLU / GELU layer]; plan: per layer the block of the next layer's DH
        transform fused in its epilogue (0 = none); f16_operands: indices of layers
        whose operand (emitted directly by the layer before) is stored as fp16 codes
        (hatq_set_operand_format), so it is converted once by its producer instead
        of once per output-channel tile by its consumer."""
        self.layers = list(layers)
        self.plan = list(plan)
        self.prepared = []
        for i, (L, (w, b), sc) in enumerate(zip(self.layers, params, scales)):
            last = i == len(self.layers) - 1
            self.prepared.append(hatq.prepare_weights(
                hatq.desc_from_spec(L), w, b, sc["s_x"], sc["s_out"], L.act, self.plan[i],
                out_f32_last and last, device=device, s_z=sc.get("s_z"), s_u=sc.get("s_u")))
        for i in sorted(set(f16_operands)):
            if not 0 < i < len(self.layers) or not (self.plan[i - 1] or self.layers[i].form == "WH"):
                raise ValueError(f"layer {i} does not take its operand straight from the layer before")
            hatq.set_operand_format(self.prepared[i], True, self.prepared[i].out_f16)
            hatq.set_operand_format(self.prepared[i - 1], self.prepared[i - 1].in_f16, True)

    def input_kinds(self, x_kind, s_in):
        """(kind, scale) of each layer's input, mirroring what each epilogue emits."""
        kinds = [(x_kind, s_in)]
        for i in range(len(self.layers) - 1):
            P = self.prepared[i]
            if self.plan[i] or self.layers[i + 1].form == "WH":
                kinds.append((hatq.IN_OPERAND, P.s_y))
            else:
                kinds.append((hatq.IN_I8, P.s_y))
        return kinds

    def shapes(self, n, h, w):
        out = []
        for P in self.prepared:
            s = P.out_shape(n, h, w)
            out.append(s)
            _, h, w, _ = s
        return out

    def alloc(self, n, h, w, device="cuda"):
        """Output buffers and one scratch buffer large enough for any layer input."""
        import torch
        outs, scratch = [], 0
        hh, ww = h, w
        for P in self.prepared:
            scratch = max(scratch, n * hh * ww * P.c_in)
            s = P.out_shape(n, hh, ww)
            outs.append(torch.empty(s, dtype=getattr(torch, P.out_dtype), device=device))
            hh, ww = s[1], s[2]
        return outs, torch.empty(max(scratch, 16), dtype=torch.int8, device=device)

    def forward(self, x, x_kind, s_in, outs=None, scratch=None, stream=None):
        n, h, w, _ = x.shape
        if outs is None:
            outs, scratch = self.alloc(n, h, w, x.device)
        kinds = self.input_kinds(x_kind, s_in)
        cur = x
        for i, P in enumerate(self.prepared):
            k, s = kinds[i]
            hatq.layer(cur, k, s, P, y=outs[i], scratch=scratch, stream=stream)
            cur = outs[i]
        return outs

    def launches(self, x_kind, s_in):
        return sum(hatq.layer_launches(k, s, P) for (k, s), P in zip(self.input_kinds(x_kind, s_in), self.prepared))
