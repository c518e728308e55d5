"""Library reference for the oracle's pins: the same Whisper-style decoder built
from torch.nn.TransformerDecoderLayer (pre-LN, erf GELU, eps 1e-5) in float64.

Only the CPU tests use it.  It shares nothing with ``oracle/``: attention,
LayerNorm, GELU, the causal and padding masks and the head-averaged attention
weights all come from torch.nn, so a dropped term, a wrong scale, a transposed
operand or a wrong mask in the oracle shows up as a mismatch.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn as nn
import torch.nn.functional as F

import workload as W


def _t(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float64).copy())


class TorchDecoder:
    def __init__(self, dims: W.ModelDims, blob: np.ndarray):
        self.dims = dims
        d, H, Fd = dims.d_model, dims.n_heads, dims.d_ffn
        g = lambda n: _t(W.weight_view(dims, blob, n))
        self.tok = g("tok_emb")
        self.pos = g("pos_emb")
        self.lnf = nn.LayerNorm(d, eps=1e-5).double()
        with torch.no_grad():
            self.lnf.weight.copy_(g("lnf_g"))
            self.lnf.bias.copy_(g("lnf_b"))
        self.layers = []
        for l in range(dims.n_layers):
            p = f"L{l}."
            m = nn.TransformerDecoderLayer(d, H, dim_feedforward=Fd, dropout=0.0,
                                           activation="gelu", layer_norm_eps=1e-5,
                                           batch_first=True, norm_first=True).double().eval()
            z = torch.zeros(d, dtype=torch.float64)
            with torch.no_grad():
                m.self_attn.in_proj_weight.copy_(torch.cat([g(p + "wq"), g(p + "wk"), g(p + "wv")]))
                m.self_attn.in_proj_bias.copy_(torch.cat([g(p + "bq"), z, g(p + "bv")]))
                m.self_attn.out_proj.weight.copy_(g(p + "wo"))
                m.self_attn.out_proj.bias.copy_(g(p + "bo"))
                m.multihead_attn.in_proj_weight.copy_(torch.cat([g(p + "wcq"), g(p + "wck"), g(p + "wcv")]))
                m.multihead_attn.in_proj_bias.copy_(torch.cat([g(p + "bcq"), z, g(p + "bcv")]))
                m.multihead_attn.out_proj.weight.copy_(g(p + "wco"))
                m.multihead_attn.out_proj.bias.copy_(g(p + "bco"))
                m.linear1.weight.copy_(g(p + "w1"))
                m.linear1.bias.copy_(g(p + "b1"))
                m.linear2.weight.copy_(g(p + "w2"))
                m.linear2.bias.copy_(g(p + "b2"))
                for i in (1, 2, 3):
                    getattr(m, f"norm{i}").weight.copy_(g(p + f"ln{i}_g"))
                    getattr(m, f"norm{i}").bias.copy_(g(p + f"ln{i}_b"))
            self.layers.append(m)

    @torch.no_grad()
    def forward(self, tokens, enc_states, enc_len, anchor_layer=None):
        """Full-sequence forward of one utterance (no cache): tokens at positions
        0..n-1.  Returns logits [n, V] and, if anchor_layer is given, the
        head-averaged cross-attention weights [n, enc_len] of that layer."""
        n = len(tokens)
        tok = torch.as_tensor(np.asarray(tokens, dtype=np.int64))
        x = (F.embedding(tok, self.tok) + self.pos[:n]).unsqueeze(0)
        mem = _t(enc_states[:enc_len]).unsqueeze(0)
        causal = nn.Transformer.generate_square_subsequent_mask(n, dtype=torch.float64)
        captured = {}
        for l, m in enumerate(self.layers):
            hook = None
            if anchor_layer is not None and l == anchor_layer:
                def grab(mod, args, kwargs, out):
                    if captured.get("busy"):
                        return
                    captured["busy"] = True
                    _, w = mod(args[0], mem, mem, need_weights=True, average_attn_weights=True)
                    captured["busy"] = False
                    captured["w"] = w[0]
                hook = m.multihead_attn.register_forward_hook(grab, with_kwargs=True)
            x = m(x, mem, tgt_mask=causal, tgt_is_causal=True)
            if hook is not None:
                hook.remove()
        logits = self.lnf(x[0]) @ self.tok.T
        return logits.numpy(), (captured["w"].numpy() if "w" in captured else None)

    def greedy(self, prompt, enc_states, enc_len, total_len):
        """Plain greedy decoding by full recomputation at every step."""
        seq = list(int(t) for t in prompt)
        while len(seq) < total_len:
            logits, _ = self.forward(seq, enc_states, enc_len)
            seq.append(int(np.argmax(logits[-1])))
        return seq
