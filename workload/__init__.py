"""Seeded synthetic workloads for the draft-verify step.

This module only draws inputs: decoder weights, encoder states, prompts,
utterance lengths and the draft-corruption stream.  It holds none of the
decoder's arithmetic and none of the acceptance rule, so both the CPU oracle
(``oracle/``) and the CUDA path (``paper_2608_12703_gb300``) can take their
inputs from it without sharing any computation.

The paper's evaluation audio, trained checkpoints and trained drafts are not
available; the shapes below follow its workloads instead:

* utterances of at most 30 s, i.e. at most 1500 Whisper encoder frames
  (App. "Official-Split Position Effect" excludes clips over 30 s);
* Whisper-large-v3 / Whisper-small shaped decoders (Sec. 3 "Models and
  Protocol" names Whisper as the cross-architecture target);
* batch 1 and batch 64 (Sec. 5 "Deployment Scope");
* draft blocks of up to K tokens (Sec. 3 "Speculative Loop").

Random streams (numpy PCG64 through ``default_rng``):
  seed 0 weights, 1 encoder states, 2 draft corruption, 3 prompt, 4 lengths,
  5 draft-model weights.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

MAX_POS = 448          # Whisper decoder context (learned positional table)
MAX_ENC = 1500         # 30 s at 20 ms per encoder frame
PROMPT_LEN = 4         # fixed prompt length (the paper does not fix one)

SEED_WEIGHTS = 0
SEED_ENCODER = 1
SEED_CORRUPT = 2
SEED_PROMPT = 3
SEED_LENGTHS = 4
SEED_DRAFT = 5


@dataclasses.dataclass(frozen=True)
class ModelDims:
    n_layers: int
    d_model: int
    n_heads: int
    d_ffn: int
    vocab: int
    dtype: str                      # "fp32" or "bf16": storage of weights/KV
    max_pos: int = MAX_POS
    max_enc: int = MAX_ENC
    anchor_layer: int = -1          # -1 -> floor(3 L / 4), 0-based

    @property
    def head_dim(self) -> int:
        return self.d_model // self.n_heads

    @property
    def anchor(self) -> int:
        return self.anchor_layer if self.anchor_layer >= 0 else (3 * self.n_layers) // 4


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic decoding job: a decoder shape plus a batch of utterances."""
    name: str
    dims: ModelDims
    batch: int
    k: int                          # maximum draft length per round
    n_out: Tuple[int, ...]          # output tokens per utterance (after the prompt)
    enc_lens: Tuple[int, ...]       # encoder frames per utterance
    err: Tuple[float, ...]          # per-utterance draft-token replacement rate
    shift: str                      # "none" | "always" | "half"
    t_max: int = MAX_ENC

    @property
    def total_lens(self) -> Tuple[int, ...]:
        return tuple(PROMPT_LEN + n for n in self.n_out)


TINY = ModelDims(n_layers=4, d_model=384, n_heads=6, d_ffn=1536, vocab=51865, dtype="fp32")
SMALL = ModelDims(n_layers=12, d_model=768, n_heads=12, d_ffn=3072, vocab=51865, dtype="bf16")
LARGE = ModelDims(n_layers=32, d_model=1280, n_heads=20, d_ffn=5120, vocab=51866, dtype="bf16")


def _uniform_lengths(batch: int, seed_offset: int):
    rng = np.random.default_rng([SEED_LENGTHS, seed_offset])
    enc = rng.integers(250, 1501, size=batch)
    n_out = np.rint(rng.lognormal(mean=math.log(60.0), sigma=0.5, size=batch))
    n_out = np.clip(n_out, 1, 224).astype(int)
    err = rng.uniform(0.1, 0.5, size=batch)
    return tuple(int(x) for x in enc), tuple(int(x) for x in n_out), tuple(float(x) for x in err)


def _make_configs() -> Dict[str, Workload]:
    c4_enc, c4_out, c4_err = _uniform_lengths(64, 0)
    cfgs = {
        "tiny-fp32-b1-k4": Workload("tiny-fp32-b1-k4", TINY, 1, 4, (64,), (1500,), (0.3,), "none"),
        "small-bf16-b16-k8": Workload("small-bf16-b16-k8", SMALL, 16, 8, (128,) * 16,
                                      (1500,) * 16, (0.25,) * 16, "none"),
        "large-bf16-b1-k8": Workload("large-bf16-b1-k8", LARGE, 1, 8, (224,), (1500,), (0.2,), "always"),
        "large-bf16-b64-k6": Workload("large-bf16-b64-k6", LARGE, 64, 6, c4_out, c4_enc, c4_err, "none"),
    }
    for k in (2, 4, 8, 16):
        for p in (0.05, 0.2, 0.5, 0.8):
            name = f"small-bf16-b32-k{k}-p{p:g}"
            cfgs[name] = Workload(name, SMALL, 32, k, (128,) * 32, (1500,) * 32, (p,) * 32, "half")
    return cfgs


CONFIGS: Dict[str, Workload] = _make_configs()


def scaled(w: Workload, **kw) -> Workload:
    """A copy of ``w`` with some fields replaced (smaller test cases)."""
    return dataclasses.replace(w, **kw)


# ----------------------------------------------------------------------------
# Weights
# ----------------------------------------------------------------------------

def layer_tensors(dims: ModelDims) -> List[Tuple[str, Tuple[int, ...]]]:
    """Per-layer tensors in blob order (Whisper decoder block, pre-LN)."""
    d, f = dims.d_model, dims.d_ffn
    return [
        ("ln1_g", (d,)), ("ln1_b", (d,)),
        ("wq", (d, d)), ("bq", (d,)), ("wk", (d, d)), ("wv", (d, d)), ("bv", (d,)),
        ("wo", (d, d)), ("bo", (d,)),
        ("ln2_g", (d,)), ("ln2_b", (d,)),
        ("wcq", (d, d)), ("bcq", (d,)), ("wck", (d, d)), ("wcv", (d, d)), ("bcv", (d,)),
        ("wco", (d, d)), ("bco", (d,)),
        ("ln3_g", (d,)), ("ln3_b", (d,)),
        ("w1", (f, d)), ("b1", (f,)), ("w2", (d, f)), ("b2", (d,)),
    ]


def weight_layout(dims: ModelDims) -> Dict[str, Tuple[int, Tuple[int, ...]]]:
    """Name -> (offset in floats, shape) for the flat fp32 weight blob.

    Order: tok_emb [V,d], pos_emb [max_pos,d], then for each layer the tensors
    of ``layer_tensors`` with names prefixed ``L{l}.``, then lnf_g, lnf_b.
    Matrices are [out_features, in_features], row-major.
    """
    out: Dict[str, Tuple[int, Tuple[int, ...]]] = {}
    off = 0

    def put(name, shape):
        nonlocal off
        out[name] = (off, shape)
        off += int(np.prod(shape))

    put("tok_emb", (dims.vocab, dims.d_model))
    put("pos_emb", (dims.max_pos, dims.d_model))
    for l in range(dims.n_layers):
        for name, shape in layer_tensors(dims):
            put(f"L{l}.{name}", shape)
    put("lnf_g", (dims.d_model,))
    put("lnf_b", (dims.d_model,))
    out["__total__"] = (off, ())
    return out


def blob_size(dims: ModelDims) -> int:
    return weight_layout(dims)["__total__"][0]


def bf16_round(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 (ties to even), kept as float32."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def make_weights(dims: ModelDims, seed: int = SEED_WEIGHTS, std: float = 0.02) -> np.ndarray:
    """Random-init weight blob: every entry std * N(0,1); LayerNorm gains 1 + that.

    std = 0.02 is the workloads' initialisation; small test models use a larger
    std so that their greedy transcripts do not lock onto one repeated token.
    bf16 models get their values rounded to bf16 once, here, so that every
    consumer reads identical parameters.
    """
    n = blob_size(dims)
    rng = np.random.default_rng(seed)
    blob = rng.standard_normal(n, dtype=np.float32)
    blob *= np.float32(std)
    lay = weight_layout(dims)
    for name, (off, shape) in lay.items():
        if name.endswith("_g"):
            blob[off:off + shape[0]] += np.float32(1.0)
    if dims.dtype == "bf16":
        chunk = 1 << 26
        for s in range(0, n, chunk):
            blob[s:s + chunk] = bf16_round(blob[s:s + chunk])
    return blob


# ----------------------------------------------------------------------------
# The one-block draft (random init): layout and the target layers it reads
# ----------------------------------------------------------------------------

def draft_taps(dims: ModelDims) -> List[int]:
    """The four target layers whose outputs (the residual stream after the
    layer) the draft combines (App. "Draft architecture": four frozen target
    representations): evenly spaced, the last one the final layer."""
    L = dims.n_layers
    return [max(0, (i + 1) * L // 4 - 1) for i in range(4)]


def draft_ffn(dims: ModelDims) -> int:
    """The draft's feed-forward width: twice its hidden width, as both of the
    paper's draft configurations (1024 / 2048 and 2048 / 4096)."""
    return 2 * dims.d_model


def draft_weight_layout(dims: ModelDims) -> Dict[str, Tuple[int, Tuple[int, ...]]]:
    """Name -> (offset, shape) of the draft's fp32 blob: the input combination
    w_in [d, 4d], b_in, one pre-LN decoder block (the target block's tensors,
    feed-forward width draft_ffn), and its final LayerNorm.  Token and position
    embeddings and the LM head are the target's (frozen)."""
    d = dims.d_model
    ddims = dataclasses.replace(dims, d_ffn=draft_ffn(dims))
    out: Dict[str, Tuple[int, Tuple[int, ...]]] = {}
    off = 0

    def put(name, shape):
        nonlocal off
        out[name] = (off, shape)
        off += int(np.prod(shape))

    put("w_in", (d, 4 * d))
    put("b_in", (d,))
    for name, shape in layer_tensors(ddims):
        put(name, shape)
    put("lnf_g", (d,))
    put("lnf_b", (d,))
    out["__total__"] = (off, ())
    return out


def make_draft_weights(dims: ModelDims, seed: int = SEED_DRAFT, std: float = 0.02) -> np.ndarray:
    """Random-init draft blob, drawn like the target's (std * N(0,1),
    LayerNorm gains 1 + that, bf16-rounded once for bf16 models)."""
    lay = draft_weight_layout(dims)
    n = lay["__total__"][0]
    rng = np.random.default_rng(seed)
    blob = rng.standard_normal(n, dtype=np.float32) * np.float32(std)
    for name, (off, shape) in lay.items():
        if name.endswith("_g"):
            blob[off:off + shape[0]] += np.float32(1.0)
    if dims.dtype == "bf16":
        blob = bf16_round(blob)
    return blob


def weight_view(dims: ModelDims, blob: np.ndarray, name: str) -> np.ndarray:
    off, shape = weight_layout(dims)[name]
    return blob[off:off + int(np.prod(shape))].reshape(shape)


# ----------------------------------------------------------------------------
# Utterance inputs
# ----------------------------------------------------------------------------

def make_encoder_states(dims: ModelDims, enc_lens: Sequence[int], t_max: int,
                        seed: int = SEED_ENCODER) -> np.ndarray:
    """Encoder output states [B, t_max, d], N(0,1); frames >= enc_lens[b] are zero."""
    B = len(enc_lens)
    out = np.zeros((B, t_max, dims.d_model), dtype=np.float32)
    for b, T in enumerate(enc_lens):
        rng = np.random.default_rng([seed, b])
        x = rng.standard_normal((T, dims.d_model), dtype=np.float32)
        out[b, :T] = bf16_round(x) if dims.dtype == "bf16" else x
    return out


def make_prompt(dims: ModelDims, batch: int, length: int = PROMPT_LEN,
                seed: int = SEED_PROMPT) -> np.ndarray:
    """One fixed prompt of token ids, repeated for every utterance: [B, P0] int32."""
    rng = np.random.default_rng(seed)
    p = rng.integers(0, dims.vocab, size=length).astype(np.int32)
    return np.tile(p, (batch, 1))


# ----------------------------------------------------------------------------
# Synthetic drafts
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Corruption:
    """Draft-corruption stream indexed by (utterance, round start position, depth).

    repl[b, P, i] >= 0 replaces draft i+1 of a round that starts at committed
    length P by that token id; -1 keeps the true token.  shift[b, P] = s > 0
    makes drafts at depth i >= s lag the truth by one position (a one-token
    slip); 0 means no slip.
    """
    repl: np.ndarray   # [B, max_pos, k] int32
    shift: np.ndarray  # [B, max_pos] int32


def make_corruption(w: Workload, seed: int = SEED_CORRUPT) -> Corruption:
    B, P, k, V = w.batch, w.dims.max_pos, w.k, w.dims.vocab
    repl = np.full((B, P, k), -1, dtype=np.int32)
    shift = np.zeros((B, P), dtype=np.int32)
    for b in range(B):
        rng = np.random.default_rng([seed, b])
        hit = rng.random((P, k)) < w.err[b]
        tok = rng.integers(0, V, size=(P, k)).astype(np.int32)
        repl[b] = np.where(hit, tok, -1)
        s = rng.integers(1, k + 1, size=P).astype(np.int32)
        if w.shift == "always":
            shift[b] = s
        elif w.shift == "half":
            shift[b] = np.where(rng.random(P) < 0.5, s, 0)
    return Corruption(repl, shift)


def round_lens(total_len: Sequence[int], kv_len: Sequence[int], k: int) -> np.ndarray:
    """Drafts offered this round: -1 once an utterance has all its tokens, else
    min(k, N - P - 2) so that a fully accepted round ends exactly at N tokens."""
    out = np.empty(len(total_len), dtype=np.int32)
    for b, (N, P) in enumerate(zip(total_len, kv_len)):
        out[b] = -1 if P + 1 >= N else min(k, N - P - 2)
    return out


def make_drafts(truth: np.ndarray, total_len: Sequence[int], kv_len: Sequence[int],
                k: int, corr: Optional[Corruption]) -> Tuple[np.ndarray, np.ndarray]:
    """Drafts for one round from a reference transcript.

    truth[b, j] is token j of utterance b's reference sequence (prompt included).
    Draft i (1-based) of a round at committed length P is truth[P + i], or
    truth[P + i - 1] when a slip s <= i is active, or the corruption token.
    Returns draft [B, k] (unused slots 0) and lens [B].
    """
    B = truth.shape[0]
    lens = round_lens(total_len, kv_len, k)
    draft = np.zeros((B, k), dtype=np.int32)
    for b in range(B):
        P = int(kv_len[b])
        for i in range(1, int(lens[b]) + 1):
            j = P + i
            if corr is not None and corr.shift[b, P] > 0 and i >= corr.shift[b, P]:
                j -= 1
            t = int(truth[b, j])
            if corr is not None and corr.repl[b, P, i - 1] >= 0:
                t = int(corr.repl[b, P, i - 1])
            draft[b, i - 1] = t
    return draft, lens
