"""Decoder weights as one file (host IO only; no device code): a JSON header and the raw bf16
tensors, so that checkpoint weights converted to bf16 could replace the seeded random ones."""
from __future__ import annotations

import torch

WEIGHTS_MAGIC = "RIFT-WEIGHTS-1"
LAYER_TENSORS = ("wq", "wk", "wv", "wo", "wg", "wu", "wd", "g_attn", "g_ffn")


def save_weights(path, dims: dict, layers: list, g_final: torch.Tensor, lm_head: torch.Tensor | None = None):
    """A decoder's weights as one file: a JSON header line (magic, dims, tensor names, shapes and
    byte offsets), then every tensor's raw bf16 bytes in header order (layers' wq, wk, wv, wo, wg,
    wu, wd, g_attn, g_ffn; g_final; lm_head if given).  Shapes follow the LLaMA convention (out x
    in), so checkpoint tensors converted to bf16 can be written the same way."""
    import json
    names, tensors = [], []
    for l, W in enumerate(layers):
        for k in LAYER_TENSORS:
            names.append(f"layers.{l}.{k}")
            tensors.append(W[k])
    names.append("g_final")
    tensors.append(g_final)
    if lm_head is not None:
        names.append("lm_head")
        tensors.append(lm_head)
    entries, off = [], 0
    for n, t in zip(names, tensors):
        nbytes = t.numel() * 2
        entries.append({"name": n, "shape": list(t.shape), "offset": off, "bytes": nbytes})
        off += nbytes
    header = json.dumps({"magic": WEIGHTS_MAGIC, "dtype": "bf16", "dims": dims, "tensors": entries}).encode()
    with open(path, "wb") as f:
        f.write(len(header).to_bytes(8, "little"))
        f.write(header)
        for t in tensors:
            f.write(t.detach().to("cpu", torch.bfloat16).contiguous().view(torch.int16).numpy().tobytes())


def load_weights(path):
    """(dims, layers, g_final, lm_head or None) from a save_weights file, as CPU bf16 tensors."""
    import json
    import numpy as np
    with open(path, "rb") as f:
        hlen = int.from_bytes(f.read(8), "little")
        header = json.loads(f.read(hlen))
        if header.get("magic") != WEIGHTS_MAGIC or header.get("dtype") != "bf16":
            raise ValueError(f"{path}: not a {WEIGHTS_MAGIC} bf16 weights file")
        blob = f.read()
    out = {}
    for e in header["tensors"]:
        raw = np.frombuffer(blob, dtype=np.int16, count=e["bytes"] // 2, offset=e["offset"])
        out[e["name"]] = torch.from_numpy(raw.copy()).view(torch.bfloat16).view(*e["shape"])
    n_layers = header["dims"]["n_layers"]
    layers = [{k: out[f"layers.{l}.{k}"] for k in LAYER_TENSORS} for l in range(n_layers)]
    return header["dims"], layers, out["g_final"], out.get("lm_head")
