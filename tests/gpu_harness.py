"""Upload a harness Case to the GPU, run kvx_translate through the C ABI, and
bring the target cache back in the oracle's layout [L_t, H_t, T_total, d_t]."""
from __future__ import annotations

from typing import Optional

import numpy as np
import torch

import paper_2608_30963_gb300 as kvx
from paper_2608_30963_gb300 import synth

from harness import Case


def to_dev(x: np.ndarray, dtype: str, device="cuda") -> torch.Tensor:
    if dtype == "bf16":
        bits = synth.f32_to_bf16_bits(x).view(np.int16)
        return torch.from_numpy(bits).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(device)


def to_host(t: torch.Tensor) -> np.ndarray:
    if t.dtype == torch.bfloat16:
        return synth.bf16_bits_to_f32(t.view(torch.int16).cpu().numpy().view(np.uint16))
    return t.float().cpu().numpy()


def i32(x, device="cuda") -> Optional[torch.Tensor]:
    return None if x is None else torch.from_numpy(np.ascontiguousarray(x, np.int32)).to(device)


class DeviceCase:
    def __init__(self, c: Case, path: int = kvx.KVX_PATH_AUTO, paged: Optional[bool] = None,
                 explicit_layer_map: bool = True, fill=float("nan"), max_position: int = 0):
        self.c = c
        s = c.spec
        self.dtype = s.dtype
        tdt = torch.bfloat16 if s.dtype == "bf16" else torch.float32
        kdt = kvx.KVX_BF16 if s.dtype == "bf16" else kvx.KVX_FP32
        lr = None if c.low_rank is None else tuple(to_dev(a, s.dtype) for a in c.low_rank)
        self.tr = kvx.Translator(s.src, s.dst, None if lr else to_dev(c.w_k, s.dtype),
                                 None if lr else to_dev(c.w_v, s.dtype),
                                 layer_map=c.layer_map.tolist() if explicit_layer_map else None,
                                 dtype=kdt, path=path, max_position=max_position, form=s.form,
                                 layers_per_target=s.layers_per_target, low_rank=lr)
        wl = c.wl
        any_l = next(iter(c.src_k))
        self.src_k_dev = {l: to_dev(c.src_k[l], s.dtype) for l in c.src_k}
        self.src_v_dev = {l: to_dev(c.src_v[l], s.dtype) for l in c.src_v}
        self.src_k = [self.src_k_dev.get(l, self.src_k_dev[any_l]) for l in range(s.src.num_layers)]
        self.src_v = [self.src_v_dev.get(l, self.src_v_dev[any_l]) for l in range(s.src.num_layers)]
        self.src_len = i32(wl.src_len)
        self.seq_off = i32(wl.tgt_seq_off)
        self.span_lo, self.span_hi = i32(wl.span_lo), i32(wl.span_hi)
        self.src_pos = i32(None if c.src_pos is None else c.src_pos.reshape(-1))
        self.tgt_pos = i32(c.tgt_pos)
        self.paged = s.paged if paged is None else paged
        Lt, Ht, dt = s.dst.num_layers, s.dst.num_kv_heads, s.dst.head_dim
        if self.paged:
            if wl.page_table is None:
                P = s.page_size
                pages = [(int(t) + P - 1) // P for t in wl.tgt_len]
                wl.num_pages, wl.max_pages = sum(pages), max(pages)
                perm = np.random.default_rng(6).permutation(wl.num_pages).astype(np.int32)
                pt = np.full((wl.batch, wl.max_pages), -1, np.int32)
                k = 0
                for b, n in enumerate(pages):
                    pt[b, :n] = perm[k:k + n]; k += n
                wl.page_table = pt
            self.page_table = i32(wl.page_table)
            shape = (wl.num_pages, s.page_size, Ht, dt)
        else:
            self.page_table = None
            shape = (wl.batch, Ht, max(wl.t_max, 1), dt)
        self.dst_k = [torch.full(shape, fill, dtype=tdt, device="cuda") for _ in range(Lt)]
        self.dst_v = [torch.full(shape, fill, dtype=tdt, device="cuda") for _ in range(Lt)]

    def run(self, stream=None):
        wl = self.c.wl
        self.tr.translate(self.src_k, self.src_v, self.src_len, self.seq_off, wl.total_tgt, self.dst_k, self.dst_v,
                          span_lo=self.span_lo, span_hi=self.span_hi, src_pos=self.src_pos, tgt_pos=self.tgt_pos,
                          page_table=self.page_table, page_size=self.c.spec.page_size,
                          num_pages=wl.num_pages if self.paged else 0, stream=stream)

    def gather_layer(self, j: int, kv: int) -> np.ndarray:
        """Target layer j as [H_t, T_total, d_t] float32."""
        wl = self.c.wl
        t = to_host((self.dst_k if kv == 0 else self.dst_v)[j])
        out = []
        for b in range(wl.batch):
            T = int(wl.tgt_len[b])
            if self.paged:
                P = self.c.spec.page_size
                idx = np.arange(T)
                rows = t[wl.page_table[b, idx // P], idx % P]          # [T, Ht, dt]
                out.append(rows.transpose(1, 0, 2))
            else:
                out.append(t[b, :, :T])
        return np.concatenate(out, axis=1)

    def gather(self):
        s = self.c.spec
        return (np.stack([self.gather_layer(j, 0) for j in range(s.dst.num_layers)]),
                np.stack([self.gather_layer(j, 1) for j in range(s.dst.num_layers)]))

    def row(self, j, h, kv, tp) -> np.ndarray:
        wl = self.c.wl
        b = int(np.searchsorted(wl.tgt_seq_off, tp, side="right") - 1)
        while wl.tgt_seq_off[b + 1] <= tp:
            b += 1
        t = tp - int(wl.tgt_seq_off[b])
        ten = (self.dst_k if kv == 0 else self.dst_v)[j]
        if self.paged:
            P = self.c.spec.page_size
            return to_host(ten[int(wl.page_table[b, t // P]), t % P, h])
        return to_host(ten[b, h, t])

    def status(self) -> int:
        return self.tr.device_status()
