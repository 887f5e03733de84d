#!/usr/bin/env python
"""Benchmark of the QSVD latent-attention hot path (arxiv 2510.16292) on GB300.

One step = one pass of the whole path over the LLaVA-7B-shaped layer
(d=4096, H=32, dh=128, r=1536): prefill of 640 tokens (576 image-like + 64
text-like; per-token int8 X, exact int8 GEMM with W_d, per-token latent
requantization fused into the cache store), then 128 decode steps (project
the new token, append it, attend over the int8 latent cache with U_k absorbed
and U_v applied last).  Inputs are seeded synthetic arrays resident in HBM
before timing.  L2 is flushed (a 256 MiB read) before the prefill and before
every decode step; the flush sits outside the timed intervals, which are CUDA
events on the launching stream around each sub-step.

value = decode tokens/s (all ranks' tokens / max-over-ranks decode time).
Secondary figures: prefill TOPS (2*T*d*r over the projection call), latent
cache GB/s, the decode step's fraction of its HBM roofline, and the causal
prefill attention of the 7B prompt and the 13B batch (tokens/s and per-kernel
fractions of the bf16 tensor peak, both entry points).

--impl reference times the CPU oracle (the plain fp64 definition) on a
bounded sample of the same workload on the host cores.
"""
from __future__ import annotations

import argparse
import ctypes
import dataclasses
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synthetic  # noqa: E402

METRIC = "decode tokens/s + latent-cache HBM GB/s; prefill int8 TOPS (LLaVA-7B shape)"
WORKLOAD = "llava7b"
FLUSH_BYTES = 256 << 20
L2_BYTES = 129 << 20          # GB300 L2 (the rotation's sizing)


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["native", "reference"], default="native")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-prefill13", action="store_true")
    p.add_argument("--no-prefill-attn", action="store_true")
    p.add_argument("--importance-probe", action="store_true",
                   help="only time the Eq. 10 importance scores of one 7B-shaped layer and print one line")
    p.add_argument("--beta-probe", action="store_true",
                   help="only time one beta of the Eq. 14 search on a 7B-shaped layer and print one line")
    p.add_argument("--u-bits", type=int, default=0, choices=[0, 8, 4],
                   help="quantize U_q, U_k, U_v per output channel to int8 or int4 (Eq. 11) and run decode "
                        "attention on the codes (qsvd_latent_decode_attn_qu); 0: bf16 up-projections")
    p.add_argument("--attn-path", type=int, default=0, choices=[0, 1, 2, 3],
                   help="decode attention kernel choice (qsvd_set_decode_attn_path): 0 automatic, 1 CUDA cores, "
                        "2 tcgen05, 3 warp-level MMA")
    p.add_argument("--decode-call", choices=["step", "pair"], default="pair",
                   help="decode API: one qsvd_decode_step call per token (step) or qsvd_latent_project + "
                        "qsvd_latent_decode_attn (pair)")
    p.add_argument("--rot", action="store_true",
                   help="rotate X by H1 on the fly (Eq. 12; weights quantized as H1 W_d) in every projection")
    p.add_argument("--prefill-probe", action="store_true",
                   help="only time causal prefill attention and print one line per shape and path")
    p.add_argument("--prefill-shapes", default=",".join(PREFILL_REPORTED), help="shapes of --prefill-probe")
    p.add_argument("--prefill-paths", default="blocks,rows", help="paths of --prefill-probe")
    p.add_argument("--prefill-sweep", default=None, metavar="ROWS,...",
                   help="only time causal prefill attention for these rows-per-group settings (0 = automatic)")
    # the tiny layer's W_d and U come from the oracle's joint SVD: it is a parity case (tests/), not a benchmark
    p.add_argument("--workload", default=WORKLOAD, choices=sorted(k for k in synthetic.WORKLOADS if k != "tiny"))
    p.add_argument("--decode-steps", type=int, default=0, help="override the workload's decode steps")
    p.add_argument("--sweep", choices=["quick", "full", "point"], default=None,
                   help="sweep the 7B-shaped layer over rank, cached length, batch and cache precision (one JSON "
                        "line per point) instead of the benchmark; 'point' runs the one point of --sweep-point")
    p.add_argument("--sweep-point", default="1536,4096,16,4", metavar="R,L,B,BITS",
                   help="rank, cached length, batch, cache bits of --sweep point")
    p.add_argument("--l2", default="rotate", choices=["rotate", "flush"],
                   help="cold-L2 method: rotate through copies of the layer larger than L2 together, or flush "
                        "L2 before every sub-step")
    return p.parse_args()


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def workload_desc(wl):
    s = wl.shape
    return (f"{wl.name}: d={s.d} H={s.H} dh={s.dh} r={s.r}, B={wl.B}, prefill {wl.n_image} image-like + "
            f"{wl.n_text} text-like tokens, {wl.decode_steps} decode steps, int{wl.lat_bits} latent cache")


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                rows.append(f)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------
# native arm
# ---------------------------------------------------------------------------
class NativeLayer:
    """One independently seeded copy of the layer: weights, latent cache, inputs."""

    def __init__(self, nb, inp, X_from=None):
        torch, q, wl, dev = nb.torch, nb.q, nb.wl, nb.dev
        s = wl.shape

        def bf16(bits):
            a = np.ascontiguousarray(bits).view(np.int16)
            return torch.from_numpy(a).view(torch.bfloat16).to(dev)

        rot = (s.d & -s.d) if nb.rot else 0             # H1 on the fly: the largest power-of-two block
        self.W = q.qsvd_quantize_weight(torch.from_numpy(inp.W_d.astype(np.float32)).to(dev), rot=rot)
        self.U = [bf16(u) for u in (inp.U_q, inp.U_k, inp.U_v)]
        # Eq. 11's Q(W^u): the decode step reads the codes instead of the bf16 values
        self.UQ = [q.qsvd_quantize_up(u, nb.u_bits) for u in self.U] if nb.u_bits else None
        if X_from is None:
            self.Xp = bf16(inp.X_prefill.reshape(wl.B * wl.prefill, s.d))
            self.Xd = bf16(inp.X_decode)                   # [S, B, d]
        else:                                              # inputs shared with another copy
            self.Xp, self.Xd = X_from.Xp, X_from.Xd
        self.cache = q.LatentCache.empty(wl.B, wl.tmax, s.r, wl.lat_bits, dev)
        self.O = torch.empty((wl.B, s.d), dtype=torch.float32, device=dev)


class NativeBench:
    """The layer step on the GPU.  L2 method `rotate` (default): K independently
    seeded copies of the layer whose weights and caches together exceed twice
    the L2, and every decode token runs through all K in turn, as in a stack of
    layers: each layer's data comes from HBM while the kernels' code stays
    cached, as it does in serving.  `flush`: one copy, L2 evicted by a 256 MiB
    read before every sub-step (code cold as well)."""

    def __init__(self, wl, rank, l2="rotate", rot=False, u_bits=0, decode_call="pair"):
        import torch
        import paper_2510_16292_gb300 as q
        self.torch, self.q, self.wl, self.rot, self.u_bits = torch, q, wl, rot, u_bits
        s = wl.shape
        self.dev = torch.device("cuda", torch.cuda.current_device())
        dev = self.dev
        B, P, S = wl.B, wl.prefill, wl.decode_steps
        self.B, self.P, self.S = B, P, S
        self.l2 = l2
        tok = (s.r + 4) if wl.lat_bits == 8 else (s.r // 2 + 2 * (s.r // 128))
        layer_bytes = 3 * self.up_bytes() + s.r * s.d + B * wl.tmax * tok      # what a decode step reads
        self.K = 1 if l2 == "flush" else max(2, min(16, -(-2 * L2_BYTES // layer_bytes)))
        self.layer_bytes = layer_bytes
        self.layers = []
        for k in range(self.K):
            share = k > 0 and B * P * s.d * 2 > L2_BYTES // 2      # large inputs cannot stay cached anyway
            inp = synthetic.gen_layer(wl, seed=rank * 64, layer=k, prefill_rows=0 if share else None,
                                      decode_steps=0 if share else None)
            self.layers.append(NativeLayer(self, inp, X_from=self.layers[0] if share else None))
        L0 = self.layers[0]
        self.W, self.U, self.cache, self.Xp, self.Xd, self.O = L0.W, L0.U, L0.cache, L0.Xp, L0.Xd, L0.O
        i32 = lambda a: torch.as_tensor(np.asarray(a, dtype=np.int32), device=dev)  # noqa: E731
        self.pseq = i32(np.repeat(np.arange(B), P))
        self.ppos = i32(np.tile(np.arange(P), B))
        self.dseq = i32(np.arange(B))
        self.dpos = [i32(np.full(B, P + t)) for t in range(S)]
        self.dlen = [i32(np.full(B, P + t + 1)) for t in range(S)]
        # one workspace of each kind: the calls run one after another on one stream
        self.wsp = torch.zeros(q.qsvd_project_workspace_bytes(B * P, s.d, s.r), dtype=torch.uint8, device=dev)
        self.wsd = torch.zeros(q.qsvd_decode_workspace_bytes(B, wl.tmax, s.r, s.H, s.dh), dtype=torch.uint8,
                               device=dev)
        # "step": one qsvd_decode_step call per token; "pair": qsvd_latent_project + qsvd_latent_decode_attn
        self.fused = decode_call == "step"
        self.wsf = torch.zeros(max(1, q.qsvd_decode_step_workspace_bytes(B, wl.tmax, s.d, s.r, s.H, s.dh)),
                               dtype=torch.uint8, device=dev)
        self.flushbuf = torch.ones(FLUSH_BYTES // 4 if l2 == "flush" else 1, dtype=torch.float32, device=dev)
        self.flush_out = torch.zeros((), dtype=torch.float32, device=dev)
        self.stream = torch.cuda.current_stream()
        self._marshal()

    def up_bytes(self):
        """Bytes of one up-projection as the decode step reads it: bf16 values,
        or int8 / int4 codes plus one fp32 scale per output channel."""
        s = self.wl.shape
        return s.r * s.d * 2 if not self.u_bits else s.r * s.d * self.u_bits // 8 + 4 * s.d

    def _marshal(self, stream=None):
        """Pre-build the ctypes argument tuples of every C-ABI call of a step,
        bound to `stream` (default: the current stream)."""
        q, wl, s = self.q, self.wl, self.wl.shape
        lib = q._lib
        self.lib = lib
        st = (stream or self.stream).cuda_stream
        self.pre_args, self.dec_proj, self.dec_attn, self.dec_fused = [], [], [], []
        for L in self.layers:
            L.cW, L.cC = L.W._c(), L.cache._c()
            L.cU = [u._c() for u in L.UQ] if L.UQ else None
            self.pre_args.append((ctypes.byref(L.cW), L.Xp.data_ptr(), self.B * self.P, 1.0, wl.lat_bits, 1.0,
                                  None, None, ctypes.byref(L.cC), self.pseq.data_ptr(), self.ppos.data_ptr(),
                                  None, None, None, self.wsp.data_ptr(), self.wsp.numel(), st))
            proj, attn, fused = [], [], []
            for t in range(self.S):
                proj.append((ctypes.byref(L.cW), L.Xd[t].data_ptr(), self.B, 1.0, wl.lat_bits, 1.0,
                             None, None, ctypes.byref(L.cC), self.dseq.data_ptr(), self.dpos[t].data_ptr(),
                             None, None, None, self.wsp.data_ptr(), self.wsp.numel(), st))
                ups = ([ctypes.byref(u) for u in L.cU] if L.cU else
                       [L.U[0].data_ptr(), L.U[1].data_ptr(), L.U[2].data_ptr()])
                attn.append((ctypes.byref(L.cC), self.dlen[t].data_ptr(), self.P + t + 1, *ups, s.H, s.dh,
                             1.0 / math.sqrt(s.dh), L.O.data_ptr(), self.wsd.data_ptr(), self.wsd.numel(), st))
                fused.append((ctypes.byref(L.cW), L.Xd[t].data_ptr(), ctypes.byref(L.cC),
                              self.dlen[t].data_ptr(), self.P + t + 1, L.U[0].data_ptr(),
                              L.U[1].data_ptr(), L.U[2].data_ptr(), s.H, s.dh, 1.0, 1.0,
                              1.0 / math.sqrt(s.dh), L.O.data_ptr(), self.wsf.data_ptr(),
                              self.wsf.numel(), st))
            self.dec_proj.append(proj)
            self.dec_attn.append(attn)
            self.dec_fused.append(fused)

    def build_graph(self):
        """Capture one whole step (flushes, sub-step events and every C-ABI
        call) into a CUDA graph; replaying it removes host launch overhead."""
        torch = self.torch
        gs = torch.cuda.Stream()
        self._marshal(stream=gs)
        E = lambda: torch.cuda.Event(enable_timing=True, external=True)  # noqa: E731
        self.gevs = [(E(), E()) for _ in range(self.S + 1)]
        gs.wait_stream(self.stream)
        with torch.cuda.stream(gs):
            self.run_step(self.make_events(), gs)          # eager warm-up on the capture stream
        gs.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=gs):
            self.run_step(self.gevs, gs)
        torch.cuda.synchronize()
        self.graph = g
        self._marshal()                                    # eager calls go back to the default stream

    def _call(self, fn, args):
        stt = fn(*args)
        if stt != 0:
            raise RuntimeError(f"qsvd status {stt}: {self.lib.qsvd_last_error().decode()}")

    def prefill(self):
        for k in range(self.K):
            self._call(self.lib.qsvd_latent_project, self.pre_args[k])

    def decode(self, t):
        """Decode token t through every copy of the layer."""
        for k in range(self.K):
            if self.fused:
                self._call(self.lib.qsvd_decode_step, self.dec_fused[k][t])
            else:
                self._call(self.lib.qsvd_latent_project, self.dec_proj[k][t])
                self._call(self.lib.qsvd_latent_decode_attn_qu if self.u_bits else self.lib.qsvd_latent_decode_attn,
                           self.dec_attn[k][t])

    def flush(self):
        """`flush` method: evict L2 by reading a 256 MiB buffer (an fp32 sum in
        place, so no temporary is written and L2 is left clean; dirty lines
        would slow the next reads with write-backs).  `rotate`: nothing."""
        if self.l2 == "flush":
            self.torch.sum(self.flushbuf, dim=(0,), out=self.flush_out)

    def run_step(self, evs, stream=None):
        """evs: list of (start, end) event pairs, one per sub-step (prefill, decode 0..S-1)."""
        st = stream or self.stream
        self.flush()
        evs[0][0].record(st)
        self.prefill()
        evs[0][1].record(st)
        for t in range(self.S):
            self.flush()
            evs[t + 1][0].record(st)
            self.decode(t)
            evs[t + 1][1].record(st)

    def replay(self):
        self.graph.replay()
        return self.gevs

    def make_events(self):
        E = self.torch.cuda.Event
        return [(E(enable_timing=True), E(enable_timing=True)) for _ in range(self.S + 1)]

    # ---- kernel-level profile (CUDA events the library records between its kernels) ----
    def profile(self, steps=1):
        torch = self.torch
        n = steps * self.K * (self.S * 12 + 8)
        events = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
        for e in events:            # torch creates the CUDA event lazily, on first record
            e.record(self.stream)
        torch.cuda.synchronize()
        handles = (ctypes.c_void_p * n)(*[ctypes.c_void_p(e.cuda_event) for e in events])
        ctx = []          # sub-step of each recorded event
        lib = self.lib
        lib.qsvd_profile_count.restype = ctypes.c_int32
        lib.qsvd_profile_label.restype = ctypes.c_char_p
        lib.qsvd_profile_events(handles, n)
        try:
            for _ in range(steps):
                self.flush()
                c0 = lib.qsvd_profile_count()
                self.prefill()
                ctx += [("prefill", None)] * (lib.qsvd_profile_count() - c0)
                for t in range(self.S):
                    self.flush()
                    c0 = lib.qsvd_profile_count()
                    self.decode(t)
                    ctx += [("decode", t)] * (lib.qsvd_profile_count() - c0)
            torch.cuda.synchronize()
            cnt = lib.qsvd_profile_count()
            labels = [lib.qsvd_profile_label(i).decode() for i in range(cnt)]
        finally:
            lib.qsvd_profile_events(None, 0)
        launches = []
        for i in range(1, cnt):
            if labels[i] == "begin":
                continue
            launches.append((labels[i], ctx[i], events[i - 1].elapsed_time(events[i]) * 1e-3))
        return launches

    def alg_bytes(self, label, ctx):
        """Minimal HBM bytes of one launch: every input read once, every output written once."""
        s, B, P = self.wl.shape, self.B, self.P
        d, r, H = s.d, s.r, s.H
        tok = r if self.wl.lat_bits == 8 else r // 2 + 2 * (r // 128)
        stok = 4 if self.wl.lat_bits == 8 else 0
        T = B * P if ctx[0] == "prefill" else B
        L = P + ctx[1] + 1 if ctx[0] == "decode" else 0
        if label == "xquant":
            return T * d * 2 + T * d + 4 * T
        if label == "proj_dp4a":
            return r * d + T * d + 4 * r + 4 * T + 4 * T * r
        if label == "proj_small":
            # W_d codes and scales, X (bf16) in; the requantized latent rows out
            return r * d + 4 * r + 2 * T * d + T * (tok + stok)
        if label == "requant":
            return 4 * T * r + T * (tok + stok) + 8 * T
        ub = self.up_bytes()
        if label == "qproj":
            return ub + B * (tok + stok) + 4 * B * d
        if label == "qabsorb":
            return ub + 4 * B * d + 4 * B * H * r
        if label in ("attn_chunk", "attn_tc", "attn_mma"):
            return B * L * (tok + stok) + 4 * B * H * r
        if label == "combine_uv":
            return ub + 4 * B * d
        if label == "decode_step":
            return self.step_roofline_bytes(ctx[1])
        return 0

    def step_roofline_bytes(self, t):
        """Bytes one decode step must move (per the path's definition): cache read,
        append, U_q/U_k/U_v, W_d codes and scales, x in, O out."""
        s, B = self.wl.shape, self.B
        d, r = s.d, s.r
        tok = (r + 4) if self.wl.lat_bits == 8 else (r // 2 + 2 * (r // 128))
        L = self.P + t + 1
        return B * L * tok + B * tok + 3 * self.up_bytes() + d * r + 4 * r + B * d * 2 + 4 * B * d

    # ---- end to end through the public binding with host buffers ----
    def e2e(self, steps, warmup):
        """Per decode token: one host -> device copy of the token's X rows for
        the K layer copies, the projection and the decode attention of every
        copy through the Python binding, one device -> host copy of their O
        rows.  Timed twice: as a CUDA graph captured from those binding calls
        and copies (one graph per step, replayed the way a decode loop in a
        server replays it) and eagerly (every call made from Python,
        host-bound).  Returns decode tokens/s of one layer for both and the
        bytes copied per step."""
        torch, q, s, K = self.torch, self.q, self.wl.shape, self.K
        hx_p = [torch.empty(L.Xp.shape, dtype=torch.bfloat16, pin_memory=True) for L in self.layers]
        for L, hp in zip(self.layers, hx_p):
            hp.copy_(L.Xp.cpu())
        hx_d = torch.empty((self.S, K, self.B, s.d), dtype=torch.bfloat16, pin_memory=True)
        for k, L in enumerate(self.layers):
            hx_d[:, k].copy_(L.Xd.cpu())
        hO = torch.empty((self.S, K, self.B, s.d), dtype=torch.float32, pin_memory=True)
        dXp = torch.empty_like(self.Xp)
        dX = torch.empty((K, self.B, s.d), dtype=torch.bfloat16, device=self.dev)
        dO = torch.empty((K, self.B, s.d), dtype=torch.float32, device=self.dev)

        def step(evs):
            self.flush()
            evs[0][0].record()
            for k, L in enumerate(self.layers):
                dXp.copy_(hx_p[k], non_blocking=True)
                q.qsvd_latent_project(L.W, dXp, 1.0, self.wl.lat_bits, 1.0, dst=L.cache, dst_seq=self.pseq,
                                      dst_pos=self.ppos, workspace=self.wsp)
            evs[0][1].record()
            for t in range(self.S):
                self.flush()
                evs[t + 1][0].record()
                dX.copy_(hx_d[t], non_blocking=True)
                for k, L in enumerate(self.layers):
                    if self.fused:
                        q.qsvd_decode_step(L.W, dX[k], L.cache, self.dlen[t], self.P + t + 1, *L.U, s.H, s.dh, dO[k],
                                           workspace=self.wsf)
                        continue
                    q.qsvd_latent_project(L.W, dX[k], 1.0, self.wl.lat_bits, 1.0, dst=L.cache,
                                          dst_seq=self.dseq, dst_pos=self.dpos[t], workspace=self.wsp)
                    if L.UQ:
                        q.qsvd_latent_decode_attn_qu(L.cache, self.dlen[t], self.P + t + 1, *L.UQ, s.H, s.dh, dO[k],
                                                     workspace=self.wsd)
                    else:
                        q.qsvd_latent_decode_attn(L.cache, self.dlen[t], self.P + t + 1, *L.U, s.H, s.dh, dO[k],
                                                  workspace=self.wsd)
                hO[t].copy_(dO, non_blocking=True)
                evs[t + 1][1].record()

        def decode_seconds(evs):
            return sum(a.elapsed_time(b) for a, b in evs[1:]) * 1e-3

        E = torch.cuda.Event
        eager = []
        for it in range(warmup + steps):
            evs = [(E(enable_timing=True), E(enable_timing=True)) for _ in range(self.S + 1)]
            step(evs)
            torch.cuda.synchronize()
            if it >= warmup:
                eager.append(decode_seconds(evs))
        gs = torch.cuda.Stream()
        gs.wait_stream(torch.cuda.current_stream())
        gevs = [(E(enable_timing=True, external=True), E(enable_timing=True, external=True))
                for _ in range(self.S + 1)]
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=gs):
            step(gevs)
        torch.cuda.synchronize()
        graphed = []
        for it in range(warmup + steps):
            g.replay()
            torch.cuda.synchronize()
            if it >= warmup:
                graphed.append(decode_seconds(gevs))
        # bytes copied inside the timed intervals (evs[1:]: the S decode tokens
        # through the K copies); the prefill's X copies are outside them
        h2d = K * self.S * self.B * s.d * 2
        d2h = K * self.S * self.B * s.d * 4
        tokens = self.B * self.S * K
        return tokens / statistics.mean(graphed), tokens / statistics.mean(eager), h2d, d2h


def prefill_gemm_probe(T=24064, d=5120, r=2048, iters=3, w4a4=False):
    """Prefill projection at the LLaVA-13B batch shape (8 x (5 x 576 + 128)
    tokens, d=5120, r=2048): time of the whole qsvd_latent_project call and of
    its tensor-core GEMM kernel (library events), cold L2 before each call.
    Inputs: seeded torch Gaussians (X with the outlier-channel pattern of the
    synthetic recipe), W_d columns scaled by j^-0.5.  w4a4: int4 codes of W_d
    and X on the fp8 (e4m3) tensor-core path, an int4 latent, measured against
    the fp8 peak (the measured bf16 peak times the nominal fp8 / bf16 ratio, 2)."""
    import torch
    import paper_2510_16292_gb300 as q
    dev = torch.device("cuda", torch.cuda.current_device())
    g = torch.Generator(device=dev)
    g.manual_seed(1234)
    X = torch.randn((T, d), generator=g, device=dev)
    X[:, torch.randperm(d, generator=g, device=dev)[: d // 100]] *= 20
    X = X.to(torch.bfloat16)
    Wd = torch.randn((d, r), generator=g, device=dev) / math.sqrt(d)
    Wd *= torch.arange(1, r + 1, device=dev, dtype=torch.float32) ** -0.5
    W = q.qsvd_quantize_weight(Wd.contiguous(), w_bits=4 if w4a4 else 8, x_bits=4 if w4a4 else 8)
    if w4a4:
        lc = torch.empty((T, r // 2), dtype=torch.uint8, device=dev)
        ls = torch.empty((T, r // 128), dtype=torch.float16, device=dev)
    else:
        lc = torch.empty((T, r), dtype=torch.int8, device=dev)
        ls = torch.empty((T,), dtype=torch.float32, device=dev)
    kname = "gemm_f8" if w4a4 else "gemm_tc"
    ws = torch.zeros(q.qsvd_project_workspace_bytes(T, d, r), dtype=torch.uint8, device=dev)
    flush = torch.ones((256 << 20) // 4, dtype=torch.float32, device=dev)
    sink = torch.zeros((), dtype=torch.float32, device=dev)
    n = 16
    events = [torch.cuda.Event(enable_timing=True) for _ in range(n)]
    for e in events:
        e.record()
    torch.cuda.synchronize()
    handles = (ctypes.c_void_p * n)(*[ctypes.c_void_p(e.cuda_event) for e in events])
    lib = q._lib
    lib.qsvd_profile_count.restype = ctypes.c_int32
    lib.qsvd_profile_label.restype = ctypes.c_char_p
    gemm, call = [], []
    for it in range(iters + 1):
        torch.sum(flush, dim=(0,), out=sink)
        lib.qsvd_profile_events(handles, n)
        q.qsvd_latent_project(W, X, lat_bits=4 if w4a4 else 8, lat_codes=lc, lat_scales=ls, workspace=ws)
        torch.cuda.synchronize()
        cnt = lib.qsvd_profile_count()
        labels = [lib.qsvd_profile_label(i).decode() for i in range(cnt)]
        lib.qsvd_profile_events(None, 0)
        if it == 0:
            continue
        gi = labels.index(kname)
        gemm.append(events[gi - 1].elapsed_time(events[gi]) * 1e-3)
        call.append(events[0].elapsed_time(events[cnt - 1]) * 1e-3)
    ops = 2.0 * T * d * r
    _, bf16_peak, kind = peaks()
    g_s, c_s = min(gemm), min(call)
    del X, W, lc, ls, ws, flush
    out = {"shape": f"T={T} d={d} r={r} (8 x 3008 tokens, LLaVA-13B layer)", "gemm_us": round(g_s * 1e6, 2),
           "gemm_tops": round(ops / g_s / 1e12, 1), "gemm_frac_of_bf16_peak": round(ops / g_s / 1e12 / bf16_peak, 4),
           "project_call_us": round(c_s * 1e6, 2), "project_call_tops": round(ops / c_s / 1e12, 1),
           "peak_kind": kind}
    if w4a4:
        out["setting"] = "W4A4 (int4 X and W_d as e4m3, kind::f8f6f4), int4 latent"
        out["gemm_frac_of_fp8_peak"] = round(ops / g_s / 1e12 / (2 * bf16_peak), 4)
        out["fp8_peak_tflops"] = round(2 * bf16_peak, 1)
        out["fp8_peak_kind"] = kind + " bf16 x nominal fp8/bf16 ratio 2"
    return out


PREFILL_SHAPES = {
    # the 7B-shaped prompt (576 image-like + 64 text-like tokens), int8 cache
    "llava7b": dict(d=4096, H=32, dh=128, r=1536, B=1, T=640, bits=8),
    # the 13B-shaped batch (8 prompts of 5 x 576 + 128 tokens), int8 cache
    "llava13b": dict(d=5120, H=40, dh=128, r=2048, B=8, T=3008, bits=8),
    # one prompt of the 13B batch (the size for kernel captures)
    "llava13b_1seq": dict(d=5120, H=40, dh=128, r=2048, B=1, T=3008, bits=8),
}
PREFILL_REPORTED = ("llava7b", "llava13b")


def prefill_attn_probe(name, iters=3, group_rows=0, path="blocks"):
    """Causal prefill attention: every token of B prompts of T tokens attends
    to its own prefix, cold L2 before each call.  path "blocks": one
    qsvd_latent_prefill call over the B prompt blocks (K and V materialised;
    the fp16 [U_q U_k U_v]^T is prepared once, outside the timed region);
    path "rows": one qsvd_latent_prefill_attn call over all B*T query rows
    (the decode kernels' absorbed form).  The cache codes, scales and U are
    seeded torch random values (the time does not depend on them; the parity
    tests check the numbers).  Reports the call's time, tokens/s, and per
    kernel its time share and tensor throughput (algorithmic flops: the
    Q/K/V product 2*L*r*3d per block, causal attention 4*H*dh per visible
    (query, key) pair; the absorbed form 4*H*r per pair) from a separate pass
    with library events between the kernels."""
    import torch
    import paper_2510_16292_gb300 as q
    c = PREFILL_SHAPES[name]
    d, H, dh, r, B, T, bits = (c[k] for k in ("d", "H", "dh", "r", "B", "T", "bits"))
    dev = torch.device("cuda", torch.cuda.current_device())
    g = torch.Generator(device=dev)
    g.manual_seed(4321)
    cache = q.LatentCache.empty(B, T, r, bits, dev)
    if bits == 8:
        cache.codes.copy_(torch.randint(-127, 128, cache.codes.shape, generator=g, device=dev, dtype=torch.int8))
        cache.scales.copy_(torch.rand(cache.scales.shape, generator=g, device=dev) * 0.02 + 0.005)
    else:
        cache.codes.copy_(torch.randint(0, 256, cache.codes.shape, generator=g, device=dev, dtype=torch.uint8))
        cache.scales.copy_((torch.rand(cache.scales.shape, generator=g, device=dev) * 0.2 + 0.05).half())
    U = [(torch.randn((r, H * dh), generator=g, device=dev) / math.sqrt(r)).to(torch.bfloat16) for _ in range(3)]
    n = B * T
    q_seq = torch.arange(B, device=dev, dtype=torch.int32).repeat_interleave(T)
    q_len = torch.arange(1, T + 1, device=dev, dtype=torch.int32).repeat(B)
    O = torch.empty((n, H * dh), dtype=torch.float32, device=dev)
    prev = q.qsvd_set_prefill_group_rows(group_rows)
    try:
        flush = torch.ones((256 << 20) // 4, dtype=torch.float32, device=dev)
        sink = torch.zeros((), dtype=torch.float32, device=dev)
        if path == "blocks":
            blocks = [(b, 0, T) for b in range(B)]
            Ut = q.qsvd_prefill_weights(*U)
            ws = torch.zeros(q.qsvd_latent_prefill_workspace_bytes(blocks, r, H, dh), dtype=torch.uint8, device=dev)
            call = lambda: q.qsvd_latent_prefill(cache, blocks, Ut, H, dh, O, workspace=ws)  # noqa: E731
        else:
            ws = torch.zeros(q.qsvd_prefill_workspace_bytes(n, T, r, H, dh), dtype=torch.uint8, device=dev)
            call = lambda: q.qsvd_latent_prefill_attn(cache, q_seq, q_len, T, *U, H, dh, O, workspace=ws)  # noqa: E731
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        times = []
        for it in range(iters + 1):
            torch.sum(flush, dim=(0,), out=sink)
            e0.record()
            call()
            e1.record()
            torch.cuda.synchronize()
            if it:
                times.append(e0.elapsed_time(e1) * 1e-3)
        # per-kernel split: events recorded by the library after each launch
        cap = 8 + 6 * (n // 16 + 1)
        events = [torch.cuda.Event(enable_timing=True) for _ in range(cap)]
        for e in events:
            e.record()
        torch.cuda.synchronize()
        handles = (ctypes.c_void_p * cap)(*[ctypes.c_void_p(e.cuda_event) for e in events])
        lib = q._lib
        lib.qsvd_profile_count.restype = ctypes.c_int32
        lib.qsvd_profile_label.restype = ctypes.c_char_p
        torch.sum(flush, dim=(0,), out=sink)
        lib.qsvd_profile_events(handles, cap)
        call()
        torch.cuda.synchronize()
        cnt = lib.qsvd_profile_count()
        labels = [lib.qsvd_profile_label(i).decode() for i in range(cnt)]
        lib.qsvd_profile_events(None, 0)
        q.qsvd_check()
    finally:
        q.qsvd_set_prefill_group_rows(prev)
    by = {}
    for i in range(1, cnt):
        e = by.setdefault(labels[i], [0, 0.0])
        e[0] += 1
        e[1] += events[i - 1].elapsed_time(events[i]) * 1e-3
    tot = sum(v[1] for v in by.values())
    pairs = B * T * (T + 1) // 2                       # visible (query, key) pairs
    if path == "blocks":
        flops = {"qkv_gemm": 2.0 * n * r * 3 * d, "fa": 4.0 * H * dh * pairs}
    else:
        att = next((k for k in ("attn_tc", "attn_mma", "attn_chunk") if k in by), "attn_tc")
        flops = {att: 4.0 * H * r * pairs, "qproj": 2.0 * n * r * d, "qabsorb": 2.0 * n * r * d,
                 "combine_uv": 2.0 * n * r * d}
    _, bf16_peak, kind = peaks()
    t = min(times)
    kern = {}
    for k, v in sorted(by.items()):
        kern[k] = {"launches": v[0], "us": round(v[1] * 1e6, 1), "share": round(v[1] / tot, 4)}
        if k in flops:
            kern[k]["tflops"] = round(flops[k] / v[1] / 1e12, 1)
            kern[k]["frac_of_bf16_peak"] = round(flops[k] / v[1] / 1e12 / bf16_peak, 4)
    out = {"path": path, "shape": f"{B} x {T} tokens, d={d} H={H} r={r} int{bits}", "rows": n,
           "call_us": round(t * 1e6, 1), "tokens_per_s": round(n / t, 1),
           "call_tflops": round(sum(flops.values()) / t / 1e12, 1), "kernels": kern, "peak_kind": kind}
    del cache, U, O, ws, flush
    return out


def importance_probe(iters=3, N=1, m=4096, n=12288, k=4096):
    """Offline Eq. 10 scores of every singular value of a 7B-shaped W_concat
    (E x 3E, E = 4096) for N calibration gradients: 2 N m n k algorithmic
    flops, done as three tf32 tensor-core products (the 3xTF32 split keeps
    fp32 accuracy).  Inputs: seeded torch Gaussians (the time does not depend
    on the values).  Peak: the measured dense bf16 rate x the nominal tf32 /
    bf16 ratio (1.1 / 2.25 PFLOP/s); frac counts the three tf32 products."""
    import torch
    import paper_2510_16292_gb300 as q
    dev = torch.device("cuda", torch.cuda.current_device())
    g = torch.Generator(device=dev)
    g.manual_seed(99)
    U = torch.randn((m, k), generator=g, device=dev)
    s = torch.rand((k,), generator=g, device=dev)
    Vt = torch.randn((k, n), generator=g, device=dev)
    G = torch.randn((N, m, n), generator=g, device=dev)
    ws = torch.empty(int(q._lib.qsvd_importance_workspace_bytes(N, m, k)), dtype=torch.uint8, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    for it in range(iters + 1):
        e0.record()
        q.qsvd_importance_scores(U, s, Vt, G, workspace=ws)
        e1.record()
        torch.cuda.synchronize()
        if it:
            times.append(e0.elapsed_time(e1) * 1e-3)
    q.qsvd_check()
    t = min(times)
    flops = 2.0 * N * m * n * k
    _, bf16_peak, kind = peaks()
    peak = bf16_peak * 1.1 / 2.25
    return {"importance_scores": f"N={N} m={m} n={n} k={k}", "ms": round(t * 1e3, 3),
            "tflops": round(flops / t / 1e12, 2), "tf32_tflops": round(3 * flops / t / 1e12, 2), "bound": "tensor",
            "peak_tflops": round(peak, 1), "frac": round(3 * flops / t / 1e12 / peak, 4),
            "peak_kind": f"{kind} bf16 x 1.1 / 2.25 (nominal tf32 / bf16)"}


def beta_probe(iters=3, N=512, E=4096, r=1536):
    """One beta of Eq. 14's grid search on a 7B-shaped layer (E = 4096,
    n_out = 3E, r = 1536) with N calibration tokens: the factors of Eq. 3
    (W_d, and Q(W^u) from fp64 Wu_r), the per-channel weight quantizer, the
    projection of the calibration tokens (int8 latent) and the objective.
    Inputs: seeded torch values (the time does not depend on them).  The
    factors' kernel reads Wd_r and Wu_r in fp64 (HBM-bound); the objective is
    an exact integer product of codes, N x 3E x r multiply-adds."""
    import torch
    import paper_2510_16292_gb300 as q
    dev = torch.device("cuda", torch.cuda.current_device())
    g = torch.Generator(device=dev)
    g.manual_seed(98)
    n = 3 * E
    Wd_r = torch.randn((E, r), generator=g, device=dev, dtype=torch.float64) / E ** 0.5
    Wu_r = torch.randn((r, n), generator=g, device=dev, dtype=torch.float64) / r ** 0.5
    sig = torch.linspace(8.0, 0.1, r, device=dev, dtype=torch.float64)
    fd, fu = sig ** 0.5, sig ** 0.5
    X = (torch.randn((N, E), generator=g, device=dev) * 0.5).to(torch.bfloat16)
    Y = torch.randn((N, n), generator=g, device=dev)
    lc = torch.empty((N, r), dtype=torch.int8, device=dev)
    ls = torch.empty((N,), dtype=torch.float32, device=dev)
    E_ = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    tf, to, tt = [], [], []
    for it in range(iters + 1):
        e0, e1, e2, e3 = E_(), E_(), E_(), E_()
        e0.record()
        W_d, U = q.qsvd_beta_factors(Wd_r, Wu_r, fd, fu)
        e1.record()
        W = q.qsvd_quantize_weight(W_d)
        q.qsvd_latent_project(W, X, lat_codes=lc, lat_scales=ls)
        e2.record()
        q.qsvd_beta_objective(Y, lc, ls, 8, r, U)
        e3.record()
        torch.cuda.synchronize()
        if it:
            tf.append(e0.elapsed_time(e1) * 1e-3)
            to.append(e2.elapsed_time(e3) * 1e-3)
            tt.append(e0.elapsed_time(e3) * 1e-3)
    q.qsvd_check()
    hbm, _, kind = peaks()
    fbytes = E * r * (8 + 4) + r * n * (8 + 1) + n * 4
    t_f, t_o, t_t = min(tf), min(to), min(tt)
    return {"beta_probe": f"E={E} n_out={n} r={r} N={N}, int8 latent and Q(W^u)",
            "factors_ms": round(t_f * 1e3, 3), "factors_gbs": round(fbytes / t_f / 1e9, 1),
            "factors_frac_of_hbm": round(fbytes / t_f / 1e9 / hbm, 4),
            "objective_ms": round(t_o * 1e3, 3), "objective_int_tops": round(2.0 * N * n * r / t_o / 1e12, 2),
            "one_beta_ms": round(t_t * 1e3, 3), "peak_kind": kind}


def cross_rank(values, op="max"):
    """Per-rank totals reduced over the ranks of the default process group
    (max: the job takes as long as its slowest rank; min: the slowest rank's
    throughput).  Without a process group, or with one rank, the values are
    returned unchanged."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return [float(v) for v in values]
    dev = torch.device("cuda", torch.cuda.current_device()) if dist.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.MIN)
    return [float(v) for v in t.cpu()]


def job_throughput(units_per_rank, world, slowest_seconds):
    """Whole-job throughput: the units every rank processed over the slowest
    rank's time (weak scaling: each rank runs its own replica)."""
    return units_per_rank * world / slowest_seconds


def run_native(args, rank, world, local_rank):
    import torch
    torch.cuda.set_device(local_rank)
    wl = synthetic.WORKLOADS[args.workload]
    if args.decode_steps:
        wl = dataclasses.replace(wl, decode_steps=args.decode_steps)
    if args.decode_call == "step" and (args.rot or args.u_bits):
        raise SystemExit("--decode-call step takes bf16 up-projections and unrotated weights")
    nb = NativeBench(wl, rank, l2=args.l2, rot=args.rot, u_bits=args.u_bits, decode_call=args.decode_call)
    K = nb.K
    S = wl.decode_steps
    hbm, _, peak_kind = peaks()

    nb.build_graph()
    for _ in range(args.warmup):
        nb.replay()
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank)
    clocks.start()
    t_wall = time.perf_counter()
    pre, dec, per_dec = [], [], []
    for k in range(args.steps):
        evs = nb.replay()
        torch.cuda.synchronize()                   # events are re-recorded by the next replay
        pre.append(evs[0][0].elapsed_time(evs[0][1]) * 1e-3)
        d_t = [evs[t + 1][0].elapsed_time(evs[t + 1][1]) * 1e-3 for t in range(S)]
        per_dec.append([x / K for x in d_t])          # per copy of the layer
        dec.append(sum(d_t))
    if world > 1:
        torch.distributed.barrier()
    t_wall = time.perf_counter() - t_wall
    clk = clocks.stop()
    dec_total, pre_total = cross_rank([sum(dec), sum(pre)], "max")
    value = job_throughput(wl.B * S * K * args.steps, world, dec_total)
    s = wl.shape
    prefill_ops = 2 * wl.B * wl.prefill * s.d * s.r
    prefill_tops = world * K * prefill_ops * args.steps / pre_total / 1e12
    tok_bytes = (s.r + 4) if wl.lat_bits == 8 else (s.r // 2 + 2 * (s.r // 128))
    cache_bytes = K * sum(wl.B * (wl.prefill + t + 1) * tok_bytes for t in range(S))
    roof_s = K * sum(nb.step_roofline_bytes(t) for t in range(S)) / (hbm * 1e9)
    step_frac = roof_s / statistics.mean(dec)

    # kernel-level profile (separate pass of the same step) -> dominant kernel + roofline
    launches = nb.profile(steps=1)
    by = {}
    for lab, ctx, dt in launches:
        e = by.setdefault(lab, {"launches": 0, "time_s": 0.0, "bytes": 0})
        e["launches"] += 1
        e["time_s"] += dt
        e["bytes"] += nb.alg_bytes(lab, ctx)
    tot_t = sum(e["time_s"] for e in by.values())
    dom = max(by, key=lambda k: by[k]["time_s"])
    de = by[dom]
    achieved = de["bytes"] / de["time_s"] / 1e9
    kernels = {k: {"launches": v["launches"], "avg_us": round(v["time_s"] / v["launches"] * 1e6, 2),
                   "share": round(v["time_s"] / tot_t, 4),
                   "gbs": round(v["bytes"] / v["time_s"] / 1e9, 1)} for k, v in sorted(by.items())}
    launches_per_step = len(launches)

    e2e = None
    if not args.no_e2e:
        e2e_val, e2e_eager, h2d, d2h = nb.e2e(steps=min(args.steps, 3), warmup=3)
        e2e_val, e2e_eager = (v * world for v in cross_rank([e2e_val, e2e_eager], "min"))   # slowest rank, every rank
        e2e = {"value": round(e2e_val, 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h,
               "launch": "one CUDA graph per step captured from the binding's calls and host copies",
               "eager_value": round(e2e_eager, 1)}

    pre13 = prefill_gemm_probe() if not args.no_prefill13 else None
    pre13_w4 = prefill_gemm_probe(w4a4=True) if not args.no_prefill13 else None
    pre_attn = None if args.no_prefill_attn else {
        k: {p: prefill_attn_probe(k, path=p) for p in ("blocks", "rows")} for k in PREFILL_REPORTED}
    if rank != 0:
        return
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round((dec_total + pre_total) / args.steps * 1e3, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int8/fp32",
        "data": "synthetic",
        "config": {"workload": workload_desc(wl) + (" + online H1 rotation of X (Eq. 12)" if args.rot else "") +
                   (f" + int{args.u_bits} up-projections (Eq. 11 Q(W^u), per-output-channel scales)"
                    if args.u_bits else ""),
                   "global_batch": world * wl.B,
                   "seq_len": wl.tmax, "parallelism": f"replicas x{world} (one independent layer per GPU)",
                   "l2": (f"inputs larger than L2: {K} independently seeded copies of the layer "
                          f"({K} x {nb.layer_bytes / 2**20:.0f} MiB of weights and latent cache); every decode "
                          f"token runs through all copies in turn and value counts tokens through one copy"
                          if args.l2 == "rotate" else
                          "flushed (256 MiB read) before the prefill and before every decode step; "
                          "flushes outside the timed intervals"),
                   "launch": "one CUDA graph per step (captured C-ABI calls, PDL-chained kernels)",
                   "decode_call": ("qsvd_decode_step" if args.decode_call == "step" else
                                   "qsvd_latent_project + qsvd_latent_decode_attn")},
        "secondary": {
            "decode_ms_per_step": round(dec_total / args.steps * 1e3, 4),
            "prefill_ms_per_step": round(pre_total / args.steps * 1e3, 4),
            "decode_us_per_token_step": round(statistics.mean(sum(per_dec, [])) * 1e6, 3),
            "prefill_tops": round(prefill_tops, 3),
            "latent_cache_gbs": round(cache_bytes * args.steps * world / dec_total / 1e9, 2),
            "decode_step_roofline_frac": round(step_frac, 4),
            "decode_step_roofline_us": round(roof_s / (S * K) * 1e6, 3),
            "wall_s_timed_region": round(t_wall, 3),
            "kernels": kernels,
            "prefill_13b": pre13,
            "prefill_13b_w4a4": pre13_w4,
            "prefill_attn": pre_attn,
        },
        "roofline": {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1), "peak": hbm,
                     "unit": "GB/s", "frac": round(achieved / hbm, 4),
                     "traffic": captured_traffic(dom, args.workload), "traffic_unit": "bytes per launch",
                     "peak_kind": peak_kind},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
    }
    if e2e:
        out["e2e"] = e2e
    if world == 1 and not args.no_cpu_baseline and args.workload == WORKLOAD:
        out["cpu_baseline"] = cpu_baseline(wl, budget_s=15.0)
    print(json.dumps(out), flush=True)


def captured_traffic(label, workload):
    """DRAM bytes per launch of kernel `label` on `workload` from the committed
    ncu launch-list record (profiles/dram_traffic.json), or None when there is
    no record or the kernel's sources changed since the capture."""
    import hashlib
    try:
        with open(os.path.join(ROOT, "profiles", "dram_traffic.json")) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    for e in rec.get("entries", []):
        if e.get("label") != label or e.get("workload") != workload:
            continue
        h = hashlib.sha256()
        try:
            for src in e["sources"]:
                with open(os.path.join(ROOT, src), "rb") as f:
                    h.update(f.read())
        except OSError:
            return None
        return e["bytes_per_launch"] if h.hexdigest() == e["sha256"] else None
    return None


# ---------------------------------------------------------------------------
# CPU oracle (baseline leg and reference arm)
# ---------------------------------------------------------------------------
def _oracle_layer(wl, seed=0):
    from oracle import pipeline
    inp = synthetic.gen_layer(wl, seed=seed)
    w = pipeline.prepare_weights(inp)
    lay = pipeline.OracleLayer(wl.shape, w, wl.B, wl.tmax, wl.lat_bits)
    for b in range(wl.B):
        lay.prefill(b, inp.X_prefill[b])
    return inp, w, lay


def cpu_baseline(wl, budget_s=15.0):
    """Decode tokens/s of the oracle on a bounded sample: prefill, then decode
    steps until `budget_s` seconds of decode work (at most all steps)."""
    inp, w, lay = _oracle_layer(wl)
    t0 = time.perf_counter()
    n = 0
    while n < wl.decode_steps and time.perf_counter() - t0 < budget_s:
        lay.decode_step(inp.X_decode[n])
        n += 1
    dt = time.perf_counter() - t0
    return {"value": round(wl.B * n / dt, 2), "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
            "sample": f"{n} of {wl.decode_steps} decode steps of {wl.name} after its full prefill "
                      f"(numpy fp64, BLAS on all host cores)"}


def run_reference(args, rank, world):
    if rank != 0:
        return
    wl = synthetic.WORKLOADS[WORKLOAD]
    inp, w, lay = _oracle_layer(wl)
    per = 4                                   # decode steps per reference step
    times = []
    pos = 0
    for k in range(args.warmup + args.steps):
        if pos + per > wl.decode_steps:       # restart the decode from the prefilled cache
            inp, w, lay = _oracle_layer(wl)
            pos = 0
        t0 = time.perf_counter()
        for t in range(per):
            lay.decode_step(inp.X_decode[pos + t])
        dt = time.perf_counter() - t0
        pos += per
        if k >= args.warmup:
            times.append(dt)
    total = sum(times)
    value = wl.B * per * args.steps / total
    sample = f"{per} decode steps of {wl.name} per step (numpy fp64 oracle, BLAS on all host cores)"
    out = {"impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "tokens/s", "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(total / args.steps * 1e3, 3),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": {"workload": workload_desc(wl)},
           "cpu_baseline": {"value": round(value, 2), "unit": "tokens/s", "cores": os.cpu_count(),
                            "kind": "oracle", "sample": sample},
           "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# ---------------------------------------------------------------------------
# sweep over the 7B-shaped layer (rank x cached length x batch x cache precision)
# ---------------------------------------------------------------------------
SWEEP_FULL = dict(r=(1024, 1536, 2048, 3072), L=(1024, 4096, 16384, 32768), B=(1, 8, 32, 64), bits=(8, 4))
SWEEP_QUICK = dict(r=(1536, 3072), L=(1024, 32768), B=(1, 64), bits=(8, 4))


def set_attn_path(args):
    if args.attn_path:
        import paper_2510_16292_gb300 as q
        q.qsvd_set_decode_attn_path(args.attn_path)


def run_sweep(args):
    """One JSON line per point: decode tokens/s of one layer and the fraction
    of the step's HBM roofline (bytes a decode step must read: the latent
    cache, the three up-projections and W_d).  The cache of each point is
    filled with seeded codes and scales as if prefilled (the sweep measures
    decode); weights are seeded Gaussians of the recipe's scales.  Cold L2:
    the points' layers rotate as in the main benchmark when one layer's
    decode bytes are below twice the L2."""
    import torch
    import paper_2510_16292_gb300 as q
    dev = torch.device("cuda", torch.cuda.current_device())
    hbm, _, peak_kind = peaks()
    if args.sweep == "point":
        r_, L_, B_, bits_ = (int(v) for v in args.sweep_point.split(","))
        grid = dict(r=(r_,), L=(L_,), B=(B_,), bits=(bits_,))
    else:
        grid = SWEEP_FULL if args.sweep == "full" else SWEEP_QUICK
    d, H, dh = 4096, 32, 128
    g = torch.Generator(device=dev)
    g.manual_seed(2510)
    for r in grid["r"]:
        for bits in grid["bits"]:
            for B in grid["B"]:
                for L in grid["L"]:
                    tok = (r + 4) if bits == 8 else (r // 2 + 2 * (r // 128))
                    layer_bytes = 3 * r * d * 2 + r * d + B * L * tok
                    K = 1 if layer_bytes >= 2 * L2_BYTES else max(2, -(-2 * L2_BYTES // layer_bytes))
                    layers = []
                    for _ in range(K):
                        Wd = torch.randn((d, r), generator=g, device=dev) / math.sqrt(d)
                        W = q.qsvd_quantize_weight(Wd)
                        del Wd
                        U = [(torch.randn((r, d), generator=g, device=dev) / math.sqrt(r)).to(torch.bfloat16)
                             for _ in range(3)]
                        cache = q.LatentCache.empty(B, L + 1, r, bits, dev)
                        if bits == 8:
                            cache.codes.copy_(torch.randint(-127, 128, cache.codes.shape, generator=g, device=dev,
                                                            dtype=torch.int8))
                            cache.scales.copy_(torch.rand(cache.scales.shape, generator=g, device=dev) * 0.02 + 0.01)
                        else:
                            cache.codes.copy_(torch.randint(0, 256, cache.codes.shape, generator=g, device=dev,
                                                            dtype=torch.uint8))
                            cache.scales.copy_((torch.rand(cache.scales.shape, generator=g, device=dev) * 0.2
                                                + 0.1).half())
                        X = torch.randn((B, d), generator=g, device=dev).to(torch.bfloat16)
                        O = torch.empty((B, d), dtype=torch.float32, device=dev)
                        layers.append((W, U, cache, X, O))
                    seq = torch.arange(B, dtype=torch.int32, device=dev)
                    pos = torch.full((B,), L, dtype=torch.int32, device=dev)
                    lens = torch.full((B,), L + 1, dtype=torch.int32, device=dev)
                    wsp = torch.zeros(q.qsvd_project_workspace_bytes(B, d, r), dtype=torch.uint8, device=dev)
                    wsd = torch.zeros(q.qsvd_decode_workspace_bytes(B, L + 1, r, H, dh), dtype=torch.uint8,
                                      device=dev)
                    st = torch.cuda.Stream()
                    st.wait_stream(torch.cuda.current_stream())      # inputs and workspaces were filled there
                    steps = 4
                    E = lambda: torch.cuda.Event(enable_timing=True, external=True)  # noqa: E731
                    evs = [(E(), E()) for _ in range(steps)]

                    def one(k):
                        W, U, cache, X, O = layers[k]
                        q.qsvd_latent_project(W, X, 1.0, bits, 1.0, dst=cache, dst_seq=seq, dst_pos=pos,
                                              workspace=wsp, stream=st)
                        q.qsvd_latent_decode_attn(cache, lens, L + 1, *U, H, dh, O, workspace=wsd, stream=st)

                    with torch.cuda.stream(st):
                        for k in range(K):
                            one(k)
                    torch.cuda.synchronize()
                    gr = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(gr, stream=st):
                        for a, b in evs:
                            a.record(st)
                            for k in range(K):
                                one(k)
                            b.record(st)
                    for _ in range(3):
                        gr.replay()
                    torch.cuda.synchronize()
                    ts = []
                    for _ in range(3):
                        gr.replay()
                        torch.cuda.synchronize()
                        ts += [a.elapsed_time(b) * 1e-3 / K for a, b in evs]
                    q.qsvd_check()
                    t = statistics.median(ts)
                    roof = layer_bytes / (hbm * 1e9)
                    # one layer's step time t is measured over K independently seeded layer
                    # copies in rotation; the 32-layer stack takes 32 such steps per token
                    print(json.dumps({"sweep": {"r": r, "L": L, "B": B, "bits": bits, "layer_copies": K},
                                      "decode_tokens_s_32_layers": round(B / (32 * t), 1),
                                      "decode_tokens_s_per_layer": round(B / t, 1),
                                      "us_per_layer_step": round(t * 1e6, 2),
                                      "step_roofline_us": round(roof * 1e6, 2), "roofline_frac": round(roof / t, 4),
                                      "peak_gbs": hbm, "peak_kind": peak_kind}), flush=True)
                    del layers, wsd, wsp, gr
                    torch.cuda.empty_cache()


def main():
    args = parse()
    set_attn_path(args)
    if args.sweep:
        run_sweep(args)
        return
    if args.importance_probe:
        print(json.dumps(importance_probe(iters=args.steps)), flush=True)
        return
    if args.beta_probe:
        print(json.dumps(beta_probe(iters=args.steps)), flush=True)
        return
    if args.prefill_probe:
        for name in args.prefill_shapes.split(","):
            for path in args.prefill_paths.split(","):
                print(json.dumps({"prefill_attn": name, **prefill_attn_probe(name, iters=args.steps, path=path)}),
                      flush=True)
        return
    if args.prefill_sweep is not None:
        for rows in (int(x) for x in args.prefill_sweep.split(",")):
            for name in PREFILL_REPORTED:
                print(json.dumps({"prefill_attn": name, "group_rows": rows,
                                  **prefill_attn_probe(name, iters=args.steps, group_rows=rows, path="rows")}),
                      flush=True)
        return
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if world > 1:
        import torch
        torch.cuda.set_device(local_rank)
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    try:
        run_native(args, rank, world, local_rank)
    finally:
        if world > 1:
            import torch
            torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
