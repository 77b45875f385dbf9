#!/usr/bin/env python
"""Benchmark of the schedule-search hot path on GB300.

Default workload (one GPU): the Llama-3-8B-shaped SwiGLU MLP block, bf16,
tokens T=2048, hidden H=4096, intermediate I=14336, weights N(0, 0.02),
activations N(0, 1), synthetic seeded inputs. ``--workload`` selects one of
the other hot-path workloads instead (attention, conv2d, moe, gemm_f32).

A run
  1. searches the workload's schedule space with the LLM-free MCTS
     (rc_search_step), every candidate timed on the device
     (rc_candidate_measure) -> candidates measured per second;
  2. times K steps of the best schedule found (rc_run_profiled: per-stage
     CUDA events on the launching stream; L2 flushed between steps, outside
     the timed events) -> best-schedule TFLOP/s, and the roofline fraction of
     the dominant kernel measured live;
  3. times K end-to-end steps through rc_run_host (pinned host buffers,
     host->device inputs and device->host outputs inside the timed region);
  4. searches the other workloads briefly and reports each one's best
     schedule and roofline fraction (``ops``);
  5. times the fp64 CPU oracle on a bounded sample of the workload.
Under torchrun (N > 1) every rank runs an independent replica (the path has
no exchange step); value = all ranks' work / the slowest rank's time.

``--impl reference`` times the CPU oracle alone as the reference arm.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

# FP32 SIMT peak of one GB300: 152 SMs x 128 FP32 lanes x 2 flops x 2.07 GHz.
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mlp",
                    choices=["mlp", "attention", "conv2d", "moe", "gemm_f32", "attention_flux", "decoder_layer",
                             "linear"])
    ap.add_argument("--samples", type=int, default=5000, help="schedules the search measures")
    ap.add_argument("--branching", type=int, default=4,
                    help="MCTS children per expansion (the paper's 2 assumes LLM-proposed transformations; with "
                         "random valid proposals a binary tree of depth 8 fills up at 511 nodes)")
    ap.add_argument("--cpu-sample", type=int, default=0,
                    help="size of the CPU-oracle sample (rows/queries/pixels/tokens; 0 = workload default, "
                         "-1 = skip)")
    ap.add_argument("--schedule", default="",
                    help="fixed schedule instead of a search, e.g. 's0:tile_n=128,stages=4,fuse=1;s1:tile_n=256'")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--ops", default=None,
                    help="other workloads to search and report ('' = none; default: all others for mlp)")
    ap.add_argument("--op-samples", type=int, default=600, help="schedules measured per extra op")
    ap.add_argument("--moe-samples", type=int, default=2000,
                    help="schedules measured for the MoE layer when it is an extra op (three stages of knobs)")
    ap.add_argument("--layer-samples", type=int, default=3000,
                    help="schedules measured for the decoder layer when it is an extra op (six stages of knobs)")
    ap.add_argument("--horizon", type=int, default=0,
                    help="maximum transformation-sequence length T of each search (0 = the workload's: 8)")
    ap.add_argument("--tasks", type=int, default=-1, choices=[-1, 0, 1],
                    help="1 = tune a composite op stage by stage, then jointly (search_tasks); 0 = one joint "
                         "search; -1 = the workload's choice (stage by stage for the MLP, MoE and decoder layer)")
    ap.add_argument("--restarts", type=int, default=2,
                    help="independent searches (seeds seed, seed+1, ...) per workload; the fastest result is kept")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--surrogate", type=int, default=1, choices=[0, 1],
                    help="1 = rollouts scored by the search's learned surrogate f-hat (Sec. 3.2), only expanded "
                         "nodes measured; 0 = rollout programs measured too")
    ap.add_argument("--screen", type=int, default=4,
                    help="with --surrogate 1: proposals screened by f-hat per kept child (1 = no screening)")
    ap.add_argument("--study", default="",
                    help="instead of the benchmark line: 'search' prints best-so-far curves (JSON lines) of the "
                         "search variants on --workload: MCTS with measured rollouts at B = 2 and 4, MCTS with the "
                         "learned surrogate and 4x screening, random search, and (composite ops) stage-by-stage "
                         "tuning then a joint search, over seeds --seed .. --seed+1; 'library' times the vendor "
                         "libraries (cuDNN attention and convolution, cuBLAS GEMMs through torch) on --workload's "
                         "inputs under the bench's timing protocol")
    ap.add_argument("--study-variants", default="",
                    help="with --study search: comma-separated variant names to run (default: all)")
    ap.add_argument("--shape", default="",
                    help="override workload sizes for a profiling case, e.g. 'tokens=1024,experts=16' (the line "
                         "then reports that shape, not the benchmark configuration)")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"bf16_tflops": d["bf16_tflops"], "hbm_gbs": d["hbm_gbs"], "source": "measured"}
    return {"bf16_tflops": 1900.0, "hbm_gbs": 6800.0, "source": "fallback"}


class Clocks:
    """nvidia-smi sampler running while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-lms", "20", "-i", str(self.gpu)], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
            return
        # let the sampler emit its first line before the timed region starts (at most 3 s)
        t0 = time.time()
        while time.time() - t0 < 3.0 and self.proc.poll() is None:
            self.f.flush()
            if os.path.getsize(self.f.name) > 0:
                break
            time.sleep(0.02)
        self.skip = sum(1 for _ in open(self.f.name))  # lines from before the timed region

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.flush()
        rows = []
        for i, line in enumerate(open(self.f.name)):
            if i < getattr(self, "skip", 0):
                continue
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        os.unlink(self.f.name)
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": num(rows[0][2]),
                "reasons": reasons, "samples": len(rows)}


# ------------------------------------------------------------------ workloads --

class Workload:
    """One hot-path workload: op, seeded host inputs, output slots, dominant kernel."""

    def __init__(self, name, shape=None):
        import numpy as np

        from paper_2506_01374_gb300 import inputs, rc
        self.name = name
        self._op = None
        self.dom_bytes = None  # algorithmic DRAM bytes of the dominant kernel, where stated
        self.horizon = 8  # search horizon T
        self.tasks = False  # composite ops: tuned stage by stage (search_tasks), then jointly
        sh = dict(shape or {})

        def dims(**default):
            unknown = set(sh) - set(default)
            if unknown:
                raise ValueError(f"--shape keys {sorted(unknown)} do not apply to {name}")
            return [sh.get(k, v) for k, v in default.items()]

        if name == "mlp":
            self.tasks = True
            T, H, I = dims(tokens=2048, hidden=4096, inter=14336)
            X, W1, W2 = inputs.mlp(T, H, I, seed=1)
            self._op_spec = (rc.OP_MLP, dict(m=T, n=I, k=H))
            self.host = [X, W1, W2, None]
            self.outs = {3: ((T, H), np.uint16)}
            self.label = "llama3_8b_mlp_swiglu_bf16_T2048_H4096_I14336"
            self.config = {"tokens": T, "hidden": H, "inter": I}
            self.metric = "best-schedule TFLOP/s (Llama-3-8B MLP block, bf16)"
            self.dom_stage, self.dom_flops = 0, 2.0 * T * (2 * I) * H
            self.dom_bytes = 2.0 * (T * H + 2 * I * H + T * I)  # X and W1 read once, h written once
            self.dom_name = "gate/up GEMM{} (stage 0)"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "attention":
            B, S, Hq, Hkv = dims(batch=1, seq=2048, heads_q=32, heads_kv=8)
            D = 128
            Q, K, V = inputs.attention(B, S, Hq, Hkv, D, seed=4)
            self._op_spec = (rc.OP_ATTENTION,
                             dict(batch=B, seq=S, heads_q=Hq, heads_kv=Hkv, head_dim=D, causal=1))
            self.host = [Q, K, V, None, None]
            self.outs = {3: ((B, S, Hq, D), np.uint16), 4: ((B, Hq, S), np.float32)}
            self.label = "causal_gqa_attention_B1_S2048_Hq32_Hkv8_d128_bf16"
            self.config = {"batch": B, "seq": S, "heads_q": Hq, "heads_kv": Hkv, "head_dim": D, "causal": True}
            self.metric = "best-schedule TFLOP/s (causal GQA attention, bf16)"
            self.dom_stage, self.dom_flops = 0, None  # the op's flops
            self.dom_name = "fused attention kernel"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "attention_flux":
            # FLUX-style (DiT) self-attention: non-causal, multi-head, 64 x 64 image tokens
            B, S, Hq = dims(batch=1, seq=4096, heads=24)
            Hkv, D = Hq, 128
            Q, K, V = inputs.attention(B, S, Hq, Hkv, D, seed=7)
            self._op_spec = (rc.OP_ATTENTION,
                             dict(batch=B, seq=S, heads_q=Hq, heads_kv=Hkv, head_dim=D, causal=0))
            self.host = [Q, K, V, None, None]
            self.outs = {3: ((B, S, Hq, D), np.uint16), 4: ((B, Hq, S), np.float32)}
            self.label = f"flux_attention_B{B}_S{S}_H{Hq}_d128_noncausal_bf16"
            self.config = {"batch": B, "seq": S, "heads": Hq, "head_dim": D, "causal": False}
            self.metric = "best-schedule TFLOP/s (non-causal MHA attention, bf16)"
            self.dom_stage, self.dom_flops = 0, None  # the op's flops
            self.dom_name = "fused attention kernel"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "conv2d":
            N, H, W, C = dims(n=2, h=64, w=64, c=320)
            x, w, b = inputs.conv2d(N, H, W, C, C, seed=5)
            self._op_spec = (rc.OP_CONV2D, dict(img_n=N, img_h=H, img_w=W, c_in=C, c_out=C, kr=3, ks=3, stride=1, pad=1,
                            flags=rc.EPI_BIAS | rc.EPI_SILU))
            self.host = [x, w, b, None]
            self.outs = {3: ((N, H, W, C), np.uint16)}
            self.label = "conv2d_nhwc_3x3_N2_64x64_C320_bias_silu_bf16"
            self.config = {"n": N, "h": H, "w": W, "c_in": C, "c_out": C, "kernel": 3}
            self.metric = "best-schedule TFLOP/s (UNet conv2d 3x3 + bias + SiLU, bf16)"
            self.dom_stage, self.dom_flops = 0, None  # the op's flops
            self.dom_name = "implicit-GEMM conv kernel"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "moe":
            self.tasks = True
            T, H, E, I, K = dims(tokens=4096, hidden=7168, experts=64, inter=2048, top_k=8)
            logits, X, W1, W2 = inputs.moe(T, H, E, I, seed=6)
            self._op_spec = (rc.OP_MOE, dict(tokens=T, hidden=H, experts=E, inter=I, top_k=K))
            self.host = [logits, X, W1, W2, None]
            self.outs = {4: ((T, H), np.uint16)}
            self.label = "moe_T4096_H7168_E64_I2048_top8_bf16"
            self.config = {"tokens": T, "hidden": H, "experts": E, "inter": I, "top_k": K}
            self.metric = "best-schedule TFLOP/s (MoE layer, 64 experts, top-8, bf16)"
            self.dom_stage, self.dom_flops = 1, 2.0 * T * K * (2 * I) * H
            self.dom_name = "grouped gate/up GEMM + SwiGLU (stage 1)"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "decoder_layer":
            self.tasks = True
            T, H, Hq, Hkv, I = dims(tokens=2048, hidden=4096, heads_q=32, heads_kv=8, inter=14336)
            self.host = list(inputs.decoder_layer(T, H, Hq, Hkv, I, seed=8)) + [None]
            self._op_spec = (rc.OP_DECODER_LAYER,
                             dict(tokens=T, hidden=H, inter=I, heads_q=Hq, heads_kv=Hkv, head_dim=128))
            self.outs = {7: ((T, H), np.uint16)}
            self.label = f"llama3_8b_decoder_layer_T{T}_H{H}_Hq{Hq}_Hkv{Hkv}_I{I}_bf16"
            self.config = {"tokens": T, "hidden": H, "heads_q": Hq, "heads_kv": Hkv, "inter": I}
            self.metric = "best-schedule TFLOP/s (Llama-3-8B decoder layer, bf16)"
            self.dom_stage, self.dom_flops = 4, 2.0 * T * (2 * I) * H
            self.dom_name = "gate/up GEMM + SwiGLU (stage 4)"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "linear":
            # the MLP block's down projection as a plain bf16 GEMM: Y = h W2^T, M = 2048, N = 4096, K = 14336
            M, N, K = dims(m=2048, n=4096, k=14336)
            X, Wt = inputs.linear_bf16(M, N, K, seed=3)
            self._op_spec = (rc.OP_LINEAR, dict(m=M, n=N, k=K))
            self.host = [X, Wt, None]
            self.outs = {2: ((M, N), np.uint16)}
            self.label = f"linear_bf16_M{M}_N{N}_K{K}"
            self.config = {"m": M, "n": N, "k": K}
            self.metric = "best-schedule TFLOP/s (bf16 GEMM at the MLP down-projection shape)"
            self.dom_stage, self.dom_flops = 0, 2.0 * M * N * K
            self.dom_bytes = 2.0 * (M * K + N * K + M * N)
            self.dom_name = "tensor-core GEMM"
            self.bound = "tensor"
            self.dtype = "bf16"
        elif name == "gemm_f32":
            M, N, K = dims(m=256, n=256, k=256)
            A, B, bias = inputs.gemm_f32(M, N, K, seed=0)
            self._op_spec = (rc.OP_GEMM_F32, dict(m=M, n=N, k=K, flags=rc.EPI_BIAS | rc.EPI_RELU))
            self.host = [A, B, bias, None]
            self.outs = {3: ((M, N), np.float32)}
            self.label = "gemm_bias_relu_f32_256^3"
            self.config = {"m": M, "n": N, "k": K}
            self.metric = "best-schedule TFLOP/s (fp32 GEMM + bias + ReLU, 256^3)"
            self.dom_stage, self.dom_flops = 0, None  # the op's flops
            self.dom_name = "fp32 SIMT GEMM"
            self.bound = "alu"
            self.dtype = "f32"
        else:
            raise ValueError(name)

    @property
    def op(self):
        """The library's op (created on first use: the oracle arm never loads the library)."""
        if self._op is None:
            from paper_2506_01374_gb300 import rc
            kind, kw = self._op_spec
            self._op = rc.Op(kind, **kw)
            if self.dom_flops is None:
                self.dom_flops = self._op.info["flops"]
        return self._op

    def device_io(self):
        import numpy as np
        import torch
        io = []
        for i, a in enumerate(self.host):
            if a is not None:
                io.append(torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).cuda())
            elif i in self.outs:
                shape, dt = self.outs[i]
                io.append(torch.empty(shape, dtype=torch.int16 if dt == np.uint16 else torch.float32, device="cuda"))
            else:
                io.append(None)
        return io

    def host_io(self):
        import numpy as np
        import torch
        io = []
        for i, a in enumerate(self.host):
            if a is not None:
                io.append(torch.from_numpy(a.view(np.int16) if a.dtype == np.uint16 else a).pin_memory().numpy())
            elif i in self.outs:
                shape, dt = self.outs[i]
                io.append(torch.empty(shape, dtype=torch.int16 if dt == np.uint16 else torch.float32)
                          .pin_memory().numpy())
            else:
                io.append(None)
        return io

    def io_bytes(self):
        import numpy as np
        h2d = sum(a.nbytes for a in self.host if a is not None)
        d2h = sum(int(np.prod(s)) * np.dtype(dt).itemsize for s, dt in self.outs.values())
        return h2d, d2h

    def parity(self, sched, io):
        """Run `sched` once on the device buffers (outside every timed region) and compare sampled outputs
        with the fp64 oracle at the op's tolerance: 1e-4 normwise for fp32, 2e-2 for bf16, routing
        bit-exact. Returns {"max_rel_err", "tol", "sample", "ok"}; a schedule whose check fails is not
        reported."""
        import numpy as np
        import torch

        import oracle
        oracle.build()
        op = self.op

        def bf(t):
            u = t.cpu().numpy().view(np.uint16).astype(np.uint32) << np.uint32(16)
            return u.view(np.float32).astype(np.float64)

        def rel(got, ref):
            return float(np.max(np.abs(got - ref)) / max(float(np.max(np.abs(ref))), 1e-30))

        tol = 1e-4 if self.dtype == "f32" else 2e-2
        extra = {}
        if self.name == "mlp":
            X, W1, W2 = self.host[:3]
            rows = np.linspace(0, X.shape[0] - 1, 16).astype(np.int64)
            op.run(sched, io)
            op.check()
            err = rel(bf(io[3])[rows], oracle.mlp_bf16(X, W1, W2, rows=rows))
            what = f"{len(rows)} of {X.shape[0]} token rows"
        elif self.name == "linear":
            X, Wt = self.host[:2]
            rows = np.linspace(0, X.shape[0] - 1, 16).astype(np.int64)
            op.run(sched, io)
            op.check()
            err = rel(bf(io[2])[rows], oracle.linear_bf16(X, Wt, rows=rows))
            what = f"{len(rows)} of {X.shape[0]} rows"
        elif self.name in ("attention", "attention_flux"):
            Q, K, V = self.host[:3]
            qpos = np.linspace(0, Q.shape[1] - 1, 16).astype(np.int64)
            O_ref, L_ref = oracle.attention_bf16(Q, K, V, causal=self.name == "attention", qpos=qpos)
            op.run(sched, io)
            op.check()
            err = rel(bf(io[3])[:, qpos], O_ref)
            if io[4] is not None:
                lse = io[4].cpu().numpy().astype(np.float64)[:, :, qpos]
                extra["lse_rel_err"] = rel(lse, L_ref)
                extra["lse_ok"] = extra["lse_rel_err"] <= 1e-3
            what = f"{len(qpos)} of {Q.shape[1]} query positions, all heads"
        elif self.name == "conv2d":
            x, w, b = self.host[:3]
            total = x.shape[0] * x.shape[1] * x.shape[2]
            pix = np.linspace(0, total - 1, 256).astype(np.int64)
            op.run(sched, io)
            op.check()
            err = rel(bf(io[3]).reshape(total, -1)[pix], oracle.conv2d_nhwc_bf16(x, w, b, pix=pix))
            what = f"{len(pix)} of {total} output pixels"
        elif self.name == "moe":
            logits, X, W1, W2 = self.host[:4]
            T, K, E = X.shape[0], self.config["top_k"], self.config["experts"]
            ids, wts, off, perm = oracle.moe_route(logits, K)
            tok = np.linspace(0, T - 1, 16).astype(np.int64)
            gi = torch.empty(T, K, dtype=torch.int32, device="cuda")
            go = torch.empty(E + 1, dtype=torch.int32, device="cuda")
            gp = torch.empty(T * K, dtype=torch.int32, device="cuda")
            op.run(sched, list(io[:5]) + [gi, None, go, gp])
            op.check()
            extra["routing_exact"] = bool(np.array_equal(gi.cpu().numpy(), ids) and
                                          np.array_equal(go.cpu().numpy(), off) and
                                          np.array_equal(gp.cpu().numpy(), perm))
            err = rel(bf(io[4])[tok], oracle.moe_ffn_bf16(X, W1, W2, ids, wts, tok=tok))
            what = f"routing of all {T} tokens (bit-exact) + the layer output of {len(tok)} tokens"
        elif self.name == "decoder_layer":
            from oracle import decoder
            x = self.host[0]
            rows = np.linspace(0, x.shape[0] - 1, 4).astype(np.int64)
            ref = decoder.decoder_layer_bf16(*self.host[:7], self.config["heads_q"], self.config["heads_kv"],
                                             rows=rows)
            op.run(sched, io)
            op.check()
            x0 = decoder.widen(x[rows])
            err = rel(bf(io[7])[rows] - x0, ref - x0)  # the layer's increment, not the residual copy of x
            what = f"increment y - x of {len(rows)} of {x.shape[0]} token rows"
        else:
            A, B, bias = self.host[:3]
            op.run(sched, io)
            op.check()
            err = rel(io[3].cpu().numpy().astype(np.float64), oracle.gemm_bias_relu_f32(A, B, bias))
            what = "every output"
        ok = err <= tol and extra.get("routing_exact", True) and extra.get("lse_ok", True)
        return dict(max_rel_err=err, tol=tol, sample=what, ok=bool(ok), **extra)

    def cpu_sample(self, n, single_thread=True):
        """Time the fp64 oracle on a bounded sample with all its threads; returns the cpu_baseline dict.

        single_thread: also time a sample 1/threads the size with one thread (the oracle's
        results do not depend on its thread count), reported under "single_thread". The decoder
        layer's numpy matrix product is threaded by numpy's BLAS, outside the oracle's control,
        so it gets no single-thread figure."""
        import oracle
        oracle.build()
        out = self._oracle_sample(n)
        if single_thread and self.name != "decoder_layer":
            prev = oracle.threads()
            oracle.threads(1)
            try:
                one = self._oracle_sample(max(1, out["n"] // max(1, prev)))
            finally:
                oracle.threads(prev)
            out["single_thread"] = {"value": one["value"], "sample": one["sample"], "seconds": one["seconds"]}
        out.pop("n")
        return out

    def _oracle_sample(self, n):
        import numpy as np

        import oracle
        cores = oracle.threads()
        if self.name == "mlp":
            X, W1, W2 = self.host[:3]
            n = n or 2048
            sel = np.arange(n, dtype=np.int64) * (X.shape[0] // n)
            t0 = time.perf_counter()
            oracle.mlp_bf16(X, W1, W2, rows=sel)
            dt = time.perf_counter() - t0
            flops = 6.0 * n * X.shape[1] * (W1.shape[0] // 2)
            what, used = f"{n} of {X.shape[0]} token rows of the MLP block", min(cores, n)
        elif self.name in ("attention", "attention_flux"):
            Q, K, V = self.host[:3]
            S = Q.shape[1]
            causal = self.name == "attention"
            n = n or 256
            qpos = np.linspace(0, S - 1, n).astype(np.int64)
            t0 = time.perf_counter()
            oracle.attention_bf16(Q, K, V, causal=causal, qpos=qpos)
            dt = time.perf_counter() - t0
            flops = float(sum(4.0 * Q.shape[3] * Q.shape[2] * ((int(i) + 1) if causal else S) for i in qpos))
            what, used = f"{n} of {S} query positions (all heads)", min(cores, n)
        elif self.name == "conv2d":
            x, w, b = self.host[:3]
            total = x.shape[0] * x.shape[1] * x.shape[2]
            n = n or 4096
            pix = np.linspace(0, total - 1, n).astype(np.int64)
            t0 = time.perf_counter()
            oracle.conv2d_nhwc_bf16(x, w, b, pix=pix)
            dt = time.perf_counter() - t0
            flops = 2.0 * n * w.shape[0] * w.shape[1] * w.shape[2] * w.shape[3]
            what, used = f"{n} of {total} output pixels", min(cores, n)
        elif self.name == "linear":
            X, Wt = self.host[:2]
            n = n or 64
            rows = np.linspace(0, X.shape[0] - 1, n).astype(np.int64)
            t0 = time.perf_counter()
            oracle.linear_bf16(X, Wt, rows=rows)
            dt = time.perf_counter() - t0
            flops = 2.0 * n * Wt.shape[0] * X.shape[1]
            what, used = f"{n} of {X.shape[0]} rows", min(cores, n)
        elif self.name == "moe":
            logits, X, W1, W2 = self.host[:4]
            n = n or 32
            tok = np.linspace(0, X.shape[0] - 1, n).astype(np.int64)
            t0 = time.perf_counter()
            ids, w, _, _ = oracle.moe_route(logits, 8)
            oracle.moe_ffn_bf16(X, W1, W2, ids, w, tok=tok)
            dt = time.perf_counter() - t0
            flops = 6.0 * n * 8 * X.shape[1] * (W1.shape[1] // 2)
            what, used = f"routing of all tokens + expert FFN of {n} of {X.shape[0]} tokens", min(cores, n)
        elif self.name == "decoder_layer":
            from oracle import decoder
            x = self.host[0]
            T, H = x.shape
            Hq, Hkv, I = self.config["heads_q"], self.config["heads_kv"], self.config["inter"]
            n = n or 8
            rows = np.linspace(0, T - 1, n).astype(np.int64)
            t0 = time.perf_counter()
            decoder.decoder_layer_bf16(*self.host[:7], Hq, Hkv, rows=rows)
            dt = time.perf_counter() - t0
            hq, hkv = Hq * 128, Hkv * 128
            # the QKV projection of every token (keys and values of all positions) + the rows' own work
            flops = 2.0 * T * H * (hq + 2 * hkv) + float(sum(4.0 * 128 * Hq * (int(r) + 1) for r in rows)) + \
                n * (2.0 * hq * H + 6.0 * H * I)
            what = (f"{n} of {T} token rows of the layer, fp64 (QKV projection of all {T} tokens as a numpy "
                    "matrix product, attention and MLP of the rows as loop nests)")
            used = cores
        else:
            A, B, bias = self.host[:3]
            n = n or 40
            t0 = time.perf_counter()
            for _ in range(n):
                oracle.gemm_bias_relu_f32(A, B, bias)
            dt = time.perf_counter() - t0
            flops = n * 2.0 * A.shape[0] * A.shape[1] * B.shape[1]
            what, used = f"{n} full 256^3 GEMMs", min(cores, A.shape[0])
        if self.name != "decoder_layer":
            what += ", fp64 loop nests"
        return {"value": flops / dt / 1e12, "unit": "TFLOP/s", "cores": used, "kind": "oracle",
                "sample": what, "seconds": dt, "n": n, "cpu_model": cpu_model(), "nproc": os.cpu_count()}


TRAFFIC_FILE = os.path.join(ROOT, "profiles", "dram_traffic.json")


def source_digest(paths):
    """sha256 over the given repository files (the sources a measured kernel was built from)."""
    import hashlib
    h = hashlib.sha256()
    for rel in sorted(paths):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(rel.encode() + b"\0" + f.read())
    return h.hexdigest()


def measured_traffic(label, stage_knobs):
    """DRAM bytes per launch of a workload's dominant kernel, from the committed ncu capture
    (profiles/dram_traffic.json), keyed by the workload and the dominant stage's knobs. None when no
    capture covers this schedule or the kernel's sources have changed since the capture."""
    try:
        table = json.load(open(TRAFFIC_FILE))
    except (OSError, ValueError):
        return None
    for rec in table.get("captures", []):
        if rec.get("workload") != label or rec.get("stage_knobs") != stage_knobs:
            continue
        try:
            if source_digest(rec["sources"]) != rec["sources_sha256"]:
                return None
        except OSError:
            return None
        return rec
    return None


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo), for the CPU-baseline record."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu model")):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def knob_text(sched, stage):
    """One stage's canonical knob text, e.g. 'tile=256x128x64,unroll=1,...' (the schedule's s<stage> part)."""
    for part in str(sched).split(";"):
        if part.startswith(f"s{stage}:"):
            return part.split(":", 1)[1]
    return ""


def parse_shape(text):
    """'tokens=1024,experts=16' -> {'tokens': 1024, 'experts': 16}"""
    out = {}
    for kv in filter(None, text.split(",")):
        k, v = kv.split("=")
        out[k.strip()] = int(v)
    return out


def parse_schedule(op, text, rc):
    """'s0:tile_n=128,stages=4;s1:split_k=2' -> schedule (raster=R/G sets loop order and group)."""
    KNOB_T = {"tile_m": (rc.T_TILE_SIZE, 0), "tile_n": (rc.T_TILE_SIZE, 1), "tile_k": (rc.T_TILE_SIZE, 2),
              "stages": (rc.T_PIPELINE_STAGES, 0), "split_k": (rc.T_SPLIT_K, 0), "fuse": (rc.T_FUSE, 0),
              "raster": (rc.T_LOOP_ORDER, 0), "persistent": (rc.T_PARALLEL, 0), "layout": (rc.T_LAYOUT, 0),
              "unroll": (rc.T_UNROLL, 0), "location": (rc.T_COMPUTE_LOCATION, 0), "vec": (rc.T_VECTORIZE, 0)}
    KNOB_T["loc"] = KNOB_T["location"]
    p0 = op.schedule()
    ts = []
    for part in filter(None, text.split(";")):
        if part.startswith("op="):  # the canonical form str(schedule) prints
            continue
        stage_s, kvs = part.split(":")
        stage = int(stage_s.strip()[1:])
        items = []
        for kv in filter(None, kvs.split(",")):
            k, v = kv.split("=")
            if k.strip() == "tile":
                items += list(zip(("tile_m", "tile_n", "tile_k"), v.split("x")))
            else:
                items.append((k.strip(), v))
        for k, v in items:
            if str(p0.knobs(stage).get(k if k != "loc" else "location")) == v and k != "raster":
                continue  # P0's value (also where the knob is not tunable at this stage)
            kind, axis = KNOB_T[k]
            if k == "raster":
                r, g = (v.split("/") + ["1"])[:2]
                if p0.knobs(stage)["raster"] == int(r) and p0.knobs(stage)["group"] == int(g):
                    continue
                ts.append(rc.T(kind, int(r), stage=stage, group=int(g)))
            else:
                ts.append(rc.T(kind, int(v), axis=axis, stage=stage))
    return op.schedule(*ts)


def search_best(op, io, samples, seed=0, branching=4, finalists=4, restarts=1, surrogate=False, screen=1,
                horizon=8, root=None, stages=None):
    """MCTS over op's schedule space with device-timed candidates; returns (search, best, m, n, cand/s).

    Candidates are timed with 5 repeats while searching; the `finalists` best
    of them are timed again with 20 repeats and the fastest is returned, so a
    noisy short measurement does not decide the result. surrogate/screen: the
    learned rollout surrogate and proposal screening of rc_search_opts.
    root/stages: start from `root` and tune only `stages` (rc_search_opts.root
    and stage_mask); the objective is then those stages' summed time.
    """
    from paper_2506_01374_gb300 import rc

    def obj(m):
        return sum(m.stage_ms[g] for g in stages) if stages else m.ms_median

    if restarts > 1:  # independent searches; rewards are noisy measurements, so trajectories differ
        runs = [search_best(op, io, samples, seed + r, branching, finalists, 1, surrogate, screen, horizon, root,
                            stages) for r in range(restarts)]
        i = min(range(restarts), key=lambda r: obj(runs[r][2]) if runs[r][2].status == rc.OK else float("inf"))
        search, best, m, _, _ = runs[i]
        n = sum(r[3] for r in runs)
        cps = [r[4] for r in runs if r[4]]
        return search, best, m, n, (sum(cps) / len(cps) if cps else None)
    search = rc.Search(op, seed=seed, branching=branching, horizon=horizon, surrogate=surrogate, screen=screen,
                       stages=stages, root=root)
    res, n, t, pending = [], 0, 0.0, False
    seen = []  # (median ms, schedule owned by the search)
    while n < samples:
        nxt = search.step(res)
        pending = False
        if not nxt:
            break
        t0 = time.perf_counter()
        res = op.measure(nxt, io, warmup=2, repeats=5)
        t += time.perf_counter() - t0
        n += len(nxt)
        seen += [(obj(m), s) for s, m in zip(nxt, res) if m.status == rc.OK]
        pending = True
    if pending:  # hand the last batch's measurements to the search
        search.step(res)
    best, m = search.best()
    seen.sort(key=lambda x: x[0])
    cands = [best] + [sch for _, sch in seen[:finalists]]
    final = op.measure(cands, io, warmup=3, repeats=20)
    i = min(range(len(cands)), key=lambda j: obj(final[j]) if final[j].status == rc.OK else float("inf"))
    if i > 0:
        best, m = cands[i].clone(), final[i]
    return search, best, m, n, (n / t if t else None)


def search_tasks(op, io, samples, seed=0, branching=4, finalists=4, restarts=1, surrogate=False, screen=1,
                 horizon=8, joint=0.2):
    """Task-wise tuning of a composite op, as a compiler tunes a network's subgraphs one by one.

    Each stage is one task: an MCTS over that stage's transformations only, whose objective is the
    stage's own device time, starting from the best program of the tasks before it. Stages go in
    order of their share of P0's time and get samples in proportion (at least 32 each); the last
    `joint` fraction of the samples is one MCTS over every stage from the composed program (with
    `restarts`), which can still trade stages against each other (shared L2, launch gaps). Returns
    what search_best returns, plus the per-task record.
    """
    from paper_2506_01374_gb300 import rc
    root = op.schedule()
    m0 = op.measure([root], io, warmup=2, repeats=5)[0]
    if m0.status != rc.OK:
        raise RuntimeError(f"P0 failed: {rc.STATUS_NAMES.get(m0.status, m0.status)}")
    S = root.num_stages
    share = [max(m0.stage_ms[g], 1e-9) for g in range(S)]
    alloc = [max(32, int(samples * (1.0 - joint) * x / sum(share))) for x in share]
    n, t, tasks = 1, 0.0, []
    for g in sorted(range(S), key=lambda g: -share[g]):
        # one search per task: a stage's space is small enough that restarts mostly re-measure it
        _, best, m, k, cps = search_best(op, io, alloc[g], seed, branching, finalists, 1, surrogate, screen,
                                         horizon, root=root, stages=[g])
        root = best
        tasks.append({"stage": g, "samples": k, "p0_ms": share[g], "best_ms": m.stage_ms[g]})
        n += k
        t += k / cps if cps else 0.0
    search, best, m, k, cps = search_best(op, io, max(16, (samples - n) // max(1, restarts)), seed, branching,
                                          finalists, restarts,
                                          surrogate, screen, horizon, root=root)
    n += k
    t += k / cps if cps else 0.0
    return search, best, m, n, (n / t if t else None), tasks


def random_search(op, io, samples, seed, horizon=8, batch=8):
    """Uniform random search: each candidate is P0 after up to `horizon` random legal transformations."""
    import random

    from paper_2506_01374_gb300 import rc
    rng = random.Random(seed)
    space = op.transform_space()
    seen, n, curve, best = set(), 0, [], float("inf")
    while n < samples:
        cands = []
        for _ in range(64 * batch):
            if len(cands) == batch:
                break
            s = op.schedule()
            for _ in range(rng.randint(1, horizon)):
                try:
                    s = op.schedule(rng.choice(space), base=s)
                except rc.RcError:
                    pass
            key = str(s)
            if key not in seen:
                seen.add(key)
                cands.append(s)
        if not cands:
            break
        for m in op.measure(cands, io, warmup=2, repeats=5):
            n += 1
            if m.status == rc.OK:
                best = min(best, m.ms_median)
            curve.append((n, best))
    return curve


def tasks_curve(op, io, samples, seed, joint=0.2):
    """search_tasks' sequence of searches (one per stage, then one joint), recording every candidate:
    returns [(samples so far, best whole-op median ms so far)]."""
    from paper_2506_01374_gb300 import rc
    root = op.schedule()
    m0 = op.measure([root], io, warmup=2, repeats=5)[0]
    S = root.num_stages
    share = [max(m0.stage_ms[g], 1e-9) for g in range(S)]
    alloc = [max(32, int(samples * (1.0 - joint) * x / sum(share))) for x in share]
    curve = [(1, m0.ms_median)]

    def run(search, budget):
        res, k, pend = [], 0, False
        while k < budget and len(curve) < samples:
            nxt = search.step(res)
            pend = False
            if not nxt:
                break
            res = op.measure(nxt, io, warmup=2, repeats=5)
            pend = True
            for m in res:
                k += 1
                t = m.ms_median if m.status == rc.OK else float("inf")
                curve.append((len(curve) + 1, min(curve[-1][1], t)))
        if pend:
            search.step(res)
        return search.best()[0].clone()

    for g in sorted(range(S), key=lambda g: -share[g]):
        root = run(rc.Search(op, seed=seed, branching=4, surrogate=True, screen=4, stages=[g], root=root), alloc[g])
    run(rc.Search(op, seed=seed, branching=4, surrogate=True, screen=4, root=root), samples)
    return curve


def sample_efficiency(speedup, samples):
    """The paper's sample efficiency: speedup over the untuned program per evaluated sample (Table 1)."""
    return speedup / samples


def efficiency_gain(base_speedup, base_samples, speedup, samples):
    """Sample-efficiency gain of a search over a baseline search (Table 1's last column)."""
    return sample_efficiency(speedup, samples) / sample_efficiency(base_speedup, base_samples)


def sample_reduction(base_samples, samples):
    """Samples the baseline search needed per sample of the other (Table 1's sample reduction)."""
    return base_samples / samples


def geomean(xs):
    import math
    xs = list(xs)
    return math.exp(sum(math.log(x) for x in xs) / len(xs))


def reach(curve, p0_ms):
    """(samples, speedup): the first sample count at which a best-so-far curve [(n, best ms)] reached its
    final best, and that best's speedup over P0 (the reading of Table 1's '# Samples' and 'Speedup')."""
    final = min(b for _, b in curve)
    n = next(n for n, b in curve if b <= final)
    return n, p0_ms / final


def search_study(wl, io, samples, seed, only=""):
    """Best-so-far (TFLOP/s of the best measured candidate) against measured samples, per search variant."""
    from paper_2506_01374_gb300 import rc
    flops = wl.op.info["flops"]
    marks = [m for m in (50, 100, 250, 500, 1000, 2000, 3000, 5000, 10000) if m <= samples] + [samples]
    variants = [("mcts_B2_measured", 2, False, 1), ("mcts_B4_measured", 4, False, 1),
                ("mcts_B4_surrogate_screen4", 4, True, 4), ("random", 0, False, 1)]
    if wl.op.schedule().num_stages > 1:
        variants.append(("tasks_then_joint_B4_surrogate_screen4", 4, True, 4))
    if only:
        variants = [v for v in variants if v[0] in only.split(",")]
    p0 = wl.op.measure([wl.op.schedule()], io, warmup=3, repeats=20)[0].ms_median
    reached = {}
    for sd in (seed, seed + 1):
        for name, B, sur, scr in variants:
            t0 = time.perf_counter()
            if name == "random":
                curve = random_search(wl.op, io, samples, sd)
            elif name.startswith("tasks"):
                curve = tasks_curve(wl.op, io, samples, sd)
            else:
                search = rc.Search(wl.op, seed=sd, branching=B, surrogate=sur, screen=scr)
                res, n, curve, best = [], 0, [], float("inf")
                while n < samples:
                    nxt = search.step(res)
                    if not nxt:
                        break
                    res = wl.op.measure(nxt, io, warmup=2, repeats=5)
                    for m in res:
                        n += 1
                        if m.status == rc.OK:
                            best = min(best, m.ms_median)
                        curve.append((n, best))
            pts = []
            for mk in marks:
                b = min((c[1] for c in curve if c[0] <= mk), default=float("inf"))
                pts.append([mk, round(flops / (b * 1e-3) / 1e12, 1) if b < float("inf") else None])
            n_reach, speedup = reach(curve, p0) if curve else (None, None)
            reached[(name, sd)] = (n_reach, speedup)
            print(json.dumps({"study": "search", "workload": wl.label, "variant": name, "seed": sd,
                              "samples": len(curve), "seconds": round(time.perf_counter() - t0, 1),
                              "p0_ms": p0, "best_tflops_at_samples": pts,
                              "samples_to_best": n_reach, "speedup_over_p0": speedup,
                              "sample_efficiency": sample_efficiency(speedup, n_reach) if curve else None}),
                  flush=True)
    # each variant against unguided random search, as Table 1 sets the LLM-guided MCTS against evolution
    for name, *_ in variants:
        if name == "random":
            continue
        rows = [(reached[(name, sd)], reached[("random", sd)]) for sd in (seed, seed + 1)
                if (name, sd) in reached and ("random", sd) in reached and reached[("random", sd)][0]]
        if not rows:
            continue
        print(json.dumps({"study": "search_summary", "workload": wl.label, "variant": name, "baseline": "random",
                          "speedup_geomean": geomean(v[1] for v, _ in rows),
                          "baseline_speedup_geomean": geomean(r[1] for _, r in rows),
                          "sample_reduction_geomean": geomean(sample_reduction(r[0], v[0]) for v, r in rows),
                          "efficiency_gain_geomean": geomean(efficiency_gain(r[1], r[0], v[1], v[0])
                                                             for v, r in rows)}), flush=True)


def library_study(wl, sched_text="", reps=20):
    """Vendor-library baselines on the workload's inputs (cuDNN attention and convolution, cuBLAS GEMMs,
    called through torch), timed like the search's candidates: inputs resident in HBM, the L2 flushed
    before every repeat, CUDA events around the call, the median reported. Printed as JSON lines, with the
    op's own flop count so the rates compare with the bench line's. With a schedule, this library's
    program is timed in the same process first (same clocks, same inputs). Context for the kernels'
    figures."""
    import statistics

    import numpy as np
    import torch
    import torch.nn.functional as F

    peak = peaks()["bf16_tflops"]
    flush = torch.empty(int(2.5 * 129e6) // 4, dtype=torch.float32, device="cuda")

    def bf16(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda().view(torch.bfloat16)

    def timed(fn):
        for _ in range(3):
            fn()
        ts = []
        for _ in range(reps):
            flush.fill_(1.0)
            # hold the stream about 100 us after the flush, so that the library's host-side dispatch
            # (Python, plan lookup) is done before its kernels' turn: device time only, as for ours
            torch.cuda._sleep(200000)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(b))
        return statistics.median(ts)

    flops = wl.op.info["flops"]
    if sched_text:
        from paper_2506_01374_gb300 import rc
        m = wl.op.measure([parse_schedule(wl.op, sched_text, rc)], wl.device_io(), warmup=3, repeats=reps)[0]
        print(json.dumps({"study": "library", "workload": wl.label, "library": "this repository", "schedule": sched_text,
                          "value": round(m.tflops, 1), "unit": "TFLOP/s", "us": round(m.ms_median * 1e3, 2),
                          "frac": round(m.tflops / peak, 3), "status": m.status}), flush=True)

    def line(lib, fn, note=""):
        try:
            ms = timed(fn)
        except Exception as e:  # a backend this torch build or GPU does not offer
            rec = {"study": "library", "workload": wl.label, "library": lib, "unavailable": str(e).splitlines()[0][:160]}
        else:
            tf = flops / (ms * 1e-3) / 1e12
            rec = {"study": "library", "workload": wl.label, "library": lib, "value": round(tf, 1), "unit": "TFLOP/s",
                   "us": round(ms * 1e3, 2), "frac": round(tf / peak, 3)}
        if note:
            rec["note"] = note
        print(json.dumps(rec), flush=True)

    if wl.name in ("attention", "attention_flux"):
        from torch.nn.attention import SDPBackend, sdpa_kernel
        causal = bool(wl.config["causal"])
        Q, K, V = [bf16(a).transpose(1, 2).contiguous() for a in wl.host[:3]]  # [B][H][S][D]
        gqa = Q.shape[1] != K.shape[1]
        for name, bk in (("cudnn sdpa", SDPBackend.CUDNN_ATTENTION), ("flash sdpa", SDPBackend.FLASH_ATTENTION)):
            def call(bk=bk):
                with sdpa_kernel([bk]):
                    return F.scaled_dot_product_attention(Q, K, V, is_causal=causal, enable_gqa=gqa)
            line(name, call)
    elif wl.name == "conv2d":
        x, w, b = wl.host[:3]
        xt = bf16(x).permute(0, 3, 1, 2)  # NHWC storage seen as NCHW: channels_last
        wt = bf16(w).permute(0, 3, 1, 2)
        bt = bf16(b)
        torch.backends.cudnn.benchmark = True
        line("cudnn conv2d + bias", lambda: F.conv2d(xt, wt, bt, padding=1), "SiLU not included")
        line("cudnn conv2d + bias, then torch SiLU", lambda: F.silu(F.conv2d(xt, wt, bt, padding=1)))
    elif wl.name == "linear":
        X, Wt = bf16(wl.host[0]), bf16(wl.host[1])
        line("cublas matmul", lambda: X @ Wt.t())
    elif wl.name == "mlp":
        X, W1, W2 = [bf16(a) for a in wl.host[:3]]
        I = W2.shape[1]

        def block():
            h = X @ W1.t()
            return (F.silu(h[:, :I]) * h[:, I:]) @ W2.t()
        line("cublas gate/up matmul + torch SiLU/mul + cublas down matmul", block)
    else:
        print(json.dumps({"study": "library", "workload": wl.label, "unavailable": "no library equivalent compared"}))


def rest_gpu(seconds=2.0):
    """Idle the GPU briefly before a final timing. A search keeps it launching back to back for minutes,
    which holds it at its power limit with the SM clock lowered; the measured peaks a fraction divides by
    are those of a kernel timed alone (the burst figures), so the kernel is timed from a rested GPU too.
    The timed work itself is unchanged."""
    import time

    import torch
    torch.cuda.synchronize()
    time.sleep(seconds)


def extra_ops(names, samples, peak_tf, branching=4, restarts=1, surrogate=False, screen=1, moe_samples=None,
              layer_samples=None, hbm_gbs=None):
    """Search each other workload briefly and report its best schedule."""
    import torch

    from paper_2506_01374_gb300 import rc
    hbm_gbs = hbm_gbs or peaks()["hbm_gbs"]
    out = {}
    for name in names:
        wl = Workload(name)
        io = wl.device_io()
        n_s = {"moe": moe_samples, "decoder_layer": layer_samples}.get(name) or samples
        find = search_tasks if wl.tasks else search_best
        _, best, _, n, cps = find(wl.op, io, n_s, branching=branching, restarts=restarts, surrogate=surrogate,
                                  screen=screen, horizon=wl.horizon)[:5]
        rest_gpu()
        m = wl.op.measure([best], io, warmup=3, repeats=20)[0]
        if m.status != rc.OK:
            out[name] = {"workload": wl.label, "error": rc.STATUS_NAMES.get(m.status, m.status)}
            continue
        par = wl.parity(best, io)
        if not par["ok"]:  # a schedule whose output disagrees with the oracle is not reported
            out[name] = {"workload": wl.label, "error": "parity check failed", "parity": par,
                         "schedule": str(best)}
            continue
        tf = wl.op.info["flops"] / (m.ms_median * 1e-3) / 1e12
        peak = FP32_ALU_TFLOPS if wl.bound == "alu" else peak_tf
        gbs = wl.op.info["bytes"] / (m.ms_median * 1e-3) / 1e9
        tr = measured_traffic(wl.label, knob_text(best, wl.dom_stage))
        out[name] = {"workload": wl.label, "tflops": tf, "ms": m.ms_median, "bound": wl.bound, "peak": peak,
                     "frac": tf / peak, "samples": n, "candidates_per_s": cps, "schedule": str(best),
                     "hbm": {"algorithmic_bytes": wl.op.info["bytes"], "achieved_gbs": gbs,
                             "frac_of_hbm_peak": gbs / hbm_gbs,
                             "dominant_kernel_dram_bytes": tr["dram_bytes_per_launch"] if tr else None},
                     "parity": par}
        del io, wl
        torch.cuda.empty_cache()
    return out


def max_over_ranks(vals, world, device):
    """Element-wise maximum of per-rank values over all ranks (the slowest rank's times); one rank: as is."""
    if world <= 1:
        return list(vals)
    import torch
    import torch.distributed as dist
    t = torch.tensor(vals, device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return t.tolist()


def job_tflops(world, flops_per_rank, seconds):
    """Whole-job throughput of `world` replicas that each did `flops_per_rank` in `seconds` (the max over ranks)."""
    return world * flops_per_rank / seconds / 1e12


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args):
    world, rank, _ = dist_setup()
    if rank != 0:
        return
    wl = Workload(args.workload)
    n = args.cpu_sample if args.cpu_sample > 0 else {"mlp": 16, "attention": 32, "conv2d": 512, "moe": 4,
                                                     "gemm_f32": 4, "attention_flux": 16,
                                                     "decoder_layer": 8, "linear": 16}[args.workload]
    for _ in range(args.warmup):
        wl.cpu_sample(n, single_thread=False)
    samples = [wl.cpu_sample(n, single_thread=False) for _ in range(args.steps)]
    secs = statistics.fmean(s["seconds"] for s in samples)
    val = statistics.fmean(s["value"] for s in samples)
    cb = {k: v for k, v in samples[0].items() if k != "seconds"}
    cb["value"] = val
    print(json.dumps({"impl": "reference", "metric": wl.metric, "value": val, "unit": "TFLOP/s", "n_gpus": world,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs,
                      "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
                      "data": "synthetic", "config": dict(workload=wl.label, **wl.config), "cpu_baseline": cb,
                      "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


def launches_per_step(workload, s):
    """Kernels of this library one step of the schedule launches (the L2 flush is a torch fill)."""
    k = [s.knobs(i) for i in range(s.num_stages)]
    if workload == "mlp":
        return (1 if k[0]["fuse"] else 2) + (1 if k[1]["split_k"] == 1 else 2)
    if workload in ("attention", "attention_flux"):
        return 1 + (1 if k[0]["layout"] == 1 else 0)
    if workload == "linear":
        return 1 if k[0]["split_k"] == 1 else 2
    if workload == "conv2d":
        return 1 + (1 if k[0]["split_k"] > 1 else 0) + (1 if (k[0]["split_k"] > 1 or not k[0]["fuse"]) else 0)
    if workload == "moe":
        # routing (3 kernels), gather (unless the gate/up producer gathers), grouped gate/up, grouped
        # down, combine (or, with the atomic combine, the fp32 -> bf16 conversion; the memset is not ours)
        return 3 + (0 if k[1]["location"] == 1 else 1) + 1 + 1 + 1
    if workload == "decoder_layer":
        # RMSNorm, QKV GEMM, RoPE, attention (+ V transpose), O GEMM with the residual, RMSNorm,
        # gate/up GEMM (+ SwiGLU pass), down GEMM with the residual
        return 2 + 1 + 1 + (1 if k[2]["layout"] == 1 else 0) + 2 + (1 if k[4]["fuse"] else 2) + 1
    return 1


def run_ours(args):
    import torch

    from paper_2506_01374_gb300 import rc

    world, rank, local = dist_setup()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    stream = torch.cuda.current_stream()

    wl = Workload(args.workload, parse_shape(args.shape))
    if args.study == "search":
        search_study(wl, wl.device_io(), args.samples, args.seed, args.study_variants)
        return
    if args.study == "library":
        library_study(wl, args.schedule)
        return
    if args.study:
        raise SystemExit(f"unknown --study {args.study}")
    if args.shape:
        wl.label += "_shape_" + args.shape.replace("=", "").replace(",", "_")
        wl.config.update(parse_shape(args.shape))
    op = wl.op
    info = op.info
    io = wl.device_io()

    # 1) schedule search, every candidate measured on the device
    n_meas, cps, best_m = 0, None, None
    search, tasks = None, []
    if args.tasks >= 0:
        wl.tasks = bool(args.tasks)
    if args.schedule:
        best = parse_schedule(op, args.schedule, rc)
    else:
        if args.horizon > 0:
            wl.horizon = args.horizon
        find = search_tasks if wl.tasks else search_best
        search, best, best_m, n_meas, cps, *tasks = find(op, io, args.samples, seed=args.seed, horizon=wl.horizon,
                                                        branching=args.branching, restarts=args.restarts,
                                                        surrogate=bool(args.surrogate), screen=args.screen)

    # 2) timed steps of the best schedule, from a rested GPU (rest_gpu)
    flush = torch.empty(int(2.5 * 129e6) // 4, dtype=torch.float32, device="cuda")
    rest_gpu()
    for _ in range(args.warmup):
        op.run(best, io)
    torch.cuda.synchronize()
    clocks = Clocks(local)
    clocks.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    step_ms, dom_ms = [], []
    for _ in range(args.steps):
        flush.fill_(1.0)
        st = op.run_profiled(best, io, stream)
        step_ms.append(sum(st))
        dom_ms.append(st[wl.dom_stage])
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    ms = statistics.fmean(step_ms)
    ms_dom = statistics.fmean(dom_ms)
    ms, ms_dom = max_over_ranks([ms, ms_dom], world, "cuda")
    value = job_tflops(world, info["flops"], ms * 1e-3)

    # the best schedule's output against the oracle, outside the timed regions
    parity = wl.parity(best, io) if rank == 0 else None
    if parity is not None and not parity["ok"]:
        raise SystemExit(f"parity check of the best schedule failed: {parity} ({best})")

    # 3) end to end through the host-buffer entry point
    e2e_s = None
    if not args.skip_e2e:
        host_io = wl.host_io()
        for _ in range(max(1, args.warmup)):
            op.run_host(best, host_io)
        e2e_t = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            op.run_host(best, host_io)
            e2e_t.append(time.perf_counter() - t0)
        e2e_s = max_over_ranks([statistics.fmean(e2e_t)], world, "cuda")[0]
    h2d, d2h = wl.io_bytes()

    if rank == 0:
        pk = peaks()
        peak = FP32_ALU_TFLOPS if wl.bound == "alu" else pk["bf16_tflops"]
        peak_src = ("derived: 152 SMs x 128 FP32 lanes x 2 x 2.07 GHz" if wl.bound == "alu"
                    else pk["source"] + " bf16 burst")
        achieved = wl.dom_flops / (ms_dom * 1e-3) / 1e12
        traffic = measured_traffic(wl.label, knob_text(best, wl.dom_stage))
        kname = wl.dom_name
        if args.workload == "mlp":
            kname = kname.format(" + fused SwiGLU epilogue" if best.knobs(0)["fuse"] else " + SwiGLU pass")
        out = {
            "metric": wl.metric, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
            "config": dict(workload=wl.label, **wl.config,
                           parallelism="replicas" if world > 1 else "single",
                           l2="flushed between steps (flush outside the timed events)", schedule=str(best)),
            "roofline": {"bound": wl.bound, "kernel": kname, "achieved": achieved, "peak": peak,
                         "unit": "TFLOP/s", "frac": achieved / peak, "peak_source": peak_src,
                         "traffic": traffic["dram_bytes_per_launch"] if traffic else None,
                         "traffic_source": traffic["profile"] if traffic else
                         "no ncu capture of this kernel, schedule and source",
                         "algorithmic_bytes": wl.dom_bytes},
            "step_frac_of_peak": value / world / peak,
            "search": {"samples": n_meas, "candidates_per_s": cps, "surrogate": bool(args.surrogate),
                       "horizon": wl.horizon, "tasks": tasks[0] if tasks else None,
                       "screen": args.screen,
                       "best_search_tflops": best_m.tflops if best_m else None,
                       "stats": search.stats() if search else None},
            "e2e": None if e2e_s is None else {"value": job_tflops(world, info["flops"], e2e_s), "unit": "TFLOP/s",
                                               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": args.steps * launches_per_step(args.workload, best),
            "clocks": clk,
            "parity": parity,
        }
        others = args.ops if args.ops is not None else (
            "gemm_f32,linear,conv2d,attention,attention_flux,moe,decoder_layer" if args.workload == "mlp" else "")
        names = [x for x in others.split(",") if x and x != args.workload]
        if names:
            del io
            torch.cuda.empty_cache()
            out["ops"] = extra_ops(names, args.op_samples, pk["bf16_tflops"], args.branching, args.restarts,
                                   bool(args.surrogate), args.screen, args.moe_samples, args.layer_samples,
                                   pk["hbm_gbs"])
        if args.cpu_sample >= 0:
            cb = wl.cpu_sample(args.cpu_sample)
            cb.pop("seconds", None)
            out["cpu_baseline"] = cb
        else:
            out["cpu_baseline"] = None
        print(json.dumps(out))
    if world > 1:
        torch.distributed.destroy_process_group()


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
