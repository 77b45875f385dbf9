#!/usr/bin/env python
"""Benchmark of the schedule-search hot path on GB300.

Workload (one GPU): the Llama-3-8B-shaped SwiGLU MLP block, bf16, tokens
T=2048, hidden H=4096, intermediate I=14336, weights N(0, 0.02), activations
N(0, 1), synthetic seeded inputs. A run
  1. searches the block's schedule space with the LLM-free MCTS
     (rc_search_step), every candidate timed on the device
     (rc_candidate_measure) -> candidates measured per second;
  2. times K steps of the best schedule found (rc_run_profiled: per-stage
     CUDA events on the launching stream; L2 flushed between steps, outside
     the timed events) -> best-schedule TFLOP/s and the roofline fraction of
     the dominant kernel (the gate/up GEMM with the fused SwiGLU epilogue);
  3. times K end-to-end steps through rc_run_host (pinned host buffers,
     host->device inputs and device->host output inside the timed region);
  4. times the fp64 CPU oracle on a bounded sample of token rows.
Under torchrun (N > 1) every rank runs an independent replica (the path
has no exchange step); value = all ranks' work / the slowest rank's time.

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

T_TOK, HID, INTER = 2048, 4096, 14336
WORKLOAD = "llama3_8b_mlp_swiglu_bf16_T2048_H4096_I14336"
METRIC = "best-schedule TFLOP/s (Llama-3-8B MLP block, bf16)"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--samples", type=int, default=400, help="schedules the search measures")
    ap.add_argument("--cpu-rows", type=int, default=2048,
                    help="token rows of the CPU-oracle sample (0 = skip)")
    ap.add_argument("--schedule", default="",
                    help="fixed schedule instead of a search, e.g. 's0:tile_n=128,stages=4,fuse=1;s1:tile_n=256'")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--ops", default="gemm_f32,conv2d,attention,moe",
                    help="other workloads to search and report per op ('' = none)")
    ap.add_argument("--op-samples", type=int, default=48, help="schedules measured per extra op")
    ap.add_argument("--seed", type=int, default=0)
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
                                          "-lms", "100", "-i", str(self.gpu)], stdout=self.f,
                                         stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

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
        for line in open(self.f.name):
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


def parse_schedule(op, text, rc):
    """'s0:tile_n=128,stages=4;s1:split_k=2' -> schedule (raster=R/G sets loop order and group)."""
    KNOB_T = {"tile_n": (rc.T_TILE_SIZE, 1), "stages": (rc.T_PIPELINE_STAGES, 0), "split_k": (rc.T_SPLIT_K, 0),
              "fuse": (rc.T_FUSE, 0), "raster": (rc.T_LOOP_ORDER, 0), "persistent": (rc.T_PARALLEL, 0)}
    ts = []
    for part in filter(None, text.split(";")):
        stage_s, kvs = part.split(":")
        stage = int(stage_s.strip()[1:])
        for kv in filter(None, kvs.split(",")):
            k, v = kv.split("=")
            kind, axis = KNOB_T[k.strip()]
            if k.strip() == "raster":
                r, g = (v.split("/") + ["1"])[:2]
                ts.append(rc.T(kind, int(r), stage=stage, group=int(g)))
            else:
                ts.append(rc.T(kind, int(v), axis=axis, stage=stage))
    return op.schedule(*ts)


# FP32 SIMT peak of one GB300: 152 SMs x 128 FP32 lanes x 2 flops x 2.07 GHz.
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12


def search_best(op, io, samples, seed=0):
    """MCTS over op's schedule space with device-timed candidates; returns (best, m, n, cand/s)."""
    from paper_2506_01374_gb300 import rc
    search = rc.Search(op, seed=seed)
    res, n, t, pending = [], 0, 0.0, False
    while n < samples:
        nxt = search.step(res)
        pending = False
        if not nxt:
            break
        t0 = time.perf_counter()
        res = op.measure(nxt, io, warmup=2, repeats=5)
        t += time.perf_counter() - t0
        n += len(nxt)
        pending = True
    if pending:  # hand the last batch's measurements to the search
        search.step(res)
    best, m = search.best()
    return search, best, m, n, (n / t if t else None)


def extra_ops(args, peak_tf):
    """Search each other workload of the hot path and report its best schedule."""
    import numpy as np
    import torch

    from paper_2506_01374_gb300 import inputs, rc

    def dev(a):
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16) if a.dtype == np.uint16 else a).cuda()

    out = {}
    for name in [x for x in args.ops.split(",") if x]:
        if name == "gemm_f32":
            A, B, bias = inputs.gemm_f32(256, 256, 256, seed=0)
            op = rc.Op(rc.OP_GEMM_F32, m=256, n=256, k=256, flags=rc.EPI_BIAS | rc.EPI_RELU)
            io = [dev(A), dev(B), dev(bias), torch.empty(256, 256, dtype=torch.float32, device="cuda")]
            wl, bound, peak = "gemm_bias_relu_f32_256^3", "alu", FP32_ALU_TFLOPS
        elif name == "conv2d":
            x, w, b = inputs.conv2d(2, 64, 64, 320, 320, seed=5)
            op = rc.Op(rc.OP_CONV2D, img_n=2, img_h=64, img_w=64, c_in=320, c_out=320, kr=3, ks=3, stride=1, pad=1,
                       flags=rc.EPI_BIAS | rc.EPI_SILU)
            io = [dev(x), dev(w), dev(b), torch.empty(2, 64, 64, 320, dtype=torch.int16, device="cuda")]
            wl, bound, peak = "conv2d_nhwc_3x3_N2_64x64_C320_bias_silu_bf16", "tensor", peak_tf
        elif name == "attention":
            Q, K, V = inputs.attention(1, 2048, 32, 8, 128, seed=4)
            op = rc.Op(rc.OP_ATTENTION, batch=1, seq=2048, heads_q=32, heads_kv=8, head_dim=128, causal=1)
            io = [dev(Q), dev(K), dev(V), torch.empty(1, 2048, 32, 128, dtype=torch.int16, device="cuda"),
                  torch.empty(1, 32, 2048, dtype=torch.float32, device="cuda")]
            wl, bound, peak = "causal_gqa_attention_S2048_Hq32_Hkv8_d128_bf16", "tensor", peak_tf
        elif name == "moe":
            logits, X, W1, W2 = inputs.moe(4096, 7168, 64, 2048, seed=6)
            op = rc.Op(rc.OP_MOE, tokens=4096, hidden=7168, experts=64, inter=2048, top_k=8)
            io = [dev(logits), dev(X), dev(W1), dev(W2), torch.empty(4096, 7168, dtype=torch.int16, device="cuda")]
            del W1, W2
            wl, bound, peak = "moe_T4096_H7168_E64_I2048_top8_bf16", "tensor", peak_tf
        else:
            continue
        search, best, m, n, cps = search_best(op, io, args.op_samples)
        # time the best schedule again with more repeats
        m2 = op.measure([best], io, warmup=3, repeats=20)[0]
        tf = op.info["flops"] / (m2.ms_median * 1e-3) / 1e12
        out[name] = {"workload": wl, "tflops": tf, "ms": m2.ms_median, "bound": bound, "peak": peak,
                     "frac": tf / peak, "samples": n, "candidates_per_s": cps, "schedule": str(best)}
        del io
        torch.cuda.empty_cache()
    return out


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def cpu_oracle_sample(X, W1, W2, rows: int):
    """Time the fp64 oracle on `rows` token rows of the MLP block."""
    import numpy as np

    import oracle
    sel = np.arange(rows, dtype=np.int64) * (X.shape[0] // max(rows, 1))
    oracle.build()
    t0 = time.perf_counter()
    oracle.mlp_bf16(X, W1, W2, rows=sel)
    dt = time.perf_counter() - t0
    flops = 6.0 * rows * HID * INTER
    return {"value": flops / dt / 1e12, "unit": "TFLOP/s", "cores": min(os.cpu_count() or 1, rows),
            "kind": "oracle", "sample": f"{rows} of {T_TOK} token rows of the MLP block, fp64 loop nests",
            "seconds": dt}


def run_reference(args):
    world, rank, _ = dist_setup(args)
    if rank != 0:
        return
    from paper_2506_01374_gb300 import inputs
    X, W1, W2 = inputs.mlp(T_TOK, HID, INTER, seed=1)
    rows = max(1, min(args.cpu_rows, 16))
    for _ in range(args.warmup):
        cpu_oracle_sample(X, W1, W2, rows)
    ts = [cpu_oracle_sample(X, W1, W2, rows)["seconds"] for _ in range(args.steps)]
    ms = 1e3 * sum(ts) / len(ts)
    val = 6.0 * rows * HID * INTER / (ms * 1e-3) / 1e12
    cb = {"value": val, "unit": "TFLOP/s", "cores": min(os.cpu_count() or 1, rows), "kind": "oracle",
          "sample": f"{rows} of {T_TOK} token rows per step, fp64 loop nests"}
    print(json.dumps({"impl": "reference", "metric": METRIC, "value": val, "unit": "TFLOP/s", "n_gpus": world,
                      "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
                      "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
                      "config": {"workload": WORKLOAD, "tokens": T_TOK, "hidden": HID, "inter": INTER},
                      "cpu_baseline": cb,
                      "e2e": {"value": val, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


def run_ours(args):
    import numpy as np
    import torch

    from paper_2506_01374_gb300 import inputs, rc

    world, rank, local = dist_setup(args)
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    stream = torch.cuda.current_stream()

    X, W1, W2 = inputs.mlp(T_TOK, HID, INTER, seed=1)
    dX = torch.from_numpy(X.view(np.int16)).cuda()
    d1 = torch.from_numpy(W1.view(np.int16)).cuda()
    d2 = torch.from_numpy(W2.view(np.int16)).cuda()
    dY = torch.empty(T_TOK, HID, dtype=torch.int16, device="cuda")
    io = [dX, d1, d2, dY]
    op = rc.Op(rc.OP_MLP, m=T_TOK, n=INTER, k=HID)
    info = op.info

    # 1) schedule search, every candidate measured on the device
    search = rc.Search(op, seed=args.seed)
    res, n_meas, t_search = [], 0, 0.0
    if args.schedule:
        best = parse_schedule(op, args.schedule, rc)
        best_m = None
    else:
        search, best, best_m, n_meas, cps = search_best(op, io, args.samples, seed=args.seed)
        t_search = n_meas / cps if cps else 0.0

    # 2) timed steps of the best schedule
    flush = torch.empty(int(2.5 * 129e6) // 4, dtype=torch.float32, device="cuda")
    for _ in range(args.warmup):
        op.run(best, io)
    torch.cuda.synchronize()
    clocks = Clocks(local)
    clocks.start()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    step_ms, stage0_ms = [], []
    for _ in range(args.steps):
        flush.fill_(1.0)
        st = op.run_profiled(best, io, stream)
        step_ms.append(sum(st))
        stage0_ms.append(st[0])
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    clk = clocks.stop()
    ms = statistics.fmean(step_ms)
    ms_stage0 = statistics.fmean(stage0_ms)
    if world > 1:
        t = torch.tensor([ms, ms_stage0], device="cuda", dtype=torch.float64)
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms, ms_stage0 = t.tolist()
    value = world * info["flops"] / (ms * 1e-3) / 1e12

    # 3) end to end through the host-buffer entry point
    hX = torch.from_numpy(X.view(np.int16)).pin_memory().numpy()
    h1 = torch.from_numpy(W1.view(np.int16)).pin_memory().numpy()
    h2 = torch.from_numpy(W2.view(np.int16)).pin_memory().numpy()
    hY = torch.empty(T_TOK, HID, dtype=torch.int16).pin_memory().numpy()
    host_io = [hX, h1, h2, hY]
    e2e_s = None
    if not args.skip_e2e:
        for _ in range(max(1, args.warmup)):
            op.run_host(best, host_io)
        e2e_t = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            op.run_host(best, host_io)
            e2e_t.append(time.perf_counter() - t0)
        e2e_s = statistics.fmean(e2e_t)
        if world > 1:
            t = torch.tensor([e2e_s], device="cuda", dtype=torch.float64)
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            e2e_s = t.item()
    h2d = X.nbytes + W1.nbytes + W2.nbytes
    d2h = T_TOK * HID * 2

    if rank == 0:
        pk = peaks()
        gate_up_flops = 2.0 * T_TOK * (2 * INTER) * HID
        achieved = gate_up_flops / (ms_stage0 * 1e-3) / 1e12
        k0, k1 = best.knobs(0), best.knobs(1)
        launches_per_step = (1 if k0["fuse"] else 2) + (1 if k1["split_k"] == 1 else 2)
        kname = "gate/up GEMM" + (" + fused SwiGLU epilogue" if k0["fuse"] else " + SwiGLU pass") + " (stage 0)"
        out = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": WORKLOAD, "tokens": T_TOK, "hidden": HID, "inter": INTER,
                       "parallelism": "replicas" if world > 1 else "single",
                       "l2": "flushed between steps (flush outside the timed events)",
                       "schedule": str(best)},
            "roofline": {"bound": "tensor", "kernel": kname,
                         "achieved": achieved, "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": achieved / pk["bf16_tflops"], "peak_source": pk["source"] + " bf16 burst",
                         "traffic": None},
            "step_frac_of_peak": value / world / pk["bf16_tflops"],
            "search": {"samples": n_meas, "candidates_per_s": n_meas / t_search if t_search else None,
                       "best_search_tflops": best_m.tflops if best_m else None, "stats": search.stats()},
            "e2e": None if e2e_s is None else {"value": world * info["flops"] / e2e_s / 1e12, "unit": "TFLOP/s",
                                               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h},
            "gpu_launches": args.steps * launches_per_step,
            "clocks": clk,
        }
        if args.ops:
            out["ops"] = extra_ops(args, pk["bf16_tflops"])
        if args.cpu_rows > 0:
            out["cpu_baseline"] = cpu_oracle_sample(X, W1, W2, args.cpu_rows)
            out["cpu_baseline"].pop("seconds", None)
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
