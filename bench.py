"""Benchmark: one DQT training step of a ternary LLaMA MLP GEMM set on GB300.

Workload (the headline configuration): hidden 2048, intermediate 5632,
tokens 8192 (batch 4 x seq 2048); BitLinear gate and up [2048 -> 5632] and
down [5632 -> 2048], ternary int8 codes from AbsMean of N(0, 0.02), bf16
activations ~ N(0, 1), upstream gradients ~ N(0, 1e-2), AdamW moments fp32.
The down projection's input is a synthetic N(0, 1) activation (no SwiGLU on
the measured path).  One step runs, through the C ABI:

  act_quant(X)  -> codes image + dequantised X (shared by gate and up)
  act_quant(H)  -> the same for the down projection's input
  codes_to_bf16 for the three weights (exact images of the int8 codes)
  forward GEMM  x3, dX GEMM x3, fused dW GEMM + AdamW + SR update x3

Metric: tokens/s of the whole step (higher is better).  `value` is timed with
CUDA events on the launching stream with inputs resident in HBM; `e2e` adds,
every step, the pinned-host -> device copy of that step's activations and
gradients and the device -> host read of the step's changed-code counts.
The step's working set (~1.5 GB) is far larger than the 129 MB L2, so no
flush is needed between steps.

`--act fp8` runs the FP8-environment variant of the same step (Sec. 4.3):
E4M3 activations and weight images, and the forward GEMMs on the 8-bit
floating-point tensor cores (kind::f8f6f4); the backward is unchanged.

`--optimizer adafactor` replaces the fused AdamW epilogue by Adafactor with
SR (gradient GEMM, factored statistics, per-element step; Sec. 4.3) and
`--packed` stores the ternary codes 2 bits each (Sec. 1).

`--impl reference` times the CPU oracle instead (bounded sample of the same
step, extrapolated).  Under torchrun each rank runs an independent replica
(weak scaling, no collective on the data path).
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

T_TOK, HID, INTER = 8192, 2048, 5632
WORKLOAD = "ternary DQT LLaMA MLP GEMM set (gate/up 2048->5632, down 5632->2048), 8192 tokens"
METRIC = "DQT BitLinear fwd+bwd+SR-update tokens/s"
PROJ = [("gate", HID, INTER), ("up", HID, INTER), ("down", INTER, HID)]


# the device code of the GEMM kernels and of the streaming update that
# finishes the weight-gradient GEMM's last wave
GEMM_SOURCES = ("gemm_tc.cu", "dqt_device.cuh", "sr_update.cu")


def kernel_fingerprint(files=GEMM_SOURCES):
    """Short hash of the GEMM kernels' sources, comments and layout left out:
    the ncu counters quoted below belong to one version of the code."""
    import hashlib
    import re
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2412_04787_gb300", "csrc")
    for f in files:
        with open(os.path.join(csrc, f), encoding="utf-8") as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        src = " ".join(src.split())
        h.update(f.encode() + b"\0" + src.encode())
    return h.hexdigest()[:12]


# DRAM bytes (read + write) of one gate-shape call of the fused dW + update
# (T=8192, K=2048, N=5632: the 2-SM GEMM and the streaming kernel that
# finishes its last-wave tiles; the up and down calls move the same numbers
# of operand and optimiser-state bytes), from one ncu capture, keyed by the
# GEMM-source fingerprint it was taken on (see profiles/).  A stale entry
# reports null.
# With gate and up stacked, the mean over the step's two dW launches (the
# stacked gate/up call and the down call, each its GEMM and streaming kernel).
DW_TRAFFIC_STACKED = {"e8a6edbac357": ((499344640 + 147830784)
                                         + (258470912 + 57011456 + 33059840 + 256)) // 2,
                      "58ba5df98181": ((464767488 + 147933696)
                                         + (258423552 + 57020416 + 33059584 + 256)) // 2,
                      "769ac7621d63": ((563601152 + 158165760)
                                         + (259388672 + 57002752 + 33059840 + 3328)) // 2,
                      "b62587c26333": ((563893248 + 158965760)
                                         + (259276032 + 57066240 + 33059328 + 256)) // 2,
                      "e40fd6702992": ((516993536 + 147382272)
                                         + (259118848 + 57005568 + 33063680 + 768)) // 2}
# DRAM bytes (read + write, ncu) of the grouped launch of both dW problems
DW_TRAFFIC_GROUP = {"7eaccd5d9509": 873590272 + 328523520}
DW_TRAFFIC_BYTES = {"ac36c0aa63c5": 261135360 + 57050112 + 33049600,
                    "82d12725fdfa": 262571008 + 61169152 + 33047808,
                    "a25cf8632190": 261430272 + 59386112 + 33048064}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return d, "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index, window="the timed region"):
        self.index = index
        self.window = window
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.out, _ = self.proc.communicate()

    def summary(self):
        rows = []
        for line in (self.out or "").strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) >= 9:
                rows.append(f)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"],
                    "window": self.window}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows), "window": self.window}


class MLPStep:
    """Device buffers and the launch sequence of one DQT MLP training step."""

    def __init__(self, dev, seed=1234, fp8=False, optimizer="adamw", packed=False, bits=1.58,
                 operands="int8", tail_slices=True, stack_gate_up=False, next_image=True,
                 dw_group=False):
        from paper_2412_04787_gb300 import dqt, inputs

        self.dqt = dqt
        self.dev = dev
        self.fp8 = fp8
        self.optimizer = optimizer
        self.packed = packed
        self.bits = bits
        # int8: the hot-path C ABI on int8 codes (no operand images in HBM for
        # the forward; dX and dW convert into per-stream workspaces); img: the
        # *_img calls on images shared between GEMMs (the FP8, packed and
        # Adafactor variants always take images)
        self.i8 = operands == "int8" and not fp8 and not packed and optimizer == "adamw"
        # gate and up as two stacked weights of one call (the forward and the
        # fused dW + update; dX stays per weight): image operands, AdamW, int8
        # codes
        self.stack = stack_gate_up and not self.i8 and not packed and optimizer == "adamw"
        # the step's two weight-gradient problems (gate and up stacked, and
        # down) in one persistent launch (dqt_bitlinear_bwd_dw_update_group)
        self.group = dw_group and self.stack
        self.grid = dqt.grid(bits)
        # FP8 forward on codes beyond 16 in magnitude: the split E4M3 image
        # [N, 2K] (dqt_codes_to_fp8_split's layout, written by the update like
        # the other images)
        self.w8_split = fp8 and dqt.fp8_split_grid(self.grid)
        T = T_TOK
        # two seeded input sets, alternated step by step, so that the
        # optimiser sees changing gradients as in training
        self.host_sets = []
        for r in range(2):
            h = {"X": inputs.normal((T, HID), 1.0, seed=1 + 100 * r, dtype=torch.bfloat16),
                 "H": inputs.normal((T, INTER), 1.0, seed=2 + 100 * r, dtype=torch.bfloat16)}
            for i, (name, K, N) in enumerate(PROJ):
                h["dY_" + name] = inputs.normal((T, N), 1e-2, seed=10 + i + 100 * r,
                                                dtype=torch.bfloat16)
            if self.stack:
                # the gradient of the stacked output [gate | up] as a SwiGLU
                # backward writes it; the dX GEMMs read each half in place
                h["dY_gu"] = torch.cat([h.pop("dY_gate"), h.pop("dY_up")], dim=1)
            self.host_sets.append(h)
        self.host = self.host_sets[0]
        self.dev_sets = [{k: v.to(dev) for k, v in h.items()} for h in self.host_sets]
        if self.stack:
            for d in self.dev_sets:
                d["dY_gate"], d["dY_up"] = d["dY_gu"][:, :INTER], d["dY_gu"][:, INTER:]
        self.d = self.dev_sets[0]
        self.alternate = True
        self.W, self.s_w, self.m, self.v, self.W_img, self.Y, self.dX, self.Xdq = {}, {}, {}, {}, {}, {}, {}, {}
        self.W8 = {}
        if self.stack:
            # one buffer of codes, moments and image for both weights; each
            # weight's own per-tensor scale
            self.W_gu = torch.empty((2 * INTER, HID), dtype=torch.int8, device=dev)
            self.m_gu = torch.zeros((2 * INTER, HID), dtype=torch.float32, device=dev)
            self.v_gu = torch.zeros((2 * INTER, HID), dtype=torch.float32, device=dev)
            self.W_img_gu = torch.empty((2 * INTER, HID), dtype=torch.bfloat16, device=dev)
            if fp8:
                self.W8_gu = torch.empty((2 * INTER, HID * (2 if self.w8_split else 1)),
                                         dtype=torch.uint8, device=dev)
            self.Y_gu = torch.empty((T, 2 * INTER), dtype=torch.bfloat16, device=dev)
        for i, (name, K, N) in enumerate(PROJ):
            W0 = inputs.normal((N, K), 0.02, seed=20 + i).to(dev)
            self.W[name], self.s_w[name] = dqt.dqt_absmean_init(W0, self.grid)
            del W0
            if self.stack and name in ("gate", "up"):
                half = slice(0, INTER) if name == "gate" else slice(INTER, 2 * INTER)
                self.W_gu[half].copy_(self.W[name])
                self.W[name] = self.W_gu[half]
                self.m[name], self.v[name] = self.m_gu[half], self.v_gu[half]
                self.W_img[name] = self.W_img_gu[half]
                if fp8:
                    self.W8[name] = self.W8_gu[half]
                self.Y[name] = self.Y_gu[:, half]
                self.dX[name] = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
                continue
            if packed:
                self.W[name] = dqt.dqt_pack_ternary(self.W[name])
            if optimizer == "adamw":
                self.m[name] = torch.zeros((N, K), dtype=torch.float32, device=dev)
                self.v[name] = torch.zeros((N, K), dtype=torch.float32, device=dev)
            else:  # Adafactor's factored statistics (row and column means)
                self.m[name] = torch.zeros(N, dtype=torch.float32, device=dev)
                self.v[name] = torch.zeros(K, dtype=torch.float32, device=dev)
            if not self.i8:  # the int8-operand calls make their images in workspaces
                self.W_img[name] = torch.empty((N, K), dtype=torch.bfloat16, device=dev)
            if fp8:
                self.W8[name] = torch.empty((N, K * (2 if self.w8_split else 1)), dtype=torch.uint8,
                                            device=dev)
            self.Y[name] = torch.empty((T, N), dtype=torch.bfloat16, device=dev)
            self.dX[name] = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
        # image operands with AdamW on int8 codes: each weight-gradient call
        # writes the image of the codes it updates into the second of two
        # image buffers (the next step's forward and dX operand), so that no
        # step converts codes to images; the buffers swap after every step
        # (with the FP8 forward, the E4M3 image of the forward beside the bf16
        # image of dX, both written by the update)
        self.nimg = next_image and not self.i8 and not packed and optimizer == "adamw"
        if self.nimg:
            self.W_img_next, self.W8_next = {}, {}
            if self.stack:
                self.W_img_gu_next = torch.empty_like(self.W_img_gu)
                if fp8:
                    self.W8_gu_next = torch.empty_like(self.W8_gu)
            for name, K, N in PROJ:
                if self.stack and name in ("gate", "up"):
                    half = slice(0, INTER) if name == "gate" else slice(INTER, 2 * INTER)
                    self.W_img_next[name] = self.W_img_gu_next[half]
                    if fp8:
                        self.W8_next[name] = self.W8_gu_next[half]
                else:
                    self.W_img_next[name] = torch.empty((N, K), dtype=torch.bfloat16, device=dev)
                    if fp8:
                        self.W8_next[name] = torch.empty_like(self.W8[name])
                dqt.dqt_codes_to_bf16(self.W[name], self.W_img[name])  # the first step's images
                if fp8 and self.w8_split:
                    dqt.dqt_codes_to_fp8_split(self.W[name], self.W8[name])
                elif fp8:
                    dqt.dqt_codes_to_fp8(self.W[name], self.grid, self.W8[name])
        # per activation: (scale, forward operand, dequantised bf16 image); the
        # forward operand is the int8 codes (no image), the bf16 code image,
        # or the E4M3 bytes with fp8
        self.aq = {}
        for src, K in (("X", HID), ("H", INTER)):
            self.aq[src] = (torch.empty(T, dtype=torch.float32, device=dev),
                            torch.empty((T, K), dtype=(torch.int8 if self.i8 else
                                                       torch.uint8 if fp8 else torch.bfloat16),
                                        device=dev),
                            None if self.i8 else
                            torch.empty((T, K), dtype=torch.bfloat16, device=dev))
        self.changed = torch.zeros(3, dtype=torch.int64, device=dev)
        self.af_ws = None
        if optimizer == "adafactor":
            nb = max(dqt.dqt_bwd_dw_adafactor_workspace_size(T, N, K) for _, K, N in PROJ)
            # one workspace per concurrent stream (gate and up run side by side)
            self.af_ws = [torch.empty(nb, dtype=torch.uint8, device=dev) for _ in range(4)]
        self.sr = {name: dqt.sr_stream(seed=seed, tensor_id=i) for i, (name, _, _) in enumerate(PROJ)}
        self.step_no = 0
        # weight-gradient workspace, one per stream: with int8 operands the
        # X_tilde image first, then the token-sliced last wave's partials
        if self.i8:
            nbw = max(dqt.dqt_bwd_dw_workspace_size(T, N, K) for _, K, N in PROJ)
            self.dw_ws = [torch.empty(nbw, dtype=torch.uint8, device=dev) for _ in range(4)]
            nbx = max(dqt.dqt_bwd_dx_workspace_size(T, N, K) for _, K, N in PROJ)
            self.dx_ws = [torch.empty(nbx, dtype=torch.uint8, device=dev) for _ in range(4)]
            nbf = max(dqt.dqt_fwd_workspace_size(T, K, N) for _, K, N in PROJ)
            self.fwd_ws = [torch.empty(nbf, dtype=torch.uint8, device=dev) for _ in range(4)]
        else:
            nbw = max(dqt.dqt_bwd_dw_img_workspace_size(T, N, K) for _, K, N in PROJ)
            self.dw_ws = [torch.empty(max(nbw, 16), dtype=torch.uint8, device=dev) if nbw else False
                          for _ in range(4)]
        # forward and dX workspace for the partials of their sliced last wave,
        # one per stream (the GEMMs of one stream run one after the other)
        nbt = max(max(dqt.dqt_fwd_img_workspace_size(T, K, N),
                      dqt.dqt_bwd_dx_img_workspace_size(T, N, K)) for _, K, N in PROJ)
        self.tail_ws = [torch.empty(max(nbt, 16), dtype=torch.uint8, device=dev)
                        if nbt and tail_slices else False for _ in range(4)]
        # kernel launches per step: act_quant 2, weight images 3 (+3 E4M3),
        # forward 3, dX 3, and per projection the dW GEMM, the streaming
        # kernel of its sliced last wave (when the shape has one), and for
        # Adafactor the five statistics kernels and the step; with int8
        # operands each forward call converts both operands (3 x 2 images
        # instead of the 3 shared weight images), each dX call the weight
        # and each dW call X_tilde (3 + 3)
        dw = [1 + (1 if dqt.dqt_bwd_dw_img_workspace_size(T, N, K) > 0 else 0) for _, K, N in PROJ]
        # (the forward's and dX's cut last wave is summed inside the GEMM: no
        # launch of its own)
        self.launches_per_step = 2 + 3 + 3 + 3 + sum(dw) + (3 if fp8 else 0) + (6 if self.i8 else 0)
        if self.stack:
            # one weight image (two with FP8), one forward and one dW call for
            # gate and up
            nbp = dqt.dqt_bwd_dw_img_workspace_size(T, 2 * INTER, HID)
            self.launches_per_step = (2 + self.conversions() + 2 + 3 +
                                      (1 if self.group else (1 + (1 if nbp > 0 else 0)) + dw[2]))
            if nbp > max(nbw, 16):
                self.dw_ws = [torch.empty(nbp, dtype=torch.uint8, device=dev) for _ in range(4)]
            nbt = max(nbt, dqt.dqt_fwd_img_workspace_size(T, HID, 2 * INTER))
            self.tail_ws = [torch.empty(max(nbt, 16), dtype=torch.uint8, device=dev)
                            if nbt and tail_slices else False for _ in range(4)]
        if self.nimg:  # the images come from the update: no conversion launches
            self.launches_per_step -= self.conversions()
        self.dw_kind = "bwd_dw_adafactor" if optimizer == "adafactor" else "bwd_dw_update"
        if self.i8:
            self.kinds = ["act_quant", "codes_to_bf16", "fwd", "bwd_dx", "codes_to_xdq",
                          self.dw_kind]
        else:
            self.kinds = (["act_quant_fp8", "codes_to_fp8", "codes_to_bf16", "fwd_fp8"] if fp8 else
                          ["act_quant", "codes_to_bf16", "fwd"]) + ["bwd_dx", self.dw_kind]
        if optimizer == "adafactor":
            self.launches_per_step += 3 * 6
        if self.nimg:  # no conversion launches: the updates write the images
            self.kinds = [k for k in self.kinds if k not in ("codes_to_bf16", "codes_to_fp8")]

        # streams 0-2 carry the step's critical chain (act_quant X -> gate/up
        # forward -> act_quant H -> down forward -> down dX -> gate/up
        # backward); the down projection's dW (stream 3) is off it, so its
        # blocks take the SMs only when the chain leaves some free
        self.streams = [torch.cuda.Stream(device=dev, priority=-1 if i < 3 else 0) for i in range(4)]
        self.dp = None

    def conversions(self):
        """Weight-image conversion launches per step with image operands: one
        per weight buffer (gate and up stacked: one buffer), twice with the
        FP8 forward (E4M3 and bf16)."""
        return (2 if self.stack else 3) * (2 if self.fp8 else 1)

    def enable_dp(self):
        """Data-parallel exchange per weight (one rank per GPU): the dW GEMM
        writes the rank's fp32 gradient; then a reduce-scatter, the AdamW + SR
        update of this rank's shard (its moments only, ZeRO-1) and an
        all-gather of the int8 codes (paper_2412_04787_gb300/dp.py)."""
        from paper_2412_04787_gb300 import dp
        if self.packed or self.optimizer != "adamw":
            raise SystemExit("the data-parallel exchange runs the AdamW step on int8 codes")
        if self.nimg:  # the shard update writes codes only: images by conversion again
            self.launches_per_step += self.conversions()
            self.nimg = False
        self.group = False
        self.dp = {}
        for name, _, _ in PROJ:
            upd = dp.DataParallelUpdater(self.W[name])
            self.dp[name] = upd
            self.W[name] = upd.codes_view()  # the GEMMs read the gathered codes
            self.m[name] = self.v[name] = None
        # per projection: the shard's update kernel (the collectives are NCCL's)
        self.launches_per_step += len(PROJ)
        self.kinds = [k for k in self.kinds if k != self.dw_kind] + ["bwd_dw", "dp_exchange"]

    def run(self, timers=None, serial=False):
        """Enqueue one step.  The launches follow the dependency graph of a
        LLaMA MLP (gate and up read the same quantised X; the down projection
        reads the SwiGLU output H, here a synthetic stand-in that still waits
        for both forwards; each projection's dX and dW are independent; the
        gate/up backward waits for the down projection's dX) on four streams
        joined at the end, so that the persistent kernels fill each other's
        last-wave idle SMs.  `timers` maps a kernel kind to a list that
        receives (start, end) CUDA events recorded on the kernel's stream."""
        dqt = self.dqt
        self.step_no += 1
        if self.alternate:
            self.d = self.dev_sets[self.step_no % 2]
        hp = dqt.adamw(lr=1e-3, step=self.step_no)
        main = torch.cuda.current_stream()
        # serial: the same launches, in the same order, all on the current stream
        s = [main] * 4 if serial else self.streams

        def timed(kind, stream, fn):
            with torch.cuda.stream(stream):
                if timers is not None and kind in timers:
                    a = torch.cuda.Event(enable_timing=True)
                    b = torch.cuda.Event(enable_timing=True)
                    a.record(stream)
                    fn()
                    b.record(stream)
                    timers[kind].append((a, b))
                else:
                    fn()

        def after(stream, *others):
            for o in others:
                if o is stream:
                    continue
                e = torch.cuda.Event()
                e.record(o)
                stream.wait_event(e)

        # per-kernel timing (timers given) runs the conversion inside each
        # int8 dX / dW call as its own launch, on the same workspace slices,
        # so that each kernel is timed alone; the launches are the same
        parts = timers is not None

        def aq(src, stream):
            s_x, q_img, xdq = self.aq[src]
            if self.i8:
                timed("act_quant", stream, lambda: dqt.dqt_act_quant(self.d[src], q_img, s_x))
            elif self.fp8:
                timed("act_quant_fp8", stream,
                      lambda: dqt.dqt_act_quant_fp8(self.d[src], q_img, s_x, xdq))
            else:
                timed("act_quant", stream,
                      lambda: dqt.dqt_act_quant_images(self.d[src], None, s_x, q_img, xdq, want=()))

        def codes(name, stream):
            if name == "gate_up":  # both stacked weights' image in one launch
                if self.fp8:
                    timed("codes_to_fp8", stream,
                          lambda: dqt.dqt_codes_to_fp8_split(self.W_gu, self.W8_gu) if self.w8_split
                          else dqt.dqt_codes_to_fp8(self.W_gu, self.grid, self.W8_gu))
                timed("codes_to_bf16", stream,
                      lambda: dqt.dqt_codes_to_bf16(self.W_gu, self.W_img_gu))
                return
            shape = tuple(self.W_img[name].shape)
            if self.fp8:
                timed("codes_to_fp8", stream,
                      lambda: dqt.dqt_packed_to_fp8(self.W[name], shape, self.W8[name]) if self.packed
                      else dqt.dqt_codes_to_fp8_split(self.W[name], self.W8[name]) if self.w8_split
                      else dqt.dqt_codes_to_fp8(self.W[name], self.grid, self.W8[name]))
            timed("codes_to_bf16", stream,
                  lambda: dqt.dqt_packed_to_bf16(self.W[name], shape, self.W_img[name]) if self.packed
                  else dqt.dqt_codes_to_bf16(self.W[name], self.W_img[name]))

        def fwd(name, stream):
            s_x, q_img, _ = self.aq["H" if name == "down" else "X"]
            if name == "gate_up" and self.fp8:  # the stacked E4M3 weights
                timed("fwd_fp8", stream, lambda: dqt.dqt_bitlinear_fwd_fp8_pair(
                    q_img, s_x, self.W8_gu, INTER, self.s_w["gate"], self.s_w["up"], self.grid,
                    Y=self.Y_gu))
                return
            if name == "gate_up":  # the stacked weights, [gate | up] in one output
                timed("fwd", stream, lambda: dqt.dqt_bitlinear_fwd_img_pair(
                    q_img, s_x, self.W_img_gu, INTER, self.s_w["gate"], self.s_w["up"], self.grid,
                    Y=self.Y_gu, ws=self.tail_ws[s.index(stream)]))
                return
            if self.i8:
                ws = self.fwd_ws[s.index(stream)]
                if parts:
                    W = self.W[name]
                    (T_, K_), N_ = q_img.shape, W.shape[0]
                    a_bytes = (T_ * K_ * 2 + 255) // 256 * 256
                    w_bytes = (N_ * K_ * 2 + 255) // 256 * 256
                    qi = ws[: T_ * K_ * 2].view(torch.bfloat16).view(T_, K_)
                    wi = ws[a_bytes: a_bytes + N_ * K_ * 2].view(torch.bfloat16).view(N_, K_)
                    tail = ws[a_bytes + w_bytes:]
                    timed("codes_to_bf16", stream, lambda: dqt.dqt_codes_to_bf16(q_img, qi))
                    timed("codes_to_bf16", stream, lambda: dqt.dqt_codes_to_bf16(W, wi))
                    timed("fwd", stream, lambda: dqt.dqt_bitlinear_fwd_img(
                        qi, s_x, wi, self.s_w[name], self.grid, Y=self.Y[name],
                        ws=tail if tail.numel() else False))
                else:
                    dqt.dqt_bitlinear_fwd(q_img, s_x, self.W[name], self.s_w[name], self.grid,
                                          Y=self.Y[name], ws=ws)
            elif self.fp8:
                timed("fwd_fp8", stream, lambda: dqt.dqt_bitlinear_fwd_fp8(
                    q_img, s_x, self.W8[name], self.s_w[name], self.grid, Y=self.Y[name]))
            else:
                timed("fwd", stream, lambda: dqt.dqt_bitlinear_fwd_img(
                    q_img, s_x, self.W_img[name], self.s_w[name], self.grid, Y=self.Y[name],
                    ws=self.tail_ws[s.index(stream)]))

        def dx(name, stream):
            if self.i8:
                ws = self.dx_ws[s.index(stream)]
                if parts:
                    nb = 2 * self.W[name].numel()
                    img = ws[: nb].view(torch.bfloat16).view(self.W[name].shape)
                    tail = ws[(nb + 255) // 256 * 256:]
                    timed("codes_to_bf16", stream,
                          lambda: dqt.dqt_codes_to_bf16(self.W[name], img))
                    timed("bwd_dx", stream, lambda: dqt.dqt_bitlinear_bwd_dx_img(
                        self.d["dY_" + name], img, self.s_w[name], dX=self.dX[name],
                        ws=tail if tail.numel() else False))
                else:
                    dqt.dqt_bitlinear_bwd_dx(self.d["dY_" + name], self.W[name], self.s_w[name],
                                             dX=self.dX[name], ws=ws)
                return
            timed("bwd_dx", stream, lambda: dqt.dqt_bitlinear_bwd_dx_img(
                self.d["dY_" + name], self.W_img[name], self.s_w[name], dX=self.dX[name],
                ws=self.tail_ws[s.index(stream)]))

        def dw_group(stream):
            nimg = self.nimg
            timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_group([
                dict(dY=self.d["dY_gu"], Xdq=self.aq["X"][2], W=self.W_gu, m=self.m_gu, v=self.v_gu,
                     N0=INTER, s_w0=self.s_w["gate"], s_w1=self.s_w["up"], sr0=self.sr["gate"],
                     sr1=self.sr["up"], W_img_next=self.W_img_gu_next if nimg else None,
                     W8_next=self.W8_gu_next if nimg and self.fp8 else None,
                     changed_out=self.changed[0:1]),
                dict(dY=self.d["dY_down"], Xdq=self.aq["H"][2], W=self.W["down"], m=self.m["down"],
                     v=self.v["down"], s_w0=self.s_w["down"], sr0=self.sr["down"],
                     W_img_next=self.W_img_next["down"] if nimg else None,
                     W8_next=self.W8_next["down"] if nimg and self.fp8 else None,
                     changed_out=self.changed[2:3])], hp, self.grid))

        def dw(i, name, stream):
            xdq = self.aq["H" if name == "down" else "X"][2]
            ch = self.changed[i:i + 1]
            if name == "gate_up":  # the stacked weights, each with its scale and stream
                ws = self.dw_ws[s.index(stream)]
                timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img_pair(
                    self.d["dY_gu"], xdq, self.W_gu, INTER, self.s_w["gate"], self.s_w["up"],
                    self.m_gu, self.v_gu, hp, self.sr["gate"], self.sr["up"], self.grid,
                    changed_out=ch, ws=ws, W_img_next=self.W_img_gu_next if self.nimg else None,
                    W8_next=self.W8_gu_next if self.nimg and self.fp8 else None))
                return
            if self.dp and not self.i8:
                upd = self.dp[name]
                ws = self.dw_ws[s.index(stream)]
                timed("bwd_dw", stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img(
                    self.d["dY_" + name], xdq, None, self.s_w[name], None, None, None, None,
                    self.grid, dW_out=upd.grad_view(), ws=ws))
                timed("dp_exchange", stream, lambda: upd.step(
                    self.s_w[name], hp, self.sr[name], self.grid, changed_out=ch))
                return
            if self.i8 and self.dp:
                s_x, q, _ = self.aq["H" if name == "down" else "X"]
                upd = self.dp[name]
                ws = self.dw_ws[s.index(stream)]
                if parts:  # the call's conversion and gradient GEMM, timed apart
                    T_, K_ = q.shape
                    img_bytes = (T_ * K_ * 2 + 255) // 256 * 256
                    img = ws[: T_ * K_ * 2].view(torch.bfloat16).view(T_, K_)
                    rest = ws[img_bytes:]
                    timed("codes_to_xdq", stream, lambda: dqt.dqt_codes_to_xdq(q, s_x, img))
                    timed("bwd_dw", stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img(
                        self.d["dY_" + name], img, None, self.s_w[name], None, None, None, None,
                        self.grid, dW_out=upd.grad_view(), ws=rest if rest.numel() else False))
                else:
                    dqt.dqt_bitlinear_bwd_dw_update(
                        self.d["dY_" + name], q, s_x, None, self.s_w[name], None, None, None, None,
                        self.grid, dW_out=upd.grad_view(), ws=ws)
                timed("dp_exchange", stream, lambda: upd.step(
                    self.s_w[name], hp, self.sr[name], self.grid, changed_out=ch))
                return
            if self.i8:
                s_x, q, _ = self.aq["H" if name == "down" else "X"]
                ws = self.dw_ws[s.index(stream)]
                if parts:
                    T_, K_ = q.shape
                    img_bytes = (T_ * K_ * 2 + 255) // 256 * 256
                    img = ws[: T_ * K_ * 2].view(torch.bfloat16).view(T_, K_)
                    rest = ws[img_bytes:]
                    timed("codes_to_xdq", stream, lambda: dqt.dqt_codes_to_xdq(q, s_x, img))
                    timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img(
                        self.d["dY_" + name], img, self.W[name], self.s_w[name], self.m[name],
                        self.v[name], hp, self.sr[name], self.grid, changed_out=ch,
                        ws=rest if rest.numel() else False))
                else:
                    dqt.dqt_bitlinear_bwd_dw_update(
                        self.d["dY_" + name], q, s_x, self.W[name], self.s_w[name], self.m[name],
                        self.v[name], hp, self.sr[name], self.grid, changed_out=ch, ws=ws)
                return
            if self.optimizer == "adafactor":
                ws = self.af_ws[s.index(stream)]
                af = dqt.adafactor(lr=1e-2, step=self.step_no)
                timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_adafactor(
                    self.d["dY_" + name], xdq, self.W[name], self.s_w[name], self.m[name],
                    self.v[name], af, self.sr[name], self.grid, packed=self.packed,
                    changed_out=ch, ws=ws))
            elif self.packed:
                ws = self.dw_ws[s.index(stream)]
                timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_packed(
                    self.d["dY_" + name], xdq, self.W[name], self.s_w[name], self.m[name],
                    self.v[name], hp, self.sr[name], changed_out=ch, ws=ws))
            else:
                ws = self.dw_ws[s.index(stream)]
                timed(self.dw_kind, stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img(
                    self.d["dY_" + name], xdq, self.W[name], self.s_w[name], self.m[name],
                    self.v[name], hp, self.sr[name], self.grid, changed_out=ch, ws=ws,
                    W_img_next=self.W_img_next[name] if self.nimg else None,
                    W8_next=self.W8_next[name] if self.nimg and self.fp8 else None))

        for st in s:
            after(st, main)
        if self.nimg:  # this step's images were written by the last step's updates
            codes = lambda name, stream: None  # noqa: E731
        # forward: the three weight images convert while X is quantised (one
        # pass writes both the forward's code image and the dequantised image
        # the weight gradient reads: splitting it into two passes, the second
        # beside the forward GEMMs, was measured slower)
        aq("X", s[0])
        if self.stack:
            codes("gate_up", s[1])
            codes("down", s[3])
            after(s[1], s[0])
            fwd("gate_up", s[1])
        else:
            if not self.i8:
                codes("gate", s[1])
                codes("up", s[2])
                codes("down", s[3])
            after(s[1], s[0])
            after(s[2], s[0])
            fwd("gate", s[1])
            fwd("up", s[2])
        after(s[0], s[1])
        after(s[2], s[0], s[1], s[3])
        aq("H", s[2])
        fwd("down", s[2])
        # backward: down projection (dX and dW independent)
        after(s[3], s[2])
        dx("down", s[2])
        if not self.group:  # (grouped: with the gate and up update below)
            dw(2, "down", s[3])
        # backward: gate and up, after the down projection's dX
        dx_down = torch.cuda.Event()
        dx_down.record(s[2])
        for st in (s[0], s[1], s[3]):
            if st is not s[2]:
                st.wait_event(dx_down)
        # each weight-gradient GEMM is enqueued ahead of its dX: the longer
        # kernel then takes the SMs first and the dX kernels fill its last wave
        if self.group:
            dw_group(s[1])
            dx("gate", s[0])
            dx("up", s[2])
        elif self.stack:
            dw(0, "gate_up", s[1])
            dx("gate", s[0])
            dx("up", s[2])
        else:
            dw(0, "gate", s[1])
            dx("gate", s[0])
            dw(1, "up", s[3])
            dx("up", s[2])
        for st in s:
            after(main, st)
        if self.nimg:  # the images the updates wrote serve the next step
            self.W_img, self.W_img_next = self.W_img_next, self.W_img
            if self.stack:
                self.W_img_gu, self.W_img_gu_next = self.W_img_gu_next, self.W_img_gu
            if self.fp8:
                self.W8, self.W8_next = self.W8_next, self.W8
                if self.stack:
                    self.W8_gu, self.W8_gu_next = self.W8_gu_next, self.W8_gu

    # algorithmic work per launch, per kernel kind
    def work(self):
        T = T_TOK
        flops = {"fwd": [2.0 * T * K * N for _, K, N in PROJ]}
        flops["bwd_dx"] = list(flops["fwd"])
        flops["bwd_dw_update"] = list(flops["fwd"])
        if self.stack:  # gate and up in one forward and one dW call
            flops["fwd"] = [2.0 * T * HID * 2 * INTER, 2.0 * T * INTER * HID]
            flops["bwd_dw_update"] = list(flops["fwd"])
        if self.group:  # and both dW problems in one launch
            flops["bwd_dw_update"] = [sum(flops["fwd"])]
        flops["bwd_dw_adafactor"] = list(flops["fwd"])
        flops["bwd_dw"] = list(flops["fwd"])  # gradient only (data-parallel exchange)
        flops["fwd_fp8"] = list(flops["fwd"])
        # Algorithmic bytes of the method (the a1 quantiser: 2 B read + 1 B
        # written per element + 4 B per row) and, apart, the bytes of the
        # operand images the method does not have (the tensor cores' exact
        # 16-bit copies of integer codes)
        byts = {
            "act_quant": [T * HID * 3.0 + 4 * T, T * INTER * 3.0 + 4 * T],
            # bf16 in (2) + E4M3 byte (1) per element, + s_x8
            "act_quant_fp8": [T * HID * 3.0 + 4 * T, T * INTER * 3.0 + 4 * T],
            "codes_to_bf16": [0.0],
            "codes_to_fp8": [0.0 for _ in PROJ],
            "codes_to_xdq": [0.0 for _ in PROJ],
        }
        overhead = {
            # the bf16 code image and the bf16 dequantised image (2 + 2 B per element)
            "act_quant": [0.0, 0.0] if self.i8 else [T * HID * 4.0, T * INTER * 4.0],
            # the bf16 dequantised image (2 B per element)
            "act_quant_fp8": [T * HID * 2.0, T * INTER * 2.0],
            # per step: the weight images (with int8 operands, each weight twice:
            # forward and dX), and with int8 operands each forward's activation image
            "codes_to_bf16": ([3.0 * K * N for _, K, N in PROJ] * 2 +
                              [3.0 * T * K for _, K, N in PROJ]) if self.i8 else
                             [3.0 * HID * 2 * INTER, 3.0 * INTER * HID] if self.stack else
                             [(2.25 if self.packed else 3.0) * K * N for _, K, N in PROJ],
            "codes_to_fp8": [2.0 * HID * 2 * INTER, 2.0 * INTER * HID] if self.stack else
                            [(1.25 if self.packed else 2.0) * K * N for _, K, N in PROJ],
            # int8 codes read, bf16 image written, s_x read (gate, up: X; down: H)
            "codes_to_xdq": [3.0 * T * K + 4 * T for _, K, N in PROJ],
        }
        return flops, byts, overhead


def int8_api_step(dev, args, bits):
    """The same MLP step through the C ABI calls on int8 codes (each GEMM
    call makes the bf16 images it needs in its workspace): the step time in
    the same four-stream DAG, and the serial time of its image conversions."""
    st = MLPStep(dev, bits=bits, operands="int8")
    for _ in range(args.warmup):
        st.run()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.steps):
        st.run()
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    timers = {k: [] for k in st.kinds}
    for _ in range(args.steps):
        st.run(timers, serial=True)
    torch.cuda.synchronize()
    st.dqt.dqt_check_device_status()
    per = {k: sum(_elapsed(timers[k])) / args.steps for k in st.kinds}
    peaks, _ = _peaks()
    aq_bytes = (T_TOK * HID * 3.0 + 4 * T_TOK) + (T_TOK * INTER * 3.0 + 4 * T_TOK)
    return {"value": round(T_TOK / (ms / 1e3), 1), "unit": "tokens/s",
            "ms_per_step": round(ms, 4),
            "operands": "int8 codes through the C ABI (dqt_act_quant, dqt_bitlinear_fwd, "
                        "dqt_bitlinear_bwd_dx, dqt_bitlinear_bwd_dw_update)",
            "conversion_ms_per_step_serial": round(per["codes_to_bf16"] + per["codes_to_xdq"], 4),
            "act_quant_frac_of_hbm": round(aq_bytes / (per["act_quant"] / 1e3) / 1e9 /
                                           peaks["hbm_gbs"], 4),
            "kernel_ms_per_step_serial": {k: round(v, 4) for k, v in per.items()}}


def _elapsed(pairs):
    return [a.elapsed_time(b) for a, b in pairs]


def max_over_ranks(x, device):
    """Max of a per-rank float over all ranks (identity when not distributed)."""
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_tokens_per_s(world_size, tokens_per_step, steps, max_ms):
    """Whole-job throughput: every rank processed its own tokens in max_ms."""
    return world_size * tokens_per_step * steps / (max_ms / 1e3)


def _free_port():
    import socket
    with socket.socket() as so:
        so.bind(("127.0.0.1", 0))
        return so.getsockname()[1]


def run_gpu(args):
    ws, rank, local = _dist()
    # several ranks: the data-parallel exchange (default) or independent
    # replicas; --dp exchange on one GPU runs the exchange over a one-rank group
    dp_mode = args.dp if args.dp != "auto" else ("exchange" if ws > 1 else "none")
    import torch.distributed as dist
    if ws > 1 or dp_mode == "exchange":
        torch.cuda.set_device(local)
        if "MASTER_ADDR" in os.environ:
            dist.init_process_group("nccl")
        else:
            dist.init_process_group("nccl", init_method="tcp://127.0.0.1:%d" % _free_port(),
                                    rank=0, world_size=1)
    dev = torch.device("cuda", local if ws > 1 else 0)
    torch.cuda.set_device(dev)
    from paper_2412_04787_gb300 import build as dqt_build
    dqt_build.build()
    st = MLPStep(dev, fp8=args.act == "fp8", optimizer=args.optimizer, packed=args.packed,
                 bits=args.bits, operands=args.operands, tail_slices=not args.no_tail_slices,
                 stack_gate_up=stacked_gate_up(args, dp_mode),
                 next_image=not args.convert_images, dw_group=args.dw_group == "on")
    if dp_mode == "exchange":
        st.enable_dp()
    dqt = st.dqt
    stream = torch.cuda.current_stream()

    def barrier():
        if dist.is_initialized():
            dist.barrier()
        torch.cuda.synchronize()

    # the clock sampler (one nvidia-smi sample per 20 ms) covers the warm-up,
    # the timed steps, the per-kernel region and the e2e steps: the timed
    # region alone lasts only ~20-30 ms
    clk = ClockSampler(dev.index, "the warm-up, the timed steps, the per-kernel region and "
                                  "the e2e steps").__enter__()
    for _ in range(args.warmup):
        st.run()
    dqt.dqt_check_device_status()

    # ---- device-timed region: inputs resident in HBM ----
    barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(args.steps):
        st.run()
    t1.record(stream)
    barrier()
    dqt.dqt_check_device_status()
    ms = max_over_ranks(t0.elapsed_time(t1), dev)
    ms_step = ms / args.steps
    value = aggregate_tokens_per_s(ws, T_TOK, args.steps, ms)

    # ---- per-kernel timing: a second timed region of K steps with the same
    # launches serialised on one stream, CUDA events around every launch ----
    kinds = st.kinds
    timers = {k: [] for k in kinds}
    barrier()
    s0 = torch.cuda.Event(enable_timing=True)
    s1 = torch.cuda.Event(enable_timing=True)
    s0.record(stream)
    for _ in range(args.steps):
        st.run(timers, serial=True)
    s1.record(stream)
    barrier()
    dqt.dqt_check_device_status()
    serial_ms_step = s0.elapsed_time(s1) / args.steps

    # per-kernel live timings
    flops, byts, overhead = st.work()
    per = {}
    for k in kinds:
        ts = _elapsed(timers[k])
        per[k] = {"launches": len(ts), "total_ms": sum(ts), "avg_ms": sum(ts) / max(1, len(ts))}
    tot = sum(p["total_ms"] for p in per.values())
    for k in kinds:
        per[k]["share"] = per[k]["total_ms"] / tot if tot else None
    peaks, pk_kind = _peaks()
    # The per-kernel region lasts K serial steps (well under a second at the
    # default K): its kernels run at the burst clock, so the burst peak (a
    # cuBLAS GEMM timed alone) is the denominator; a region of a second or
    # more is measured against the sustained (power-capped) peak.
    serial_ms_total = serial_ms_step * args.steps
    burst = serial_ms_total < 1000.0
    peak = peaks["bf16_tflops"] if burst else peaks.get("bf16_tflops_sustained", peaks["bf16_tflops"])
    which = "burst" if burst else "sustained"
    dom = max([k for k in kinds if k in flops], key=lambda k: per[k]["total_ms"])
    dom_flops = sum(flops[dom]) * args.steps
    achieved = dom_flops / (per[dom]["total_ms"] / 1e3) / 1e12
    # E4M3 dense tensor rate: the measured bf16 rate times the nominal ratio 4.5 / 2.25
    peak8 = 2.0 * peak
    dom_peak = peak8 if dom == "fwd_fp8" else peak
    roofline = {"bound": "tensor", "kernel": dom, "achieved": round(achieved, 1),
                "peak": dom_peak, "unit": "TFLOP/s", "frac": round(achieved / dom_peak, 4),
                "peak_kind": ("e4m3 dense %s = 2 x measured bf16 %s (nominal ratio)" % (which, which)
                              if dom == "fwd_fp8" else
                              "bf16 dense %s, %s (the per-kernel region lasted %.1f ms)"
                              % (which, pk_kind, serial_ms_total)),
                "timing": "mean CUDA-event duration of its launches over a second timed region "
                          "of the same K steps run serially on one stream (%.4f ms/step)" % serial_ms_step,
                "traffic": ((DW_TRAFFIC_GROUP if st.group else
                             DW_TRAFFIC_STACKED if st.stack else DW_TRAFFIC_BYTES)
                            .get(kernel_fingerprint())
                            # (the FP8 step's update also writes E4M3 images:
                            # not the captured traffic)
                            if dom == "bwd_dw_update" and not st.packed and not st.fp8 else None),
                "kernel_fingerprint": kernel_fingerprint(),
                "algorithmic_per_launch": ("sum of 2*T*K*N FLOP over both problems of the one "
                                           "grouped launch (T=8192; gate and up stacked: K,N = "
                                           "2048,11264; down: 5632,2048)" if st.group else
                                           "2*T*K*N FLOP (T=8192; gate and up stacked: K,N = "
                                           "2048,11264; down: 5632,2048)" if st.stack else
                                           "2*T*K*N FLOP (T=8192; K,N = 2048,5632 / 5632,2048)")}
    kern = {}
    for k in kinds:
        d = dict(per[k])
        sec = per[k]["total_ms"] / 1e3
        if sec <= 0.0:
            pass  # no launch of this kind in the step
        elif k == "dp_exchange":
            pass  # reduce-scatter + shard update + all-gather: time only
        elif k in flops:
            d["tflops"] = sum(flops[k]) * args.steps / sec / 1e12
            if k == "fwd_fp8":
                d["frac_of_e4m3_" + which] = d["tflops"] / peak8
            else:
                d["frac_of_bf16_" + which] = d["tflops"] / peak
        else:
            alg = sum(byts[k]) * args.steps
            ovh = sum(overhead.get(k, [0.0])) * args.steps
            # frac_of_hbm on the method's own bytes; the operand images'
            # bytes (overhead) are reported apart
            d["algorithmic_bytes_per_launch"] = alg / max(1, len(timers[k]))
            d["overhead_bytes_per_launch"] = ovh / max(1, len(timers[k]))
            if alg > 0:
                d["gbs"] = alg / sec / 1e9
                d["frac_of_hbm"] = d["gbs"] / peaks["hbm_gbs"]
            d["moved_gbs"] = (alg + ovh) / sec / 1e9
            d["moved_frac_of_hbm"] = d["moved_gbs"] / peaks["hbm_gbs"]
        kern[k] = {kk: (round(vv, 4) if isinstance(vv, float) else vv) for kk, vv in d.items()}

    # ---- e2e: host buffers, H2D inputs + D2H result inside the timed region ----
    # Every step's activations and gradients are copied from pinned host
    # memory; the copy of step i+1 runs on a copy stream into the second of
    # two device buffer sets while step i computes (double buffering), and
    # each step's changed-code counts are read back to pinned host memory.
    pinned_sets = [{k: v.pin_memory() for k, v in h.items()} for h in st.host_sets]
    pinned = pinned_sets[0]
    res_host = torch.empty((2, 3), dtype=torch.int64).pin_memory()
    h2d = sum(v.numel() * v.element_size() for v in pinned.values())
    d2h = res_host[0].numel() * res_host.element_size()
    st.alternate = False  # here the inputs arrive from the host each step
    bufs = [st.dev_sets[0], st.dev_sets[1]]
    # the copies are split into 32 MiB pieces spread over several copy
    # streams so that more than one DMA engine drives the host link
    n_copy = 4
    copy_streams = [torch.cuda.Stream(device=dev) for _ in range(n_copy)]
    piece = 32 << 20
    jobs = []
    for k, v in pinned.items():
        flat = v.view(-1).view(torch.uint8)
        for off in range(0, flat.numel(), piece):
            jobs.append((k, off, min(piece, flat.numel() - off)))
    e_steps = max(2, min(args.steps, 50))
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)

    def h2d_copy(i, after=None):
        evs = []
        for j, cs in enumerate(copy_streams):
            if after is not None:
                cs.wait_event(after)
            with torch.cuda.stream(cs):
                src_set = pinned_sets[i % 2]
                for k, off, n in jobs[j::n_copy]:
                    dst = bufs[i % 2][k].view(-1).view(torch.uint8)[off:off + n]
                    dst.copy_(src_set[k].view(-1).view(torch.uint8)[off:off + n], non_blocking=True)
                ev = torch.cuda.Event()
                ev.record(cs)
                evs.append(ev)
        return evs

    ready = h2d_copy(0)
    for i in range(e_steps):
        for ev in ready:
            stream.wait_event(ev)
        st.d = bufs[i % 2]
        if i + 1 < e_steps:
            # the next copy may overwrite buffer (i+1)%2 only after step i-1 used it
            done = torch.cuda.Event()
            done.record(stream)
            ready = h2d_copy(i + 1, after=done)
        st.changed.zero_()
        st.run()
        res_host[i % 2].copy_(st.changed, non_blocking=True)
    e1.record(stream)
    barrier()
    st.d = bufs[0]
    st.alternate = True
    clk.__exit__(None, None, None)
    e_ms = max_over_ranks(e0.elapsed_time(e1), dev)
    dqt.dqt_check_device_status()
    e2e = {"value": round(aggregate_tokens_per_s(ws, T_TOK, e_steps, e_ms), 1), "unit": "tokens/s",
           "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": e_steps}

    # the other configurations' sub-results, on rank 0 at N = 1: the
    # single-layer step (256 x 512 x 512) and the standalone update's
    # bandwidth sweep of the 8-bit configuration
    extra = {}
    if (rank == 0 and ws == 1 and not args.no_extras and dp_mode != "exchange" and not st.i8
            and not st.fp8 and not st.packed and st.optimizer == "adamw"):
        extra["int8_c_abi_step"] = int8_api_step(dev, args, st.bits)
    if rank == 0 and ws == 1 and not args.no_extras and dp_mode != "exchange" and not st.fp8:
        lay = layer_step(1.58, 200, 10)
        extra["layer_256x512x512"] = {k: lay[k] for k in (
            "value", "unit", "us_per_step", "graph", "e2e", "changed_codes_last_step", "clocks")}
        extra["sr_update_sweep"] = sr_sweep()

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args.cpu_seconds)

    if rank == 0:
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "e4m3 forward, bf16 backward" if st.fp8 else "bf16",
            "data": "synthetic (seeded N(0,1) activations, N(0,1e-2) gradients, AbsMean-%s codes of N(0,0.02))"
                    % ("ternary" if st.bits == 1.58 else "%d-bit" % st.bits),
            "config": mlp_config(bits=st.bits, fp8=st.fp8, optimizer=st.optimizer,
                                 packed=st.packed, i8=st.i8,
                                 parallelism=_parallelism(ws, dp_mode), stacked=st.stack),
            "roofline": roofline, "kernels": kern, "e2e": e2e,
            "gpu_launches": st.launches_per_step * args.steps,
            "clocks": clk.summary(), "cpu_baseline": cpu,
            "changed_codes_last_step": changed_by_projection(
                [int(x) for x in res_host[(e_steps - 1) % 2].tolist()], st.stack),
        }
        line.update(extra)
        print(json.dumps(line))
    if dist.is_initialized():
        dist.destroy_process_group()


# ---------------------------------------------------------------------------
# CPU oracle timing (the reported baseline and the --impl reference arm)
# ---------------------------------------------------------------------------
_SAMPLE_INPUTS = {}  # per process: the generated inputs of each (seed, projection)


def _sample_inputs(seed, i, K, N):
    import oracle
    from paper_2412_04787_gb300 import inputs
    key = (seed, i)
    if key not in _SAMPLE_INPUTS:
        qmin, qmax = oracle.grid(1.58)
        X = inputs.bf16_bits(inputs.normal((T_TOK, K), 1.0, seed=seed + i, dtype=torch.bfloat16))
        dY = inputs.bf16_bits(inputs.normal((T_TOK, N), 1e-2, seed=seed + 10 + i,
                                            dtype=torch.bfloat16))
        c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=seed + 20 + i).numpy(),
                                        qmin, qmax)
        _SAMPLE_INPUTS[key] = (X, dY, c, s_w)
    return _SAMPLE_INPUTS[key]


def _oracle_sample(token_rows, weight_rows, seed=7):
    """Times the oracle, per projection, on the act-quant of all tokens (the
    weight gradient needs every token's code), the forward and dX of
    `token_rows` token rows, and dW + AdamW + SR of `weight_rows` weight rows;
    returns (seconds measured, seconds extrapolated to the full step: the
    row parts scaled by T / token_rows and N / weight_rows)."""
    import oracle

    qmin, qmax = oracle.grid(1.58)
    meas = 0.0
    full = 0.0
    for i, (name, K, N) in enumerate(PROJ):
        X, dY, c, s_w = _sample_inputs(seed, i, K, N)
        t0 = time.perf_counter()
        qa, sa, _, _ = oracle.act_quant(X)
        t1 = time.perf_counter()
        oracle.fwd(qa[:token_rows], sa[:token_rows], c, s_w)
        oracle.bwd_dx(dY[:token_rows], c, s_w)
        t2 = time.perf_counter()
        rows = np.arange(weight_rows)
        g = oracle.bwd_dw(dY, qa, sa, rows=rows).astype(np.float32)
        k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, s_w)
        z = np.zeros((weight_rows, K), np.float32)
        oracle.update(g, c[:weight_rows], z, z, k, qmin, qmax, 1234, 1, i, rows=rows)
        t3 = time.perf_counter()
        meas += t3 - t0
        full += (t1 - t0) + (t2 - t1) * T_TOK / token_rows + (t3 - t2) * N / weight_rows
    return meas, full


def _oracle_layer_full():
    """The single-layer configuration (T=256, K=512, N=512, ternary, AdamW
    step 1) through the oracle in full: act-quant, forward, dX, dW and the
    update.  Returns the seconds it took."""
    import oracle
    from paper_2412_04787_gb300 import inputs

    T, K, N = LAYER_SHAPE
    qmin, qmax = oracle.grid(1.58)
    X = inputs.bf16_bits(inputs.normal((T, K), 1.0, seed=1, dtype=torch.bfloat16))
    dY = inputs.bf16_bits(inputs.normal((T, N), 1e-2, seed=2, dtype=torch.bfloat16))
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=3).numpy(), qmin, qmax)
    t0 = time.perf_counter()
    q, s, _, _ = oracle.act_quant(X)
    oracle.fwd(q, s, c, s_w)
    oracle.bwd_dx(dY, c, s_w)
    g = oracle.bwd_dw(dY, q, s).astype(np.float32)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, s_w)
    z = np.zeros((N, K), np.float32)
    oracle.update(g, c, z, z, k, qmin, qmax, 1234, 1, 0)
    return time.perf_counter() - t0


def _oracle_sample_worker(job):
    """One host core's share of the sampled MLP step (spawned process)."""
    tr, wr, seed = job
    from oracle import build_oracle
    build_oracle.build()
    return _oracle_sample(tr, wr, seed=seed)


class OraclePool:
    """The oracle on every host core: `cores` spawned processes (never forked
    from a process that has touched the GPU), each timing the same bounded
    sample of the MLP step at once, so that memory contention between cores is
    in every measurement.  A step of the full workload on `cores` cores then
    takes mean(extrapolated single-core step) / cores."""

    def __init__(self, cores=None):
        import concurrent.futures
        import multiprocessing
        self.cores = cores or os.cpu_count() or 1
        self.ex = concurrent.futures.ProcessPoolExecutor(
            max_workers=self.cores, mp_context=multiprocessing.get_context("spawn"))
        # start every worker, build the oracle there and generate its inputs
        list(self.ex.map(_oracle_sample_worker, [(2, 1, 7 + i) for i in range(self.cores)]))

    def sample(self, tr, wr):
        """Returns (wall seconds of the sample on all cores, extrapolated
        seconds of one full step on all cores)."""
        t0 = time.perf_counter()
        res = list(self.ex.map(_oracle_sample_worker, [(tr, wr, 7 + i) for i in range(self.cores)]))
        wall = time.perf_counter() - t0
        full_1core = statistics.mean(f for _, f in res)
        return wall, full_1core / self.cores

    def close(self):
        self.ex.shutdown()


def _sample_size(seconds):
    m0, _ = _oracle_sample(2, 1)
    scale = max(1.0, seconds / max(m0, 1e-3))
    return int(min(256, max(2, 2 * scale))), int(min(128, max(1, scale)))


def cpu_baseline(seconds=15.0):
    """The oracle as it stands on the GPU machine's host: the single-layer
    configuration in full on one core, and a bounded sample of the MLP step
    on every core, extrapolated to the full step."""
    t1 = _oracle_layer_full()
    tr, wr = _sample_size(seconds)
    pool = OraclePool()
    try:
        wall, full = pool.sample(tr, wr)
    finally:
        pool.close()
    frac = wall / full  # the share of the full step's work the cores did in `wall`
    return {"value": round(T_TOK / full, 3), "unit": "tokens/s", "cores": pool.cores,
            "nproc": os.cpu_count(), "kind": "oracle",
            "sample": "%d processes at once, each %d token rows of act-quant+fwd+dX and %d weight "
                      "rows of dW+AdamW+SR per projection (plus the full act-quant dW needs), "
                      "%.1f s wall: %.4f of the 8192-token step's work; extrapolated step "
                      "%.1f s on %d cores" % (pool.cores, tr, wr, wall, frac, full, pool.cores),
            "layer_256x512x512": {"value": round(LAYER_SHAPE[0] / t1, 2), "unit": "tokens/s",
                                  "cores": 1, "seconds": round(t1, 3),
                                  "sample": "the whole single-layer step, not sampled"}}


def stacked_gate_up(args, dp_mode="replicas"):
    """Whether the MLP step runs gate and up as two stacked weights (one
    forward call, one dW + update call; MLPStep's condition; the data-parallel
    exchange keeps one weight per exchange)."""
    return (not args.separate_gate_up and args.operands == "img"
            and not args.packed and args.optimizer == "adamw" and dp_mode != "exchange")


def changed_by_projection(counts, stacked):
    """Codes the last e2e step changed, per weight-gradient call: with gate and
    up stacked their one call counts both (slot 1 is then unused)."""
    if stacked:
        return {"gate+up": counts[0], "down": counts[2]}
    return dict(zip(("gate", "up", "down"), counts))


def mlp_config(bits=1.58, fp8=False, optimizer="adamw", packed=False, i8=True, parallelism=None,
               stacked=False):
    """The `config` of the MLP step's JSON line (both arms)."""
    wname = "ternary" if bits == 1.58 else "%d-bit" % bits
    return {"workload": (WORKLOAD if bits == 1.58 else WORKLOAD.replace("ternary", wname)) +
                        (", FP8 (E4M3) forward" if fp8 else "") +
                        (", Adafactor" if optimizer == "adafactor" else "") +
                        (", 2-bit packed codes" if packed else ""),
            "tokens": T_TOK, "hidden": HID, "intermediate": INTER,
            "weights": "%s codes, %s" % (wname, "2-bit packed" if packed else "int8"),
            "optimizer": optimizer,
            "operands": "int8 codes through the C ABI" if i8 else "bf16 / E4M3 operand images",
            "parallelism": parallelism or "single GPU",
            "gate_up": ("two weights stacked in one forward call and one dW + update call, each "
                        "with its own scale and SR stream; dX per weight" if stacked else
                        "separate calls"),
            "l2": "inputs larger than L2 (step working set ~1.5 GB > 129 MB)"}


def _parallelism(ws, dp_mode):
    if dp_mode == "exchange":
        return ("data parallel over %d GPU(s): reduce-scatter of fp32 dW, ZeRO-1 sharded "
                "AdamW + SR update, all-gather of int8 codes" % ws)
    return "replicas" if ws > 1 else "single GPU"


def run_reference(args):
    """The oracle as it stands on the host cores: each step is one bounded
    sample of the MLP step run on every core at once (OraclePool); the step's
    time is that sample's wall time and `value` the throughput it implies."""
    ws, rank, _ = _dist()
    if rank != 0:
        return
    from oracle import build_oracle
    build_oracle.build()
    per_step_s = max(5.0, min(30.0, 150.0 / max(1, args.steps + args.warmup)))
    tr, wr = _sample_size(per_step_s)
    pool = OraclePool()
    try:
        for _ in range(args.warmup):
            pool.sample(2, 1)
        walls, fulls = [], []
        for _ in range(args.steps):
            wall, full = pool.sample(tr, wr)
            walls.append(wall)
            fulls.append(full)
    finally:
        pool.close()
    full = statistics.median(fulls)
    wall = statistics.median(walls)
    value = T_TOK / full
    dp_mode = args.dp if args.dp != "auto" else ("exchange" if ws > 1 else "none")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "tokens/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(wall * 1e3, 1), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64/f32 (oracle)", "data": "synthetic",
        "config": mlp_config(bits=args.bits, fp8=args.act == "fp8", optimizer=args.optimizer,
                             packed=args.packed, i8=args.operands == "int8",
                             parallelism=_parallelism(ws, dp_mode),
                             stacked=stacked_gate_up(args, dp_mode)),
        "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": pool.cores,
                         "nproc": os.cpu_count(), "kind": "oracle",
                         "sample": "each step: %d processes at once, each %d token rows of "
                                   "act-quant+fwd+dX and %d weight rows of dW+AdamW+SR per "
                                   "projection (plus the full act-quant dW needs): %.4f of the "
                                   "8192-token step's work in %.1f s" % (
                                       pool.cores, tr, wr, wall / full, wall)},
        "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


def sr_sweep(sizes=(1 << 24, 1 << 26, 1 << 28), reps=10):
    """The 8-bit standalone AdamW + SR update (22 bytes per weight: g 4, c
    1 + 1, m 4 + 4, v 4 + 4) at each size: median CUDA-event time of `reps`
    launches, each after an L2 flush (256 MiB written, then 256 MiB read)."""
    from paper_2412_04787_gb300 import dqt
    dev = torch.device("cuda", torch.cuda.current_device())
    peaks, kind = _peaks()
    g8 = dqt.grid(8)
    hp = dqt.adamw(step=3)
    sr = dqt.sr_stream()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(32 << 20, dtype=torch.int64, device=dev)
    out = []
    for n in sizes:
        gen = torch.Generator(device=dev).manual_seed(n)
        grad = torch.randn(n, device=dev, generator=gen) * 1e-3
        W = torch.randint(-128, 128, (n,), dtype=torch.int8, device=dev, generator=gen)
        m = torch.randn(n, device=dev, generator=gen) * 1e-4
        v = (torch.randn(n, device=dev, generator=gen) * 1e-4).square()
        for _ in range(3):
            dqt.dqt_sr_update(grad, W, 7958.0, m, v, hp, sr, g8)
        times = []
        for _ in range(reps):
            flush.zero_()
            flush_r.sum()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record()
            dqt.dqt_sr_update(grad, W, 7958.0, m, v, hp, sr, g8)
            b.record()
            times.append((a, b))
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in times)
        gbs = 22.0 * n / (ms / 1e3) / 1e9
        out.append({"numel": n, "median_ms": round(ms, 4), "gbs": round(gbs, 1),
                    "frac_of_hbm": round(gbs / peaks["hbm_gbs"], 4)})
        del grad, W, m, v
    dqt.dqt_check_device_status()
    return {"kernel": "sr_update (8-bit grid, fp32 gradient in memory)", "points": out,
            "peak_gbs": peaks["hbm_gbs"], "peak_kind": "copy bandwidth, %s" % kind,
            "bytes_per_weight": 22, "l2": "flushed before every launch"}


def run_kernel(args):
    """One kernel kind alone, repeated: for ncu captures and bandwidth sweeps.
    GEMMs and act_quant run at the gate projection's shape (T=8192, K=2048,
    N=5632); sr_update streams --numel weights (fp32 gradient)."""
    from paper_2412_04787_gb300 import build as dqt_build, dqt, inputs
    dqt_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    T, K, N = T_TOK, HID, INTER
    if args.shape:
        T, K, N = (int(x) for x in args.shape.split(","))
    g = dqt.grid(args.bits)
    k = args.kernel
    if k in ("sr_update", "sr_update_packed"):
        n = args.numel
        grad = torch.randn(n, device=dev) * 1e-3
        W = torch.randint(-1, 2, (n,), dtype=torch.int8, device=dev)
        m = torch.zeros(n, device=dev)
        v = torch.zeros(n, device=dev)
        hp = dqt.adamw()
        sr = dqt.sr_stream()
        if k == "sr_update":
            fn = lambda: dqt.dqt_sr_update(grad, W, 62.0, m, v, hp, sr, g)  # noqa: E731
            work, unit = 22.0 * n, "GB/s"
        else:
            Wp = dqt.dqt_pack_ternary(W)
            fn = lambda: dqt.dqt_sr_update_packed(grad, Wp, 62.0, m, v, hp, sr)  # noqa: E731
            work, unit = 20.5 * n, "GB/s"
    else:
        X = inputs.normal((T, K), 1.0, seed=1, dtype=torch.bfloat16).to(dev)
        dY = inputs.normal((T, N), 1e-2, seed=2, dtype=torch.bfloat16).to(dev)
        W, s_w = dqt.dqt_absmean_init(inputs.normal((N, K), 0.02, seed=3).to(dev), g)
        _, s_x, q_img, xdq = dqt.dqt_act_quant_images(X, want=("Xq_img", "Xdq"))
        W_img = dqt.dqt_codes_to_bf16(W)
        m = torch.zeros((N, K), device=dev)
        v = torch.zeros((N, K), device=dev)
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=dev)
        dX = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
        hp = dqt.adamw()
        sr = dqt.sr_stream()
        nbt = max(dqt.dqt_fwd_img_workspace_size(T, K, N), dqt.dqt_bwd_dx_img_workspace_size(T, N, K))
        tws = torch.empty(nbt, dtype=torch.uint8, device=dev) if nbt else False
        if args.no_tail_slices:
            tws = False
        if k == "fwd":
            fn = lambda: dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, s_w, g, Y=Y, ws=tws)  # noqa: E731
        elif k == "bwd_dx":
            fn = lambda: dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, s_w, dX=dX, ws=tws)  # noqa: E731
        elif k == "bwd_dw_update":
            fn = lambda: dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, W, s_w, m, v, hp, sr, g)  # noqa: E731
        elif k == "bwd_dw":  # gradient only (fp32 dW written, no update)
            dW = torch.empty((N, K), dtype=torch.float32, device=dev)
            fn = lambda: dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, None, s_w, None, None, None,  # noqa: E731
                                                             None, g, dW_out=dW)
        elif k == "bwd_dw_unfused":  # gradient to memory, then the standalone update
            dW = torch.empty((N, K), dtype=torch.float32, device=dev)

            def fn():
                dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, None, s_w, None, None, None, None, g,
                                                    dW_out=dW)
                dqt.dqt_sr_update(dW.view(-1), W.view(-1), s_w, m.view(-1), v.view(-1), hp, sr, g)
        elif k == "act_quant":
            fn = lambda: dqt.dqt_act_quant_images(X, None, s_x, q_img, xdq, want=())  # noqa: E731
        elif k == "act_quant_codes":  # the int8 call: codes and scales only
            Xq = torch.empty((T, K), dtype=torch.int8, device=dev)
            fn = lambda: dqt.dqt_act_quant(X, Xq, s_x)  # noqa: E731
        elif k == "codes_to_xdq":
            Xq, _ = dqt.dqt_act_quant(X)
            fn = lambda: dqt.dqt_codes_to_xdq(Xq, s_x, xdq)  # noqa: E731
        elif k == "bwd_dw_update_packed":
            Wp = dqt.dqt_pack_ternary(W)
            fn = lambda: dqt.dqt_bitlinear_bwd_dw_update_packed(dY, xdq, Wp, s_w, m, v, hp, sr)  # noqa: E731
        elif k in ("bwd_dw_adafactor", "adafactor_stats", "adafactor_apply"):
            R = torch.zeros(N, device=dev)
            Cc = torch.zeros(K, device=dev)
            af = dqt.adafactor(lr=1e-2)
            G = torch.randn((N, K), device=dev) * 1e-3
            fa, fb, scal = dqt.dqt_adafactor_stats(G, W, s_w, R, Cc, af)
            if k == "bwd_dw_adafactor":
                ws = torch.empty(dqt.dqt_bwd_dw_adafactor_workspace_size(T, N, K), dtype=torch.uint8,
                                 device=dev)
                fn = lambda: dqt.dqt_bitlinear_bwd_dw_adafactor(dY, xdq, W, s_w, R, Cc, af, sr, g,  # noqa: E731
                                                                ws=ws)
            elif k == "adafactor_stats":
                fn = lambda: dqt.dqt_adafactor_stats(G, W, s_w, R, Cc, af, a_out=fa, b_out=fb,  # noqa: E731
                                                     scalars_out=scal)
            else:
                fn = lambda: dqt.dqt_adafactor_apply(G, W, fa, fb, scal, 1, sr, g)  # noqa: E731
        elif k in ("act_quant_fp8", "fwd_fp8", "codes_to_fp8"):
            q8, s8, _ = dqt.dqt_act_quant_fp8(X)
            W8 = dqt.dqt_codes_to_fp8(W, g)
            if k == "act_quant_fp8":
                fn = lambda: dqt.dqt_act_quant_fp8(X, q8, s8, xdq)  # noqa: E731
            elif k == "codes_to_fp8":
                fn = lambda: dqt.dqt_codes_to_fp8(W, g, W8)  # noqa: E731
            else:
                fn = lambda: dqt.dqt_bitlinear_fwd_fp8(q8, s8, W8, s_w, g, Y=Y)  # noqa: E731
        elif k == "codes_to_bf16":
            fn = lambda: dqt.dqt_codes_to_bf16(W, W_img)  # noqa: E731
        else:
            raise SystemExit("unknown kernel %s" % k)
        if k in ("fwd", "bwd_dx", "bwd_dw_update", "bwd_dw", "bwd_dw_unfused", "fwd_fp8",
                 "bwd_dw_update_packed", "bwd_dw_adafactor"):
            work, unit = 2.0 * T * K * N, "TFLOP/s"
        elif k == "adafactor_stats":
            # two reads of G (4 B each) and one of the codes (1 B) per weight
            work, unit = 9.0 * N * K, "GB/s"
        elif k == "adafactor_apply":
            # G read (4 B), codes read and written (1 + 1 B) per weight
            work, unit = 6.0 * N * K, "GB/s"
        elif k == "act_quant":
            work, unit = 6.0 * T * K + 4 * T, "GB/s"
        elif k in ("act_quant_codes", "codes_to_xdq"):
            work, unit = 3.0 * T * K + 4 * T, "GB/s"
        elif k == "act_quant_fp8":
            work, unit = 5.0 * T * K + 4 * T, "GB/s"
        elif k == "codes_to_fp8":
            work, unit = 2.0 * N * K, "GB/s"
        else:
            work, unit = 3.0 * N * K, "GB/s"
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    # L2 flush between launches: write 256 MiB (> the 129 MB L2), then read
    # another 256 MiB, so that the timed kernel finds L2 full of clean lines
    # (a write-only flush would leave up to 129 MB of dirty lines whose
    # write-back the next kernel would pay for)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    flush_r = torch.ones(32 << 20, dtype=torch.int64, device=dev)
    times = []
    for _ in range(args.steps):
        flush.zero_()
        flush_r.sum()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        fn()
        b.record()
        times.append((a, b))
    torch.cuda.synchronize()
    dqt.dqt_check_device_status()
    ms = [a.elapsed_time(b) for a, b in times]
    med = statistics.median(ms)
    rate = work / (med / 1e3) / (1e12 if unit == "TFLOP/s" else 1e9)
    peaks, kind = _peaks()
    peak = peaks["bf16_tflops"] if unit == "TFLOP/s" else peaks["hbm_gbs"]
    if k == "fwd_fp8":
        peak = 2.0 * peak  # E4M3 dense = bf16 measured x the nominal ratio 4.5 / 2.25
    stream_k = k in ("sr_update", "sr_update_packed")
    print(json.dumps({"kernel": k, "numel": args.numel if stream_k else None,
                      "shape": None if stream_k else [T, K, N],
                      "median_ms": round(med, 5), "min_ms": round(min(ms), 5),
                      "rate": round(rate, 1), "unit": unit, "peak": peak,
                      "frac": round(rate / peak, 4), "peak_kind": "burst, " + kind,
                      "l2": "256 MiB written, then 256 MiB read, between launches (clean L2)"}))


DECODER_SIZES = {
    # the paper's LLaMA-structured model sizes (Sec. 4.1): ~130M and ~1B
    "130m": dict(layers=12, hidden=768, heads=12, ffn=2048, batch=16, seq=1024),
    "1b": dict(layers=22, hidden=2048, heads=32, ffn=5632, batch=8, seq=2048),
}


def run_decoder(args):
    """A LLaMA-structured decoder training step with every transformer linear
    layer a DQT BitLinear (--decoder-size 130m: 12 layers, hidden 768, 12
    heads, FFN 2048, batch 16 x seq 1024; 1b: 22 layers, hidden 2048, 32
    heads, FFN 5632, batch 8 x seq 2048; vocab 32000, ternary; synthetic
    uniform token ids; --act fp8 for the E4M3 forward).  The
    BitLinear layers update themselves during backward; the bf16 embedding,
    norms and head are stepped by torch AdamW inside the timed region.  By
    default the whole step is captured once as a CUDA graph and replayed, the
    per-step DQT constants (step, bias corrections, Philox counter) uploaded
    from pinned memory before each replay; --no-graph runs it eagerly."""
    from paper_2412_04787_gb300 import build as dqt_build
    from paper_2412_04787_gb300.decoder import DecoderConfig, DQTDecoder
    dqt_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    sz = DECODER_SIZES[args.decoder_size]
    B, S = sz["batch"], sz["seq"]
    cfg = DecoderConfig(layers=sz["layers"], hidden=sz["hidden"], heads=sz["heads"], ffn=sz["ffn"],
                        vocab=32000, bits=args.bits,
                        lr=1e-2 if args.optimizer == "adafactor" else 1e-3,
                        seed=1234, act=args.act, optimizer=args.optimizer, packed=args.packed)
    model = DQTDecoder(cfg, device=dev)
    # CUDA-graph replay needs the device-resident AdamW constants (int8 codes)
    graphable = args.optimizer == "adamw" and not args.packed
    use_graph = not args.no_graph and graphable
    if graphable:
        model.enable_graph_updates()
    # the multi-tensor (foreach) AdamW: measured faster than the fused one on
    # these bf16 parameters (embedding and head 32000 x hidden, norm gains)
    opt = torch.optim.AdamW(model.dense_parameters(), lr=1e-3, foreach=True, capturable=use_graph)
    g = torch.Generator().manual_seed(5)
    host_ids = [torch.randint(0, cfg.vocab, (B, S + 1), generator=g).pin_memory() for _ in range(2)]
    ids_dev = [h.to(dev) for h in host_ids]
    static_ids = ids_dev[0].clone()
    state = {"loss": None, "i": 0}

    def fwd_bwd_opt():
        loss = model(static_ids[:, :-1], static_ids[:, 1:])
        loss.backward()
        opt.step()
        return loss

    def run_step(src):
        i = state["i"]
        state["i"] += 1
        static_ids.copy_(src, non_blocking=True)
        if graphable:
            model.prepare_step(i % 2)
            model.upload_update_consts(i % 2)
        if use_graph:
            graph.replay()
            return state["loss"]
        loss = fwd_bwd_opt()
        opt.zero_grad(set_to_none=True)
        return loss

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for i in range(args.warmup):
            static_ids.copy_(ids_dev[i % 2])
            if graphable:
                model.prepare_step(state["i"] % 2)
                model.upload_update_consts(state["i"] % 2)
            state["i"] += 1
            fwd_bwd_opt()
            opt.zero_grad(set_to_none=True)
    torch.cuda.current_stream().wait_stream(side)
    graph = None
    if use_graph:
        graph = torch.cuda.CUDAGraph()
        opt.zero_grad(set_to_none=True)
        with torch.cuda.graph(graph):
            state["loss"] = fwd_bwd_opt()
    stream = torch.cuda.current_stream()
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index) as clk:
        t0.record(stream)
        for i in range(args.steps):
            run_step(ids_dev[i % 2])
        t1.record(stream)
        torch.cuda.synchronize()
    ms = t0.elapsed_time(t1)
    tokens = B * S
    # e2e: ids from pinned host memory each step, the loss read back each step
    loss_host = torch.empty((), dtype=torch.float32).pin_memory()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.steps):
        loss = run_step(host_ids[i % 2])
        loss_host.copy_(loss.detach(), non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e_ms = e0.elapsed_time(e1)
    bl_flops = model.bitlinear_flops_per_step(tokens)
    print(json.dumps({
        "metric": "DQT decoder training step tokens/s", "value": round(tokens * args.steps / (ms / 1e3), 1),
        "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms / args.steps, 3), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None,
        "dtype": "e4m3 BitLinear forward, bf16 elsewhere" if args.act == "fp8" else "bf16",
        "data": "synthetic uniform token ids",
        "config": {"workload": "LLaMA-structured decoder (%s), %s DQT BitLinear in q,k,v,o,gate,up,down%s%s%s"
                               % (args.decoder_size,
                                  "ternary" if args.bits == 1.58 else "%d-bit" % args.bits,
                                  ", FP8 (E4M3) forward" if args.act == "fp8" else "",
                                  ", Adafactor" if args.optimizer == "adafactor" else "",
                                  ", 2-bit packed codes" if args.packed else ""),
                   "layers": cfg.layers, "hidden": cfg.hidden, "heads": cfg.heads, "ffn": cfg.ffn,
                   "vocab": cfg.vocab, "batch": B, "seq": S, "cuda_graph": use_graph},
        "bitlinear_tflop_per_step": round(bl_flops / 1e12, 3),
        "e2e": {"value": round(tokens * args.steps / (e_ms / 1e3), 1), "unit": "tokens/s",
                "h2d_bytes_per_step": int(host_ids[0].numel() * 8), "d2h_bytes_per_step": 4},
        "final_loss": float(loss_host), "clocks": clk.summary()}))


LAYER_SHAPE = (256, 512, 512)  # T, K, N of the single-layer step


def run_layer(args):
    print(json.dumps(layer_step(args.bits, args.steps, args.warmup)))


def layer_step(bits=1.58, steps=200, warmup=10):
    """One BitLinear layer's training step at T=256, K=512, N=512 (X ~N(0,1),
    dY ~N(0,1e-2), ternary codes by AbsMean of N(0,0.02), AdamW lr 1e-3, Philox
    seed 1234): act_quant, forward, then dX and the fused dW + AdamW + SR
    update side by side on two streams (the backward after the forward, as in
    a network, where dY follows from Y); the update writes the weight's code
    image for the next step into the second of two image buffers, so it never
    touches the image dX reads.  At this size every kernel is latency-bound, so the
    K timed steps are captured as one CUDA graph (step i reads its update
    constants from row i of a device block, uploaded in one copy at the start
    of the timed region) and the time is the GPU's, not the Python launch
    path's; the result is quoted in microseconds per step.  e2e: a second
    graph whose every step also copies X and dY from pinned host memory and
    reads the changed-code count back."""
    from paper_2412_04787_gb300 import build as dqt_build
    from paper_2412_04787_gb300 import dqt, inputs
    dqt_build.build()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    T, K, N = LAYER_SHAPE
    KS = steps + steps % 2  # even: each replay starts on the image its predecessor left in imgs[0]
    grid = dqt.grid(bits)
    host = [(inputs.normal((T, K), 1.0, seed=1 + 100 * r, dtype=torch.bfloat16).pin_memory(),
             inputs.normal((T, N), 1e-2, seed=2 + 100 * r, dtype=torch.bfloat16).pin_memory())
            for r in range(2)]
    X = host[0][0].to(dev)
    dY = host[0][1].to(dev)
    W, s_w = dqt.dqt_absmean_init(inputs.normal((N, K), 0.02, seed=3).to(dev), grid)
    m = torch.zeros((N, K), dtype=torch.float32, device=dev)
    v = torch.zeros((N, K), dtype=torch.float32, device=dev)
    s_x = torch.empty(T, dtype=torch.float32, device=dev)
    q_img = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    xdq = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    W_img = torch.empty((N, K), dtype=torch.bfloat16, device=dev)
    Y = torch.empty((T, N), dtype=torch.bfloat16, device=dev)
    dX = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    changed = torch.zeros(1, dtype=torch.int64, device=dev)
    nbw = dqt.dqt_bwd_dw_img_workspace_size(T, N, K)
    ws = torch.empty(nbw, dtype=torch.uint8, device=dev) if nbw else None
    row = (dqt.lib().dqt_update_consts_size() + 63) // 64 * 64
    # the graph of KS steps is replayed R times (about a second of GPU time)
    # in the timed region; every replay's constants have a host block of
    # their own, so no block is rewritten while a copy from it may be pending
    R = max(1, 40000 // KS)
    uc_host = torch.zeros((R, KS, row), dtype=torch.uint8).pin_memory()
    uc_host_e2e = torch.zeros((KS, row), dtype=torch.uint8).pin_memory()
    uc_dev = torch.zeros((KS, row), dtype=torch.uint8, device=dev)
    sr = dqt.sr_stream(seed=1234, tensor_id=0)
    state = {"step": 0}
    ch_host = torch.empty(KS, dtype=torch.int64).pin_memory()

    # two image buffers: step i reads imgs[i % 2], its update writes imgs[(i + 1) % 2]
    imgs = [W_img, torch.empty_like(W_img)]
    dqt.dqt_codes_to_bf16(W, imgs[0])  # the first step's image
    branch = torch.cuda.Stream()

    def kernels(i):
        main = torch.cuda.current_stream()
        img, img_next = imgs[i % 2], imgs[(i + 1) % 2]
        dqt.dqt_act_quant_images(X, None, s_x, q_img, xdq, want=())
        dqt.dqt_bitlinear_fwd_img(q_img, s_x, img, s_w, grid, Y=Y)
        fork = torch.cuda.Event()
        fork.record(main)
        branch.wait_event(fork)
        with torch.cuda.stream(branch):
            dqt.dqt_bitlinear_bwd_dx_img(dY, img, s_w, dX=dX)
        dqt.dqt_bitlinear_bwd_dw_update_dev(dY, xdq, W, m, v, uc_dev[i % KS], changed_out=changed,
                                            ws=ws, W_img_next=img_next)
        join = torch.cuda.Event()
        join.record(branch)
        main.wait_event(join)

    def fill(block):
        for i in range(block.shape[0]):
            state["step"] += 1
            dqt.dqt_update_consts(dqt.adamw(lr=1e-3, step=state["step"]), sr, grid, s_w,
                                  out=block[i])

    # warm-up: eager steps, each with its own constants row; an even number,
    # so that the graph's first step finds its image in imgs[0]
    warmup += warmup % 2
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    warm = torch.zeros((warmup, row), dtype=torch.uint8).pin_memory()
    with torch.cuda.stream(side):
        for i in range(warmup):
            state["step"] += 1
            dqt.dqt_update_consts(dqt.adamw(lr=1e-3, step=state["step"]), sr, grid, s_w,
                                  out=warm[i])
            uc_dev[i % KS].copy_(warm[i], non_blocking=True)
            kernels(i)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        for i in range(KS):
            kernels(i)
    graph_e2e = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph_e2e):
        for i in range(KS):
            X.copy_(host[i % 2][0], non_blocking=True)
            dY.copy_(host[i % 2][1], non_blocking=True)
            kernels(i)
            ch_host[i:i + 1].copy_(changed, non_blocking=True)
    torch.cuda.synchronize()
    dqt.dqt_check_device_status()

    stream = torch.cuda.current_stream()
    for r in range(R):
        fill(uc_host[r])
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with ClockSampler(dev.index) as clk:
        t0.record(stream)
        for r in range(R):
            uc_dev.copy_(uc_host[r], non_blocking=True)
            graph.replay()
        t1.record(stream)
        torch.cuda.synchronize()
    dqt.dqt_check_device_status()
    ms = t0.elapsed_time(t1) / (R * KS)
    fill(uc_host_e2e)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    uc_dev.copy_(uc_host_e2e, non_blocking=True)
    graph_e2e.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    e_ms = e0.elapsed_time(e1) / KS
    return {
        "metric": "DQT BitLinear fwd+bwd+SR-update tokens/s", "value": round(T / (ms / 1e3), 1),
        "unit": "tokens/s", "n_gpus": 1, "steps": R * KS, "warmup": warmup,
        "ms_per_step": round(ms, 5), "us_per_step": round(ms * 1e3, 2),
        "graph": {"steps_per_graph": KS, "replays": R},
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) activations, N(0,1e-2) gradients, AbsMean-ternary codes of N(0,0.02))",
        "config": {"workload": "single BitLinear layer training step, 256 tokens, 512 -> 512, "
                               "ternary codes, AdamW + SR (K steps in one CUDA graph)",
                   "tokens": T, "in_features": K, "out_features": N,
                   "l2": "latency-bound: the whole working set (~2 MB) stays in L2"},
        "roofline": {"bound": "latency", "note": "3 x 0.134 GFLOP and 4.7 MB per step: "
                     "launch and pipeline latency, not a throughput roofline, bounds this size"},
        "gpu_launches": (4 + (1 if nbw else 0)) * KS * R,
        "e2e": {"value": round(T / (e_ms / 1e3), 1), "unit": "tokens/s",
                "h2d_bytes_per_step": int(X.numel() * 2 + dY.numel() * 2 + row),
                "d2h_bytes_per_step": 8},
        "changed_codes_last_step": int(ch_host[KS - 1]),
        "clocks": clk.summary()}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="dqt", choices=["dqt", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--separate-gate-up", action="store_true",
                    help="mlp: gate and up as two separate calls each (by default, with image "
                         "operands and AdamW on int8 codes, they are two stacked weights of one "
                         "forward call and one dW + update call, each weight with its own scale "
                         "and SR stream; dX per weight)")
    ap.add_argument("--dw-group", choices=("on", "off"), default="on",
                    help="MLP step with gate and up stacked: both weight-gradient problems in one "
                         "persistent launch (on) or in two calls (off)")
    ap.add_argument("--convert-images", action="store_true",
                    help="mlp, image operands: convert the codes to bf16 images at the start of "
                         "every step instead of taking the images the last step's updates wrote")
    ap.add_argument("--no-tail-slices", action="store_true",
                    help="the forward and dX GEMMs without a workspace, so their last wave is "
                         "not cut into reduction slices (A/B of that schedule; image operands)")
    ap.add_argument("--no-extras", action="store_true",
                    help="mlp: skip the single-layer step and the SR-update sweep keys")
    ap.add_argument("--kernel", default=None,
                    help="time one kernel kind alone (fwd, bwd_dx, bwd_dw_update, bwd_dw, "
                         "bwd_dw_unfused, act_quant (with both images), act_quant_codes, "
                         "codes_to_xdq, codes_to_bf16, sr_update, act_quant_fp8, codes_to_fp8, "
                         "fwd_fp8)")
    ap.add_argument("--numel", type=int, default=1 << 26, help="weights for --kernel sr_update")
    ap.add_argument("--shape", default=None, help="T,K,N for --kernel GEMMs (default 8192,2048,5632)")
    ap.add_argument("--no-graph", action="store_true", help="decoder: run the step eagerly")
    ap.add_argument("--act", default="int8", choices=["int8", "fp8"],
                    help="mlp: 8-bit activations as int8 codes (default) or E4M3 (FP8 environment)")
    ap.add_argument("--decoder-size", default="130m", choices=sorted(DECODER_SIZES))
    ap.add_argument("--tiles", type=int, default=0, choices=[0, 1],
                    help="GEMM tiling: 0 = 2-SM 256 x 256 tiles (default), 1 = 1-SM 128 x 256 tiles")
    ap.add_argument("--optimizer", default="adamw", choices=["adamw", "adafactor"],
                    help="the DQT optimiser of the BitLinear weights")
    ap.add_argument("--packed", action="store_true", help="2-bit packed ternary code storage")
    ap.add_argument("--operands", default="img", choices=["int8", "img"],
                    help="mlp: the *_img calls on operand images written once and shared "
                         "between GEMMs (default), or the C ABI calls on int8 codes, each "
                         "making its own images in its workspace")
    ap.add_argument("--dp", default="auto", choices=["auto", "exchange", "replicas"],
                    help="several ranks: the data-parallel exchange (auto, the default) or "
                         "independent replicas; exchange on one GPU uses a one-rank group")
    ap.add_argument("--bits", type=float, default=1.58,
                    help="weight grid: 1.58 (ternary, the default) or an integer width 2..8")
    ap.add_argument("--workload", default="mlp", choices=["mlp", "decoder", "layer"],
                    help="mlp: the headline BitLinear MLP GEMM set; decoder: a DQT decoder step; "
                         "layer: one 256 x 512 x 512 BitLinear step")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.tiles and args.impl == "dqt":
        from paper_2412_04787_gb300 import build as dqt_build, dqt
        dqt_build.build()
        dqt.dqt_set_gemm_tiles(args.tiles)
    if args.workload == "decoder" and args.impl == "dqt" and not args.kernel:
        run_decoder(args)
    elif args.workload == "layer" and args.impl == "dqt" and not args.kernel:
        run_layer(args)
    elif args.kernel:
        run_kernel(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
