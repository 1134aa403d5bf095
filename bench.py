#!/usr/bin/env python
"""Throughput of the CyFA core operator on GB300 (one JSON line on stdout).

Step = one pass of the operator's hot path over one synthetic batch of the 1.4B-shaped layer
(B=2, T=32768, H=16, dk=dv=128, m=127, bf16 in / fp32 accumulate): cyfa_prepare ->
cyfa_chunk_fwd -> cyfa_chunk_bwd.  The decode path (cyfa_step, B=256 H=16 d=128 with fp32
states after a 2048-token prefill) is timed separately and reported under "decode".

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With --gpus N > 1 (one process per GPU under torch.distributed.run) every rank runs its own
batch (the (b, h) sequences are independent): weak scaling with no data-path collective; the
step time is the max over ranks.  --impl reference times the fp64 CPU oracle on the host cores.
"""
import argparse
import itertools
import json
import math
import os
import subprocess
import sys
import time

# one BLAS thread per process: the oracle baseline runs one process per core
for _v in ('OPENBLAS_NUM_THREADS', 'OMP_NUM_THREADS', 'MKL_NUM_THREADS'):
    os.environ.setdefault(_v, '1')

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = 'CyFA core-op fwd/bwd tokens/s per GB300 + % bf16 TC peak; decode GB/s vs HBM'
LAYER = dict(B=2, T=32768, H=16, d=128)          # 1.4B-shaped layer
DECODE = dict(B=256, H=16, d=128, prefill=2048)   # decode workload
MS = 128

# Issued flops per (token, head) of each kernel (d = 128, m* = 128, chunk C): the products each
# kernel's equations call for, counted 2 per multiply-add, full C x C blocks.  On the CUDA-core
# kernels these are also their share of the work; the tensor-core kernels are charged by the
# counting rule below instead.
def kernel_flops_per_token_head(name, C, d=128, ms=MS):
    table = {
        'fwd_state': 4 * d * ms,                                    # Kbar, Vbar updates
        'state_pass': 4 * d * ms,
        'fwd_out': 4 * C * d + 4 * C * ms + 4 * d * ms + 4 * ms * ms,
        'bwd_intra1': (2 * C * d + 2 * C * ms + 2 * d * ms) + 4 * ms * ms
                      + (2 * C * d + 2 * C * ms + 2 * d * ms) + 6 * ms * ms
                      + (2 * C * ms + 2 * C * d + 2 * d * ms),
        'bwd_adjoint': 4 * d * ms,
        'bwd_intra2': 4 * (2 * C * ms + 2 * C * d + 2 * d * ms),
    }
    if name in TC_PRODUCTS:
        return TC_PRODUCTS[name] * TC_PRODUCT_FLOPS
    return table.get(name)


# Tensor-core kernels: 128 x 128 x 128 products (an N = 256 product counts as two) each issues
# per 128-token chunk, and the flops one such product per chunk costs per (token, head).
TC_PRODUCTS = {'tc_seg_state': 2, 'tc_seg_out': 10, 'tc_snap_fwd': 2, 'tc_bwd_chunk1': 13,
               'tc_adj_segment': 2, 'tc_snap_adj': 2, 'tc_bwd_chunk2': 12, 'tc_dm_reduce': 2}
TC_PRODUCT_FLOPS = 2 * 128 * 128 * 128 // 128
TENSOR_KERNELS = tuple(TC_PRODUCTS)
FWD_TC = ('tc_seg_state', 'tc_seg_out')      # launched once per step by cyfa_chunk_fwd


def operator_flops_per_token_head(C, d=128, ms=MS):
    """Forward count of the chunk equations (state updates, intra-chunk, inter-chunk, middle):
    key pass 2Cd + 2Cm* + 4dm*, middle 4m*^2, value pass 2Cm* + 2Cd + 4m*d (262,144 at C = 64);
    the backward counts as twice the forward."""
    key = 2 * C * d + 2 * C * ms + 4 * d * ms
    middle = 4 * ms * ms
    value = 2 * C * ms + 2 * C * d + 4 * ms * d
    return key + middle + value


def tc_algorithmic_shares(launches_per_step, C=64):
    """Algorithmic flops per (token, head) charged to each tensor-core kernel per launch.

    Rule: the forward's algorithmic count (operator_flops_per_token_head at the caller's chunk C)
    is split over the forward's tensor-core launches, and the backward's (twice the forward) over
    the backward's, in proportion to the 128^3 products each launch issues.  Recomputation and the
    masked halves of causal blocks are therefore not credited: a kernel's share is what the
    operator's equations need of it, not what it issues."""
    fwd_alg = operator_flops_per_token_head(C)
    bwd_alg = 2 * fwd_alg
    fwd_issued, bwd_issued = {}, {}
    for k, n in launches_per_step.items():
        if k not in TC_PRODUCTS:
            continue
        nf = 1 if k in FWD_TC else 0               # the forward's own launch of this kernel
        if nf:
            fwd_issued[k] = TC_PRODUCTS[k]
        if n - nf > 0:
            bwd_issued[k] = TC_PRODUCTS[k] * (n - nf)
    tf, tb = sum(fwd_issued.values()), sum(bwd_issued.values())
    share = {}
    for k, n in launches_per_step.items():
        if k not in TC_PRODUCTS:
            continue
        total = (fwd_alg * fwd_issued.get(k, 0) / tf if tf else 0.0) + \
                (bwd_alg * bwd_issued.get(k, 0) / tb if tb else 0.0)
        share[k] = total / n                         # per launch
    return share, tf * TC_PRODUCT_FLOPS, tb * TC_PRODUCT_FLOPS


def load_peaks():
    p = os.path.join(ROOT, 'MEASURED_PEAKS.json')
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return dict(hbm_gbs=j['hbm_gbs'], bf16=j['bf16_tflops'], bf16_sus=j['bf16_tflops_sustained'],
                    sm_max_mhz=j.get('sm_max_mhz', 2070.0), src='measured')
    return dict(hbm_gbs=6800.0, bf16=1900.0, bf16_sus=1700.0, sm_max_mhz=2070.0, src='fallback')


def fp32_alu_peak_tflops(sm_mhz, sms=152):
    """CUDA-core fp32 FMA peak: 152 SMs x 128 lanes x 2 flop per clock."""
    return sms * 128 * 2 * sm_mhz * 1e6 / 1e12


# ---------------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi clock and throttle-reason samples every 50 ms; only the samples taken between
    begin() and end() (the timed region, by the host clock, with half a sampling interval of
    margin) are summarised, else the nearest one on either side of it."""
    FIELDS = ('timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,'
              'clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,'
              'clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap')
    PERIOD_MS = 50

    def __init__(self, device_index):
        self.idx = device_index
        self.proc = None
        self.t_begin = self.t_end = None
        import tempfile
        self.path = os.path.join(tempfile.gettempdir(),
                                 'cyfa_bench_clocks_%d_%d.csv' % (os.getpid(), device_index))

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, 'w')
            self.proc = subprocess.Popen(
                ['nvidia-smi', '-i', str(self.idx), '--query-gpu=' + self.FIELDS,
                 '--format=csv,noheader,nounits', '-lms', str(self.PERIOD_MS)], stdout=self.fh,
                stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return
        deadline = time.time() + 5.0   # the sampler is running before the timed region starts
        while time.time() < deadline and self.proc.poll() is None:
            try:
                if os.path.getsize(self.path) > 0:
                    break
            except OSError:
                pass
            time.sleep(0.01)

    def begin(self):
        self.t_begin = time.time()

    def end(self):
        self.t_end = time.time()

    @staticmethod
    def _when(stamp):
        import datetime
        try:
            return datetime.datetime.strptime(stamp, '%Y/%m/%d %H:%M:%S.%f').timestamp()
        except ValueError:
            return None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        names = ['hw_slowdown', 'hw_thermal_slowdown', 'sw_thermal_slowdown', 'sw_power_cap']
        rows = []
        for line in open(self.path):
            parts = [x.strip() for x in line.split(',')]
            if len(parts) < 10:
                continue
            try:
                sm, smax = float(parts[2]), float(parts[3])
            except ValueError:
                continue
            active = {nm for nm, val in zip(names, parts[6:10]) if val.lower() == 'active'}
            rows.append((self._when(parts[0]), sm, smax, active))
        try:
            os.remove(self.path)
        except OSError:
            pass
        if not rows:
            return None
        use, where = rows, 'all samples'
        if self.t_begin is not None and self.t_end is not None and all(r[0] for r in rows):
            m = 0.5e-3 * self.PERIOD_MS
            inside = [r for r in rows if self.t_begin - m <= r[0] <= self.t_end + m]
            if inside:
                use, where = inside, 'timed region'
            else:
                before = [r for r in rows if r[0] < self.t_begin]
                after = [r for r in rows if r[0] > self.t_end]
                use = before[-1:] + after[:1]
                where = 'nearest samples around the timed region'
        sm = sorted(r[1] for r in use)
        reasons = set()
        for r in use:
            reasons |= r[3]
        return {'sm_mhz': sm[len(sm) // 2], 'sm_max_mhz': use[-1][2], 'reasons': sorted(reasons),
                'samples': len(use), 'sampled': where, 'period_ms': self.PERIOD_MS}


# --------------------------------------------------------------------------- cpu baseline
def _oracle_pair_worker(args):
    """One (b, h) sequence through the fp64 oracle, forward and backward; returns seconds."""
    import numpy as np
    from oracle import backward as OB, forward as OF, gates as OG
    q, k, v, c, f, bl, A, R, dO, scale = args
    t0 = time.perf_counter()
    OF.absolute_clock(q, k, v, OG.clock_increment(c), OG.forget_gate(f, A[:, None]),
                      OG.write_strength(bl), R, scale)
    OB.backward(q, k, v, c, f, bl, A, R, scale, dO)
    return time.perf_counter() - t0


def _oracle_warm(_):
    import oracle.backward  # noqa: F401
    return 0


def oracle_baseline(T_sample, H_full, cores=None, reps=1):
    """Time the oracle on `cores` (b, h) sequences of T_sample tokens of the layer's shape, one
    process per core, `reps` times over; returns (tokens/s of the full layer, cores, sample text,
    seconds per rep, slowest sequence)."""
    import multiprocessing as mp
    import numpy as np
    import torch
    from paper_2609_36259_gb300 import synth
    cores = cores or os.cpu_count() or 1
    inp = synth.make_inputs(1, T_sample, cores, LAYER['d'], seed=123, with_dO=True)
    jobs = []
    for h in range(cores):
        def P(x):
            return x[0, :, h].double().numpy()[None]
        A = np.array([float(synth.decay_scales(H_full)[h % H_full])])
        R = inp['R'][h:h + 1].double().numpy()
        jobs.append((P(inp['q']), P(inp['k']), P(inp['v']), P(inp['clock_logit']),
                     P(inp['decay_logit']), P(inp['beta_logit']), A, R, P(inp['dO']),
                     inp['scale']))
    ctx = mp.get_context('spawn')
    with ctx.Pool(cores) as pool:
        pool.map(_oracle_warm, range(cores))          # start the workers and import the oracle
        t0 = time.perf_counter()
        for _ in range(reps):
            per = pool.map(_oracle_pair_worker, jobs)
        wall = (time.perf_counter() - t0) / reps
    token_heads = cores * T_sample
    value = token_heads / H_full / wall
    sample = ('%d (b,h) sequences x %d tokens of the layer, fwd+bwd, d=128, m=127, one process '
              'per core; tokens/s = token-heads / H(=%d) / wall' % (cores, T_sample, H_full))
    return value, cores, sample, wall, max(per)


def workload_config(world, C, with_dR):
    """The workload both arms run (one line of each names the same one)."""
    B, T, H, D = LAYER['B'], LAYER['T'], LAYER['H'], LAYER['d']
    return {'workload': 'cyfa-1.4B-layer prepare+fwd+bwd', 'model': 'CyFA core operator',
            'B': B, 'T': T, 'H': H, 'dk': D, 'dv': D, 'm': 127, 'm_store': MS, 'chunk': C,
            'io_dtype': 'bf16',
            'grads': 'q, k, v, clock, decay, beta logits, A' + (', R' if with_dR else ''),
            'global_batch': B * world, 'seq_len': T, 'parallelism': 'dp%d' % world,
            'l2': 'inputs larger than L2 (q,k,v,dO %.0f MB)' % (4 * B * T * H * D * 2 / 1e6)}


# ------------------------------------------------------------------------- multi-rank
def job_step_ms(ms, dist=None, device=None):
    """The job's step time: the max over ranks of each rank's own step time (every rank must call
    this; a rank on its own returns its time)."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank, world, ms):
    """Whole-job throughput: every rank processes its own batch (weak scaling)."""
    return tokens_per_rank * world / (ms / 1e3)


# --------------------------------------------------------------------------------- ours
def run_ours(args):
    import numpy as np
    import torch
    from paper_2609_36259_gb300 import cyfa, synth

    world = int(os.environ.get('WORLD_SIZE', '1'))
    rank = int(os.environ.get('RANK', '0'))
    local = int(os.environ.get('LOCAL_RANK', '0'))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group('nccl', device_id=torch.device('cuda', local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device('cuda', torch.cuda.current_device())
    peaks = load_peaks()

    # CPU baseline first: its process pool is spawned before any GPU work of this process
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, cores, sample, wall, _ = oracle_baseline(args.oracle_tokens, LAYER['H'],
                                                    reps=args.cpu_reps)
        cpu = {'value': v, 'unit': 'tokens/s', 'cores': cores, 'kind': 'oracle',
               'sample': sample + ', mean of %d repetitions' % args.cpu_reps,
               'seconds': round(wall * args.cpu_reps, 2)}

    B, T, H, D, C = LAYER['B'], LAYER['T'], LAYER['H'], LAYER['d'], args.chunk
    d = cyfa.dims(B, T, H, D, chunk=C, cuda_cores=args.cuda_cores)
    inp = synth.make_inputs(B, T, H, D, seed=rank, device=dev, with_dO=True)
    f32 = dict(dtype=torch.float32, device=dev)
    lam = torch.empty(B, T, H, **f32)
    g = torch.empty_like(lam)
    beta = torch.empty_like(lam)
    o = torch.empty_like(inp['v'])
    dq, dk, dv = torch.empty_like(inp['q']), torch.empty_like(inp['k']), torch.empty_like(inp['v'])
    dc, dd, db = torch.empty_like(lam), torch.empty_like(lam), torch.empty_like(lam)
    dA = torch.empty(H, **f32)
    # the readout's gradient (a training step needs it)
    dR = None if args.no_dR else torch.empty(H, 127, 127, **f32)
    ws_p = cyfa.workspace(d, cyfa.CYFA_WS_PREPARE, dev)
    ws_f = cyfa.workspace(d, cyfa.CYFA_WS_FWD, dev)
    ws_b = cyfa.workspace(d, cyfa.CYFA_WS_BWD, dev)
    # the forward saves its chunk-start states for the backward (a training step keeps them)
    saved = None if args.no_saved else cyfa.saved_buffer(d, dev)
    # the library's rule for the tensor-core kernels (bf16 inputs, m = 127 here)
    tc_path = not args.cuda_cores and D == 128 and T % 128 == 0
    stream = torch.cuda.current_stream()

    def step(x):
        cyfa.cyfa_prepare(d, x['clock_logit'], x['decay_logit'], x['beta_logit'], x['A'], None,
                          lam, g, beta, None, ws_p)
        cyfa.cyfa_chunk_fwd(d, x['q'], x['k'], x['v'], lam, g, beta, x['R'], None, None, o, None,
                            None, ws_f, saved=saved)
        if args.no_bwd:
            return
        cyfa.cyfa_chunk_bwd(d, x['q'], x['k'], x['v'], lam, g, beta, x['R'], x['clock_logit'],
                            x['decay_logit'], x['A'], x['dO'], dq, dk, dv, dc, dd, db, dR, dA,
                            ws_b, saved=saved)

    for _ in range(args.warmup):
        step(inp)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    cyfa.cyfa_stats_reset()
    cyfa.cyfa_stats_timing(True)
    clocks = ClockSampler(dev.index)
    clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    clocks.begin()
    e0.record(stream)
    for _ in range(args.steps):
        step(inp)
    e1.record(stream)
    torch.cuda.synchronize()
    clocks.end()
    clk = clocks.stop()
    cyfa.cyfa_check()
    ms = e0.elapsed_time(e1) / args.steps
    stats = cyfa.cyfa_stats_get()
    cyfa.cyfa_stats_timing(False)
    ms = job_step_ms(ms, dist, dev)
    value = job_tokens_per_s(B * T, world, ms)
    launches = sum(n for n, _ in stats.values())

    # per-kernel times and the forward / backward split
    per_kernel = {k: {'launches': n, 'ms_per_launch': t / n if n else 0.0}
                  for k, (n, t) in stats.items()}
    fwd_names = ('readout_matrix', 'readout_f16', 'fwd_state', 'fwd_out', 'tc_seg_state',
                 'tc_seg_scan', 'tc_seg_out')
    # the forward's kernels are launched again inside the backward (recomputation): split by
    # launch count, one forward's worth per step belongs to cyfa_chunk_fwd
    def fwd_share(k):
        n, t = stats[k]
        return t * min(1.0, args.steps / n) if n else 0.0
    fwd_ms = sum(fwd_share(k) for k in stats if k in fwd_names) / args.steps
    prep_ms = sum(stats[k][1] for k in stats if k.startswith('prep')) / args.steps
    bwd_ms = (sum(stats[k][1] for k in stats if not k.startswith('prep')) / args.steps) - fwd_ms
    token_heads = B * T * H
    op_flops = operator_flops_per_token_head(C) * token_heads      # counting rule at the chunk C
    step_ms_kernels = fwd_ms + bwd_ms + prep_ms
    fwd = {'ms': fwd_ms, 'tokens_per_s': B * T / (fwd_ms / 1e3) if fwd_ms else None,
           'tflops_rule': op_flops / (fwd_ms / 1e3) / 1e12 if fwd_ms else None}
    bwd = {'ms': bwd_ms, 'tokens_per_s': B * T / (bwd_ms / 1e3) if bwd_ms else None,
           'tflops_rule': 2 * op_flops / (bwd_ms / 1e3) / 1e12 if bwd_ms else None}
    for ph in (fwd, bwd):
        ph['frac_bf16_peak'] = ph['tflops_rule'] / peaks['bf16'] if ph['tflops_rule'] else None
    step_tf = (3 * op_flops if not args.no_bwd else op_flops) / (ms / 1e3) / 1e12
    tensor_frac = {'rule': 'fwd %d, bwd 2x fwd flops per token-head (chunk %d); '
                           'of the measured bf16 burst peak %.1f TFLOP/s'
                           % (operator_flops_per_token_head(C), C, peaks['bf16']),
                   'fwd': fwd['frac_bf16_peak'], 'bwd': bwd['frac_bf16_peak'],
                   'step': step_tf / peaks['bf16'], 'step_tflops': step_tf}

    # roofline of every kernel, and of the dominant one.  Tensor-core kernels are charged their
    # share of the counting rule (tc_algorithmic_shares) against the bf16 burst peak: the timed
    # region is a sub-second run of millisecond steps, not a seconds-long loop under the power cap.
    per_step = {k: n / args.steps for k, (n, _) in stats.items()}
    shares, _, _ = tc_algorithmic_shares(per_step, C)
    def roofline_of(name):
        n_k, t_k = stats[name]
        if n_k == 0 or t_k <= 0:
            return None
        if name in TENSOR_KERNELS:
            fl = shares.get(name)
            issued = kernel_flops_per_token_head(name, C) * token_heads
            peak, bound = peaks['bf16'], 'tensor'
            src = '%s bf16 burst (fp16 operands: the same tensor rate)' % peaks['src']
        else:
            C_k = 64 if name.startswith('bwd') or name == 'state_pass' else C
            fl = kernel_flops_per_token_head(name, C_k)
            issued = None
            peak, bound = fp32_alu_peak_tflops(peaks['sm_max_mhz']), 'alu'
            src = 'fp32 FMA: 152 SMs x 128 lanes x 2 x %.0f MHz' % peaks['sm_max_mhz']
        if fl is None:
            return None
        achieved = fl * token_heads / (t_k / n_k / 1e3) / 1e12
        r = {'kernel': name, 'bound': bound, 'achieved': round(achieved, 3),
             'peak': round(peak, 2), 'unit': 'TFLOP/s', 'frac': round(achieved / peak, 4),
             'traffic': load_traffic(name), 'flops_per_launch': fl * token_heads,
             'issued_flops': issued, 'ms_per_launch': t_k / n_k, 'peak_source': src}
        return r
    rooflines = {k: roofline_of(k) for k in stats}
    rooflines = {k: v for k, v in rooflines.items() if v is not None}
    top = max(stats.items(), key=lambda kv: kv[1][1])[0]
    roof = rooflines.get(top)

    # decode: B=256, H=16, fp32 states after a 2048-token prefill
    dec = None
    if not args.no_decode:
        dec = run_decode(args, dev, peaks, rank)

    # packed variable-length sequences and the fixed-rate clock on the same layer
    varlen = None
    if not args.no_varlen:
        varlen = run_varlen(args, dev, rank)

    # the paper's own kernel shape (H = 4, d = 256, T = 2048, B = 32)
    paper = slots = slots255 = None
    if not args.no_paper_shape:
        paper = run_paper_shape(args, dev, rank, peaks)
        slots = run_slots_variant(args, dev, rank, peaks)
        slots255 = run_slots_255(args, dev, rank, peaks)

    mixer = None if args.no_mixer else run_mixer(args, dev, rank, peaks)

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, inp, dev, want_dR=dR is not None)

    del ws_f, ws_b
    line = {
        'metric': METRIC, 'value': value, 'unit': 'tokens/s', 'n_gpus': world,
        'steps': args.steps, 'warmup': args.warmup, 'ms_per_step': ms,
        'higher_is_better': True, 'scaling': 'weak', 'vs_baseline': None,
        'dtype': 'fp16' if tc_path else 'fp32',
        'data': 'synthetic',
        'config': workload_config(world, C, dR is not None),
        'impl_detail': {'kernel_chunk': 128 if tc_path else C,
                        'arithmetic': ('tcgen05 fp16 operands, fp32 accumulate' if tc_path
                                       else 'fp32 CUDA cores'),
                        'saved_states': saved is not None},
        'roofline': roof, 'kernel_rooflines': rooflines, 'cpu_baseline': cpu, 'e2e': e2e, 'gpu_launches': launches,
        'clocks': clk, 'tensor_frac': tensor_frac, 'fwd': fwd, 'bwd': bwd,
        'prepare_ms': prep_ms, 'kernel_ms_per_step': step_ms_kernels, 'decode': dec,
        'varlen': varlen, 'paper_shape': paper, 'slots_m63': slots, 'slots_m255': slots255,
        'mixer': mixer,
        'kernels': per_kernel,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


def load_traffic(kernel):
    """DRAM bytes per launch from the committed ncu summary, if it was taken of the current
    kernel source (its sha256 recorded beside the number)."""
    import hashlib
    p = os.path.join(ROOT, 'profiles', 'traffic.json')
    if not os.path.exists(p):
        return None
    with open(p) as f:
        j = json.load(f)
    ent = j.get(kernel)
    if not ent:
        return None
    srcs = ent.get('sources') or {ent['source']: ent.get('source_sha256')}
    for rel, want in srcs.items():
        src = os.path.join(ROOT, rel)
        if not os.path.exists(src) or hashlib.sha256(open(src, 'rb').read()).hexdigest() != want:
            return None
    return ent['bytes_per_launch']


def run_decode(args, dev, peaks, rank):
    import torch
    from paper_2609_36259_gb300 import cyfa, synth
    B, H, D, T0 = args.decode_batch, DECODE['H'], DECODE['d'], DECODE['prefill']
    S = args.decode_steps
    inp = synth.make_inputs(B, T0, H, D, seed=1000 + rank, device=dev)
    d0 = cyfa.dims(B, T0, H, D, chunk=64)
    lam, g, beta, lend = cyfa.prepare(d0, inp['clock_logit'], inp['decay_logit'],
                                      inp['beta_logit'], inp['A'], want_lambda_end=True)
    _, K, V = cyfa.forward(d0, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                           want_state=True)
    del inp, lam, g, beta
    torch.cuda.empty_cache()
    stepi = synth.make_inputs(B, S, H, D, seed=2000 + rank, device=dev)
    xs = {k: stepi[k].transpose(0, 1).contiguous() for k in
          ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit')}
    ds = cyfa.dims(B, 1, H, D)
    o = torch.empty(B, H, D, dtype=torch.bfloat16, device=dev)

    def one(t):
        cyfa.cyfa_step(ds, xs['q'][t], xs['k'][t], xs['v'][t], xs['clock_logit'][t],
                       xs['decay_logit'][t], xs['beta_logit'][t], stepi['A'], stepi['R'], K, V,
                       lend, o)
    for t in range(min(3, S)):
        one(t)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for t in range(S):
        one(t)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / S
    bytes_step = B * H * (2 * 2 * MS * D * 4 + 3 * D * 2 + D * 2 + 3 * 4 + 2 * 8)
    gbs = bytes_step / (ms / 1e3) / 1e9
    return {'workload': 'B=%d H=%d d=%d fp32 states, %d-token prefill, %d steps' % (B, H, D, T0, S),
            'ms_per_step': ms, 'tokens_per_s': B / (ms / 1e3), 'GB_per_s': gbs,
            'bytes_per_step': bytes_step, 'frac_hbm_measured': gbs / peaks['hbm_gbs'],
            'traffic': load_traffic('decode_step') if B == DECODE['B'] else None,
            'frac_hbm_8TBs': gbs / 8000.0}


def run_paper_shape(args, dev, rank, peaks):
    """prepare + forward + backward (every gradient) at the shape of the paper's kernel-latency
    figure: B = 32, T = 2048, H = 4, d_k = d_v = 256, m = 127, bf16 inputs."""
    return run_extra_shape(args, dev, rank, peaks, 32, 2048, 4, 256, 127,
                           "the paper's kernel-latency shape")


def run_slots_variant(args, dev, rank, peaks):
    """The same step on the 1.4B-shaped layer with m = 63 slots (the paper's slot ablation)."""
    return run_extra_shape(args, dev, rank, peaks, LAYER['B'], LAYER['T'], LAYER['H'],
                           LAYER['d'], 63, 'the 1.4B layer with m = 63 (slot ablation)')


def run_slots_255(args, dev, rank, peaks):
    """m = 255 slots (256 storage rows) at the shape of the paper's ablation model (400M:
    B = 32, T = 2048, H = 4, d = 256), the slot ablation's best variant."""
    return run_extra_shape(args, dev, rank, peaks, 32, 2048, 4, 256, 255,
                           'the 400M ablation shape with m = 255 (slot ablation)')


def run_extra_shape(args, dev, rank, peaks, B, T, H, D, m, what):
    import torch
    from paper_2609_36259_gb300 import cyfa, synth
    C = 64
    inp = synth.make_inputs(B, T, H, D, seed=4000 + rank, device=dev, with_dO=True, m=m)
    d = cyfa.dims(B, T, H, D, chunk=C, m=m)
    f32 = dict(dtype=torch.float32, device=dev)
    lam, g, beta = (torch.empty(B, T, H, **f32) for _ in range(3))
    o = torch.empty_like(inp['v'])
    dq, dk, dv = (torch.empty_like(inp[x]) for x in ('q', 'k', 'v'))
    dc, dd, db = (torch.empty_like(lam) for _ in range(3))
    dA, dR = torch.empty(H, **f32), torch.empty(H, m, m, **f32)
    ws = [cyfa.workspace(d, w, dev) for w in (cyfa.CYFA_WS_PREPARE, cyfa.CYFA_WS_FWD,
                                               cyfa.CYFA_WS_BWD)]
    # the forward keeps its chunk-start states for the backward where the kernels can
    saved = None if args.no_saved else cyfa.saved_buffer(d, dev)

    def fwd():
        cyfa.cyfa_prepare(d, inp['clock_logit'], inp['decay_logit'], inp['beta_logit'], inp['A'],
                          None, lam, g, beta, None, ws[0])
        cyfa.cyfa_chunk_fwd(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'], None, None,
                            o, None, None, ws[1], saved=saved)

    def step():
        fwd()
        cyfa.cyfa_chunk_bwd(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                            inp['clock_logit'], inp['decay_logit'], inp['A'], inp['dO'], dq, dk,
                            dv, dc, dd, db, dR, dA, ws[2], saved=saved)

    def timed(fn, n):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    n = max(1, min(args.steps, 20))
    ms = timed(step, n)
    ms_fwd = timed(fwd, n)
    # per-kernel split of two more steps (CUDA events around each launch)
    cyfa.cyfa_stats_reset()
    cyfa.cyfa_stats_timing(True)
    for _ in range(2):
        step()
    torch.cuda.synchronize()
    split = {k: round(t / 2, 4) for k, (_, t) in sorted(cyfa.cyfa_stats_get().items(),
                                                         key=lambda kv: -kv[1][1])}
    cyfa.cyfa_stats_timing(False)
    cyfa.cyfa_check()
    th = B * T * H
    fl = operator_flops_per_token_head(C, d=D, ms=m + 1) * th
    # the library's rule for the tensor-core kernels (bf16 inputs here)
    tc = D == 128 and 63 <= m <= 127 and T % 128 == 0
    peak = peaks['bf16'] if tc else fp32_alu_peak_tflops(peaks['sm_max_mhz'])
    tf = 3 * fl / (ms / 1e3) / 1e12
    return {'workload': 'B=%d T=%d H=%d d=%d m=%d chunk %d (%s), prepare + fwd + bwd with every '
                        'gradient' % (B, T, H, D, m, C, what),
            'path': ('tensor-core kernels (128 storage rows, m* = %d counted)' % (m + 1) if tc else
                     'fp32 CUDA-core kernels (the tensor-core kernels take bf16, d = 128, '
                     '63 <= m <= 127)'),
            'ms_per_step': ms, 'tokens_per_s': B * T / (ms / 1e3),
            'fwd_ms': ms_fwd, 'fwd_tokens_per_s': B * T / (ms_fwd / 1e3),
            'tflops_rule': tf, 'peak_tflops': peak,
            'peak_source': 'measured bf16 burst' if tc else 'fp32 FMA: 152 x 128 x 2 x clock',
            'frac_peak': tf / peak, 'saved_states': saved is not None,
            'kernel_ms_per_step': split}


def run_mixer(args, dev, rank, peaks):
    """The mixer's neighbours on the layer's activations (bf16 [B, T, H, d]): ShortConv + SiLU +
    QK RMSNorm before the operator and head RMSNorm + sigmoid gate after it, forward and backward.
    HBM-bound: algorithmic bytes are each call's tensors read and written once (parameters and
    their partial sums are under 0.1%)."""
    import torch
    from paper_2609_36259_gb300 import cyfa
    B, T, H, D = LAYER['B'], LAYER['T'], LAYER['H'], LAYER['d']
    g = torch.Generator(device=dev).manual_seed(5000 + rank)
    mk = lambda: torch.randn(B, T, H, D, generator=g, device=dev).to(torch.bfloat16)
    x = [mk() for _ in range(3)]
    dy = [mk() for _ in range(3)]
    y = [torch.empty_like(t) for t in x]
    dx = [torch.empty_like(t) for t in x]
    w = [torch.randn(H * D, 4, generator=g, device=dev) for _ in range(3)]
    dw = [torch.empty_like(t) for t in w]
    gains = [torch.ones(D, device=dev) for _ in range(3)]
    dgs = [torch.empty_like(t) for t in gains]
    d = cyfa.dims(B, T, H, D, chunk=args.chunk)
    ws = cyfa.workspace(d, cyfa.CYFA_WS_MIXER, dev)
    calls = {
        'pre_fwd': (lambda: cyfa.cyfa_mixer_pre(d, *x, *w, gains[0], gains[1], 1e-6, *y), 6),
        'pre_bwd': (lambda: cyfa.cyfa_mixer_pre_bwd(d, *x, *w, gains[0], gains[1], 1e-6, *dy,
                                                    *dx, *dw, dgs[0], dgs[1], ws), 9),
        'post_fwd': (lambda: cyfa.cyfa_mixer_post(d, x[0], x[1], gains[2], 1e-6, y[0]), 3),
        'post_bwd': (lambda: cyfa.cyfa_mixer_post_bwd(d, x[0], x[1], gains[2], 1e-6, dy[0], dx[0],
                                                      dx[1], dgs[2], ws), 5),
    }
    out = {'workload': 'B=%d T=%d H=%d d=%d bf16' % (B, T, H, D)}
    for name, (fn, ntens) in calls.items():
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n = 20
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / n
        nbytes = ntens * B * T * H * D * 2
        out[name] = {'ms': ms, 'bytes': nbytes, 'GB_per_s': nbytes / (ms / 1e3) / 1e9,
                     'frac_hbm_measured': nbytes / (ms / 1e3) / 1e9 / peaks['hbm_gbs']}
    cyfa.cyfa_check()
    return out


def run_varlen(args, dev, rank):
    """The layer's B*T tokens as one packed stream of sequences of mixed length around 2,048
    tokens (cyfa_prepare_varlen + forward + backward with every gradient, saved states), and the
    prepare of the fixed-rate clock (cyfa_prepare_fixed_rate, no scan) beside the learned one."""
    import torch
    from paper_2609_36259_gb300 import cyfa, synth
    B, T, H, D = LAYER['B'], LAYER['T'], LAYER['H'], LAYER['d']
    N = B * T
    lengths = synth.varlen_lengths(N, 2048, seed=rank)
    inp = synth.make_inputs(1, N, H, D, seed=3000 + rank, device=dev, with_dO=True)
    cu = torch.tensor([0] + list(itertools.accumulate(lengths)), dtype=torch.int32, device=dev)
    d = cyfa.dims(1, N, H, D, chunk=args.chunk)
    f32 = dict(dtype=torch.float32, device=dev)
    lam, g, beta = (torch.empty(1, N, H, **f32) for _ in range(3))
    o = torch.empty_like(inp['v'])
    dq, dk, dv = (torch.empty_like(inp[x]) for x in ('q', 'k', 'v'))
    dc, dd, db = (torch.empty_like(lam) for _ in range(3))
    dA, dR = torch.empty(H, **f32), torch.empty(H, 127, 127, **f32)
    ws_v = cyfa.workspace(d, cyfa.CYFA_WS_PREPARE_VARLEN, dev)
    ws_f = cyfa.workspace(d, cyfa.CYFA_WS_FWD, dev)
    ws_b = cyfa.workspace(d, cyfa.CYFA_WS_BWD, dev)
    saved = cyfa.saved_buffer(d, dev)

    def step():
        cyfa.cyfa_prepare_varlen(d, cu, len(lengths), inp['clock_logit'], 0.0, inp['decay_logit'],
                                 inp['beta_logit'], inp['A'], None, lam, g, beta, None, ws_v)
        cyfa.cyfa_chunk_fwd(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'], None, None,
                            o, None, None, ws_f, saved=saved)
        cyfa.cyfa_chunk_bwd(d, inp['q'], inp['k'], inp['v'], lam, g, beta, inp['R'],
                            inp['clock_logit'], inp['decay_logit'], inp['A'], inp['dO'], dq, dk,
                            dv, dc, dd, db, dR, dA, ws_b, saved=saved)

    def timed(fn, n):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(n):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    ms = timed(step, max(1, args.steps))
    cyfa.cyfa_check()
    ws_p = cyfa.workspace(d, cyfa.CYFA_WS_PREPARE, dev)
    ms_prep = timed(lambda: cyfa.cyfa_prepare(d, inp['clock_logit'], inp['decay_logit'],
                                              inp['beta_logit'], inp['A'], None, lam, g, beta,
                                              None, ws_p), 20)
    ms_prepv = timed(lambda: cyfa.cyfa_prepare_varlen(d, cu, len(lengths), inp['clock_logit'],
                                                      0.0, inp['decay_logit'], inp['beta_logit'],
                                                      inp['A'], None, lam, g, beta, None, ws_v), 20)
    ms_fixed = timed(lambda: cyfa.cyfa_prepare_fixed_rate(d, 2.0, inp['decay_logit'],
                                                          inp['beta_logit'], inp['A'], None, lam,
                                                          g, beta, None), 20)
    return {'workload': '%d tokens H=%d d=%d as %d packed sequences (log-normal lengths, mean '
                        '2048, %d..%d), prepare_varlen + fwd + bwd with every gradient'
                        % (N, H, D, len(lengths), min(lengths), max(lengths)),
            'ms_per_step': ms, 'tokens_per_s': N / (ms / 1e3),
            'prepare_ms': ms_prep, 'prepare_varlen_ms': ms_prepv,
            'prepare_fixed_rate_ms': ms_fixed}


def run_e2e(args, inp, dev, want_dR):
    """The step through the public API with pinned host buffers: every step copies all its inputs
    host->device and reads every output back.  The (b, h) sequences are independent, so the step
    runs as micro-batches of one batch row and a group of heads (host buffers laid out per
    micro-batch), spread round-robin over a few CUDA streams with a workspace each: one
    micro-batch's copies run under another's kernels, the two copy directions overlap, and the
    next step's uploads start while this step's last results come back (a stream's micro-batches
    run in order, so its device buffers are never reused early).  The per-micro-batch dA / dR
    partials are read back and summed on the host."""
    import torch
    from paper_2609_36259_gb300 import cyfa
    B, T, H, D = inp['q'].shape
    hg = args.e2e_heads if H % args.e2e_heads == 0 else H
    keys = ('q', 'k', 'v', 'clock_logit', 'decay_logit', 'beta_logit', 'dO')
    d1 = cyfa.dims(1, T, hg, D, chunk=args.chunk, cuda_cores=args.cuda_cores)
    nstream = max(1, min(args.e2e_streams, B * (H // hg)))
    streams = [torch.cuda.Stream(device=dev) for _ in range(nstream)]
    ws = [[cyfa.workspace(d1, w, dev) for w in (cyfa.CYFA_WS_PREPARE, cyfa.CYFA_WS_FWD,
                                                 cyfa.CYFA_WS_BWD)] for _ in range(nstream)]
    saved = [None if args.no_saved else cyfa.saved_buffer(d1, dev) for _ in range(nstream)]
    f32 = dict(dtype=torch.float32, device=dev)
    mbs = []
    for b in range(B):
        for h0 in range(0, H, hg):
            sl = slice(h0, h0 + hg)
            m = {'stream': len(mbs) % nstream}
            m['host'] = {k: inp[k][b:b + 1, :, sl].contiguous().cpu().pin_memory() for k in keys}
            m['x'] = {k: torch.empty(m['host'][k].shape, dtype=m['host'][k].dtype, device=dev)
                      for k in keys}
            m['x']['A'] = inp['A'][sl].contiguous()
            m['x']['R'] = inp['R'][sl].contiguous()
            lam = torch.empty(1, T, hg, **f32)
            m['gates'] = (lam, torch.empty_like(lam), torch.empty_like(lam))
            m['out'] = dict(o=torch.empty_like(m['x']['v']), dq=torch.empty_like(m['x']['q']),
                            dk=torch.empty_like(m['x']['k']), dv=torch.empty_like(m['x']['v']),
                            dc=torch.empty_like(lam), dd=torch.empty_like(lam),
                            db=torch.empty_like(lam), dA=torch.empty(hg, **f32))
            if want_dR:
                m['out']['dR'] = torch.empty(hg, 127, 127, **f32)
            m['host_out'] = {k: t.new_empty(t.shape, device='cpu').pin_memory()
                             for k, t in m['out'].items()}
            m['h0'] = h0
            mbs.append(m)
    h2d = sum(t.numel() * t.element_size() for m in mbs for t in m['host'].values())
    d2h = sum(t.numel() * t.element_size() for m in mbs for t in m['host_out'].values())

    def one():
        for m in mbs:
            si = m['stream']
            st, x, o = streams[si], m['x'], m['out']
            with torch.cuda.stream(st):
                for k in keys:
                    x[k].copy_(m['host'][k], non_blocking=True)
                lam, g, beta = m['gates']
                w = ws[si]
                cyfa.cyfa_prepare(d1, x['clock_logit'], x['decay_logit'], x['beta_logit'], x['A'],
                                  None, lam, g, beta, None, w[0], stream=st)
                cyfa.cyfa_chunk_fwd(d1, x['q'], x['k'], x['v'], lam, g, beta, x['R'], None, None,
                                    o['o'], None, None, w[1], stream=st, saved=saved[si])
                cyfa.cyfa_chunk_bwd(d1, x['q'], x['k'], x['v'], lam, g, beta, x['R'],
                                    x['clock_logit'], x['decay_logit'], x['A'], x['dO'], o['dq'],
                                    o['dk'], o['dv'], o['dc'], o['dd'], o['db'], o.get('dR'),
                                    o['dA'], w[2], stream=st, saved=saved[si])
                for k, t in o.items():
                    m['host_out'][k].copy_(t, non_blocking=True)

    for _ in range(2):
        one()
    torch.cuda.synchronize()
    n = max(1, args.steps)
    t0 = time.perf_counter()
    for _ in range(n):
        one()
    torch.cuda.synchronize()
    # the batch sums of dA and dR from the micro-batches' partials (host side, inside the clock)
    dA = torch.zeros(H)
    for m in mbs:
        dA[m['h0']:m['h0'] + hg] += m['host_out']['dA']
    if want_dR:
        dR = torch.zeros(H, 127, 127)
        for m in mbs:
            dR[m['h0']:m['h0'] + hg] += m['host_out']['dR']
    wall = (time.perf_counter() - t0) / n
    return {'value': B * T / wall, 'unit': 'tokens/s', 'h2d_bytes_per_step': h2d,
            'd2h_bytes_per_step': d2h, 'ms_per_step': wall * 1e3,
            'micro_batches': len(mbs), 'heads_per_micro_batch': hg, 'streams': nstream,
            'timing': 'host wall clock over %d back-to-back steps, synchronised at both ends' % n}


# ---------------------------------------------------------------------------- reference
def run_reference(args):
    world = int(os.environ.get('WORLD_SIZE', '1'))
    rank = int(os.environ.get('RANK', '0'))
    if rank != 0:
        return
    B, T, H = LAYER['B'], LAYER['T'], LAYER['H']
    for _ in range(args.warmup):
        pass   # the oracle has no warm state; warm-up steps would only repeat the sample
    walls = []
    vals = []
    cores = None
    sample = None
    for _ in range(args.steps):
        v, cores, sample, wall, _ = oracle_baseline(args.oracle_tokens, H)
        vals.append(v)
        walls.append(wall)
    value = sum(vals) / len(vals)
    line = {
        'impl': 'reference', 'metric': METRIC, 'value': value, 'unit': 'tokens/s',
        'n_gpus': world, 'steps': args.steps, 'warmup': args.warmup,
        'ms_per_step': 1e3 * sum(walls) / len(walls), 'higher_is_better': True,
        'scaling': 'weak', 'vs_baseline': None, 'dtype': 'f64', 'data': 'synthetic',
        'config': workload_config(world, args.chunk, not args.no_dR),
        'cpu_baseline': {'value': value, 'unit': 'tokens/s', 'cores': cores, 'kind': 'oracle',
                         'sample': sample},
        'e2e': {'value': value, 'unit': 'tokens/s', 'h2d_bytes_per_step': 0,
                'd2h_bytes_per_step': 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument('--gpus', type=int, default=1)
    ap.add_argument('--steps', type=int, default=200)
    ap.add_argument('--warmup', type=int, default=5)
    ap.add_argument('--impl', default='ours', choices=['ours', 'reference'])
    ap.add_argument('--chunk', type=int, default=64, choices=[64, 128])
    ap.add_argument('--decode-steps', type=int, default=1024)
    ap.add_argument('--decode-batch', type=int, default=DECODE['B'],
                    help='decode batch (profiling runs on smaller cases)')
    ap.add_argument('--oracle-tokens', type=int, default=4096,
                    help='tokens per (b,h) sequence of one oracle sample (cpu_baseline and the '
                         'reference arm time the same sample)')
    ap.add_argument('--cpu-reps', type=int, default=4,
                    help='oracle samples timed for cpu_baseline')
    ap.add_argument('--shape', default=None,
                    help='B,T,H override of the layer shape (profiling runs on smaller cases)')
    ap.add_argument('--no-decode', action='store_true')
    ap.add_argument('--no-e2e', action='store_true')
    ap.add_argument('--e2e-heads', type=int, default=8,
                    help='heads per micro-batch of the end-to-end step')
    ap.add_argument('--e2e-streams', type=int, default=4)
    ap.add_argument('--no-varlen', action='store_true')
    ap.add_argument('--no-paper-shape', action='store_true')
    ap.add_argument('--no-mixer', action='store_true')
    ap.add_argument('--no-dR', action='store_true',
                    help='leave the readout gradient dR out of the backward')
    ap.add_argument('--no-saved', action='store_true',
                    help='backward recomputes the chunk-start states instead of reading the '
                         'ones the forward saved')
    ap.add_argument('--no-cpu-baseline', action='store_true')
    ap.add_argument('--no-bwd', action='store_true',
                    help='time prepare + forward only (profiling runs; not the headline step)')
    ap.add_argument('--cuda-cores', action='store_true',
                    help='run the chunk calls on the fp32 CUDA-core kernels')
    args = ap.parse_args()
    if args.shape:
        LAYER['B'], LAYER['T'], LAYER['H'] = (int(x) for x in args.shape.split(','))
    if args.warmup < 3 and args.impl == 'ours':
        args.warmup = 3
    if args.impl == 'reference':
        run_reference(args)
    else:
        run_ours(args)


if __name__ == '__main__':
    main()
