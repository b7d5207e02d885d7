"""Seeded synthetic workloads for the MAPS scheduler hot path.

This module only draws random inputs. It holds none of the scheduler's
arithmetic (no residuals, quantiles, bounds, occupancy, scores or orderings):
both the CPU oracle tests and the CUDA path take its arrays as plain inputs.

The paper evaluates on ShareGPT / BurstGPT / Alpaca traces, which are not
available here; the distributions below stand in for them.  Every array is
drawn from ``numpy.random.default_rng`` children of one ``SeedSequence`` per
workload, spawned in a fixed order, so a (workload, seed) pair always yields
the same bytes.

Workloads (sizes follow the scheduler's evaluation scales):

* ``tiny``   D=4 decoders x 64 residents, H=4,096, 32 candidates, n=1,000.
* ``d16``    D=16 x 512, H=16,384, 1,024 candidates, n=10,000.
* ``d64``    D=64 x 2,048 heterogeneous capacities, H=32,768, 8,192
             candidates, n=100,000, alpha in {0.05, 0.1, 0.2}, Pareto outputs.
* ``stream`` 1,000,000 Poisson(+burst) arrivals for the streaming loop, D=32.
* ``large``  D=256 x 4,096 (1,048,576 residents), H=65,536, 65,536
             candidates, n=1,000,000, bimodal log-normal outputs.
"""
from __future__ import annotations

import numpy as np

MAX_WAIT_STEPS = 1000  # 1 s at 1 ms per decode step (Sec. 4 setup, App. A t_tok)

WORKLOADS = {
    "tiny": dict(index=0, D=4, R_per=64, H=4096, J=32, n_cal=1000,
                 alphas_ppm=(100000,), caps=(65536,), prompt=(32, 2048),
                 out="lognormal", out_params=(5.5, 1.0), clip=8192, sigma=0.4,
                 feasible_factor=2),
    "d16": dict(index=1, D=16, R_per=512, H=16384, J=1024, n_cal=10000,
                alphas_ppm=(100000,), caps=(262144,), prompt=(32, 2048),
                out="lognormal", out_params=(5.5, 1.0), clip=16384, sigma=0.4,
                feasible_factor=4),
    "d64": dict(index=2, D=64, R_per=2048, H=32768, J=8192, n_cal=100000,
                alphas_ppm=(50000, 100000, 200000),
                caps=(131072, 262144, 524288), prompt=(32, 2048),
                out="pareto", out_params=(1.5, 16.0), clip=32768, sigma=0.6,
                feasible_factor=16),
    "stream": dict(index=3, D=32, n_requests=1_000_000, batch=256,
                   cap=262144, H=16384, window=500, alpha_ppm=100000,
                   rate=200.0, burst_prob=0.1, burst_mult=5.0,
                   prompt=(32, 2048), out="lognormal", out_params=(5.5, 1.0),
                   clip=8192, sigma=0.4, pred_delay=(30.0, 0.25, 0.5), beta=1000),
    # App. A simulation setup: N decoders of C tokens, t_tok = 1 ms, theta =
    # 0.85, 10,000 requests; the trace's empirical length bins are not
    # available, tiny's prompt and output distributions stand in for them
    "rr": dict(index=5, N=4, C=50000, t_tok_us=1000, theta_ppm=850000, n_req=10000,
               prompt=(32, 2048), out="lognormal", out_params=(5.5, 1.0), clip=8192,
               rhos=(0.80, 0.90, 0.96, 1.00, 1.05, 1.10)),
    "large": dict(index=4, D=256, R_per=4096, H=65536, J=65536, n_cal=1000000,
                  alphas_ppm=(100000,), caps=(524288,), prompt=(64, 8192),
                  out="bimodal", out_params=(0.7, 4.5, 0.8, 7.5, 0.7),
                  clip=65536, sigma=0.5, feasible_factor=64),
}

DESCRIPTIONS = {
    "tiny": "Tiny: D=4 decoders x 64 residents, capacity 65,536, H=4,096, "
            "32 candidates, calibration n=1,000, alpha=0.1",
    "d16": "D16: D=16 x 512 residents, capacity 262,144, H=16,384, "
           "1,024 candidates, n=10,000, alpha=0.1",
    "d64": "D64 heterogeneous: D=64 x 2,048 residents, capacities "
           "{131,072; 262,144; 524,288}, H=32,768, 8,192 candidates, "
           "n=100,000, alpha in {0.05,0.1,0.2}",
    "stream": "Streaming loop: 1,000,000 Poisson(200/s)+burst arrivals in "
              "batches of 256 to D=32 decoders of capacity 262,144, H=16,384",
    "large": "Large: D=256 x 4,096 residents (1,048,576), capacity 524,288, "
             "H=65,536, 65,536 candidates, n=1,000,000, alpha=0.1",
}


def _lengths(rng: np.random.Generator, cfg: dict, size: int) -> np.ndarray:
    """True output lengths, rounded half-to-even and clipped to [1, clip]."""
    kind = cfg["out"]
    if kind == "lognormal":
        mu, sig = cfg["out_params"]
        x = rng.lognormal(mu, sig, size)
    elif kind == "pareto":
        shape, lo = cfg["out_params"]
        x = lo * (1.0 + rng.pareto(shape, size))
    elif kind == "bimodal":
        w, mu1, s1, mu2, s2 = cfg["out_params"]
        pick = rng.random(size) < w
        x = np.where(pick, rng.lognormal(mu1, s1, size),
                     rng.lognormal(mu2, s2, size))
    else:  # pragma: no cover - registry is fixed above
        raise ValueError(kind)
    return np.clip(np.rint(x), 1, cfg["clip"]).astype(np.int32)


def _predict(rng: np.random.Generator, cfg: dict, true: np.ndarray) -> np.ndarray:
    """Noisy length prediction: log-space Gaussian noise, clipped to [1, clip]."""
    noise = rng.normal(0.0, cfg["sigma"], true.shape[0])
    x = np.exp(np.log(true.astype(np.float64)) + noise)
    return np.clip(np.rint(x), 1, cfg["clip"]).astype(np.int32)


def _prompts(rng: np.random.Generator, cfg: dict, size: int) -> np.ndarray:
    lo, hi = cfg["prompt"]
    return rng.integers(lo, hi + 1, size=size, dtype=np.int64).astype(np.int32)


def make(name: str, seed: int | None = None, feasible: bool = False) -> dict:
    """Draw one snapshot workload (everything but ``stream``).

    Returns a dict of numpy arrays plus scalar sizes.  ``feasible=True``
    multiplies every capacity by the workload's ``feasible_factor`` so that
    both the feasible and the fallback branch of the dispatch rule occur; the
    other arrays are identical to the ``feasible=False`` draw.
    """
    cfg = WORKLOADS[name]
    if name == "stream":
        raise ValueError("use make_stream() for the streaming workload")
    D, R_per, J, n = cfg["D"], cfg["R_per"], cfg["J"], cfg["n_cal"]
    R = D * R_per
    ss = np.random.SeedSequence(cfg["index"] if seed is None else seed)
    (s_cap, s_q, s_rp, s_rt, s_rn, s_rg, s_rw, s_cp, s_ct, s_cn,
     s_lt, s_ln) = [np.random.default_rng(c) for c in ss.spawn(12)]

    caps = np.asarray(cfg["caps"], dtype=np.int64)
    cap = caps[s_cap.integers(0, len(caps), size=D)]
    if feasible:
        cap = cap * cfg["feasible_factor"]
    cap = cap.astype(np.int32)
    Q = s_q.integers(0, R_per // 4 + 1, size=D, dtype=np.int64).astype(np.int32)

    res_off = (np.arange(D + 1, dtype=np.int64) * R_per)
    res_prompt = _prompts(s_rp, cfg, R)
    res_true = _lengths(s_rt, cfg, R)
    res_pred = _predict(s_rn, cfg, res_true)
    res_gen = s_rg.integers(0, res_true.astype(np.int64)).astype(np.int32)
    res_wait = s_rw.integers(0, 2 * MAX_WAIT_STEPS + 1, size=R,
                             dtype=np.int64).astype(np.int32)
    res_dec = np.repeat(np.arange(D, dtype=np.int32), R_per)

    cand_prompt = _prompts(s_cp, cfg, J)
    cand_true = _lengths(s_ct, cfg, J)
    cand_pred = _predict(s_cn, cfg, cand_true)

    cal_true = _lengths(s_lt, cfg, n)
    cal_pred = _predict(s_ln, cfg, cal_true)

    return dict(
        name=name, D=D, H=cfg["H"], J=J, R=R, n_cal=n,
        alphas_ppm=tuple(cfg["alphas_ppm"]), max_wait=MAX_WAIT_STEPS,
        cap=cap, Q=Q, res_off=res_off, res_prompt=res_prompt,
        res_gen=res_gen, res_pred=res_pred, res_true=res_true,
        res_wait=res_wait, res_dec=res_dec,
        cand_prompt=cand_prompt, cand_pred=cand_pred, cand_true=cand_true,
        cal_true=cal_true, cal_pred=cal_pred,
    )


def make_stream(seed: int | None = None, n_requests: int | None = None) -> dict:
    """Draw the streaming workload: arrivals (ms), prompts, true lengths, preds.

    Arrivals: every 1-second window is independently a burst window with
    probability ``burst_prob``; its Poisson rate is ``rate * burst_mult`` in a
    burst and ``rate`` otherwise; arrival instants are uniform inside the
    window.  ``arrival_ms`` is the integer millisecond (= decode step) of each
    arrival, non-decreasing in request index.
    """
    cfg = WORKLOADS["stream"]
    N = cfg["n_requests"] if n_requests is None else int(n_requests)
    ss = np.random.SeedSequence(cfg["index"] if seed is None else seed)
    s_b, s_n, s_t, s_p, s_l, s_e, s_d = [np.random.default_rng(c) for c in ss.spawn(7)]
    times = []
    total = 0
    w = 0
    while total < N:
        burst = s_b.random() < cfg["burst_prob"]
        lam = cfg["rate"] * (cfg["burst_mult"] if burst else 1.0)
        c = int(s_n.poisson(lam))
        t = np.sort(s_t.random(c)) + w
        times.append(t)
        total += c
        w += 1
    t = np.concatenate(times)[:N]
    arrival_ms = np.floor(t * 1000.0).astype(np.int64)
    prompt = _prompts(s_p, cfg, N)
    true = _lengths(s_l, cfg, N)
    pred = _predict(s_e, cfg, true)
    # prediction latency (steps from arrival until the bound is available):
    # grows with the prompt, tens of ms for short prompts to several hundred
    # for the longest (App. D), with a log-normal spread; a few percent pass
    # the 1 s timeout
    a, b_, sd = cfg["pred_delay"]
    delay = (a + b_ * prompt) * np.exp(s_d.normal(0.0, sd, N))
    pred_delay_ms = np.minimum(np.rint(delay), 60000).astype(np.int32)
    return dict(name="stream", N=N, D=cfg["D"], H=cfg["H"], cap=cfg["cap"],
                batch=cfg["batch"], window=cfg["window"],
                alpha_ppm=cfg["alpha_ppm"], max_wait=MAX_WAIT_STEPS,
                arrival_ms=arrival_ms, prompt=prompt, true=true, pred=pred,
                pred_delay_ms=pred_delay_ms, beta_ms=cfg["beta"])


def make_rr(n_seeds: int = 1, rhos=None, n_req: int | None = None, seed0: int = 0) -> dict:
    """Realisations of the round-robin KV-pressure simulation (App. A).

    Per seed one workload is drawn -- prompts, output lengths and a unit-rate
    Poisson arrival sequence -- and, as in App. A, only the load intensity
    varies across the utilisations rho: the arrival rate is
    lambda = rho * N / (mean output length * t_tok), and arrival times are the
    unit-rate arrival instants divided by lambda, in integer microseconds.
    Realisation r = seed * len(rhos) + rho index.  Returns arrays
    [n_real][n_req] (arrival_us int64, prompt and out_len int32) and the
    simulation constants.
    """
    cfg = WORKLOADS["rr"]
    rhos = tuple(cfg["rhos"] if rhos is None else rhos)
    n = cfg["n_req"] if n_req is None else int(n_req)
    arr, prm, out = [], [], []
    for sd in range(n_seeds):
        ss = np.random.SeedSequence([cfg["index"], seed0 + sd])
        s_p, s_o, s_a = [np.random.default_rng(c) for c in ss.spawn(3)]
        prompt = _prompts(s_p, cfg, n)
        out_len = _lengths(s_o, cfg, n)
        unit = np.cumsum(s_a.exponential(1.0, n))  # unit-rate arrival instants
        for rho in rhos:
            lam = rho * cfg["N"] / (float(out_len.mean()) * cfg["t_tok_us"] * 1e-6)
            arr.append(np.rint(unit * 1e6 / lam).astype(np.int64))
            prm.append(prompt)
            out.append(out_len)
    return dict(name="rr", N=cfg["N"], C=cfg["C"], t_tok_us=cfg["t_tok_us"],
                theta_ppm=cfg["theta_ppm"], n_req=n, rhos=rhos, n_seeds=n_seeds,
                arrival_us=np.stack(arr), prompt=np.stack(prm), out_len=np.stack(out))
