"""Child process of test_gpu_threads.py: several host threads call the library
at once, each on its own stream with its own buffers, starting together so
that their first calls (which fill the per-device caches) race.  Afterwards
the same work runs on one thread, one call after the other, and every
result must match bit for bit.  Prints "threads ok" on success."""
import os
import sys
import threading

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import paper_2607_19490_gb300 as cg  # noqa: E402
import seeded_inputs as SI  # noqa: E402

N_THREADS = 4
ROUNDS = 5


def config(t, r):
    return SI.shrink(SI.SEVEN_B, n_canaries=16, tokens=32, seed=100 + 10 * t + r,
                     config_id=7 * t + r)


def work(t, stream, out):
    """Generate, score (default and streaming kernels), control labels and
    rank ROUNDS configurations; keep every output on the host."""
    torch.cuda.set_device(0)
    with torch.cuda.stream(stream):
        for r in range(ROUNDS):
            cfg = config(t, r)
            S, N = cfg["n_shards"], cfg["n_canaries"]
            acts, refs, labels = cg.cg_generate_pipeline(cg.PipelineDesc.from_config(cfg))
            scores = cg.cg_drift_scores(acts, refs, S, N)
            stream_scores = cg.cg_drift_scores(acts, refs, S, N, algo=cg.DRIFT_STREAM)
            ctrl = cg.cg_make_control_labels(labels[None], seed=11 + r)
            true_rank = cg.cg_auroc(scores[0][None], labels[None])
            ctrl_rank = cg.cg_auroc(scores[0][None], ctrl)
            pooled = cg.cg_auroc_pooled(scores[0][None], labels[None])
            rnd = cg.cg_random_scores(5 + r, 3, N, S, config_id0=t)
            stream.synchronize()
            out.append({
                "acts": acts.view(torch.int16).cpu().numpy(), "refs": refs.cpu().numpy(),
                "labels": labels.cpu().numpy(), "scores": scores.cpu().numpy(),
                "stream_scores": stream_scores.cpu().numpy(), "ctrl": ctrl.cpu().numpy(),
                "u2": true_rank["u2"].cpu().numpy(), "auroc": true_rank["auroc"].cpu().numpy(),
                "ctrl_auroc": ctrl_rank["auroc"].cpu().numpy(),
                "pooled": pooled["auroc"].cpu().numpy(), "random": rnd.cpu().numpy()})


def main():
    torch.cuda.set_device(0)
    results = [[] for _ in range(N_THREADS)]
    errors = []
    start = threading.Barrier(N_THREADS)
    streams = [torch.cuda.Stream() for _ in range(N_THREADS)]

    def run(t):
        try:
            start.wait()
            work(t, streams[t], results[t])
        except Exception as exc:          # reported by the parent test
            errors.append(f"thread {t}: {type(exc).__name__}: {exc}")

    threads = [threading.Thread(target=run, args=(t,)) for t in range(N_THREADS)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    torch.cuda.synchronize()
    if errors:
        print("\n".join(errors))
        sys.exit(1)
    main_stream = torch.cuda.current_stream()
    for t in range(N_THREADS):
        ref = []
        work(t, main_stream, ref)
        for r in range(ROUNDS):
            for k, v in ref[r].items():
                got = results[t][r][k]
                if v.dtype.kind == "f":
                    same = np.array_equal(v.view(np.uint8), got.view(np.uint8))
                else:
                    same = np.array_equal(v, got)
                if not same:
                    print(f"thread {t} round {r}: {k} differs from the sequential run")
                    sys.exit(1)
    print("threads ok")


if __name__ == "__main__":
    main()
