"""Offline choice of the fixed proposal budget from a device cost profile and
development traces, written from the paper (Section 3.3 "Device-profiled
configuration"; App. B, the per-position cost reduction R(K); App. D.2
"Fixed configurations and development splits": budgets ranked by pooled
throughput on development windows).

TEST INFRASTRUCTURE: only tests and the benchmark's checks import it; it
shares no code with the library's C++ (csrc/budget.cu).

Each trace (reference text, producer text) is replayed with the oracle's
candidate buffer: the producer's whole text is published before the first
call, the target commits the reference text, and a call with k candidates
costs cost[k], the profiled mean time of width K = k + 1.
"""
from oracle import candidates as C


def cost_reduction(mean_call_time):
    """R(K) = 100 (1 - V(K) / (K V(1))) for K = 1..len(mean_call_time),
    mean_call_time[K - 1] being the mean call time of width K."""
    v1 = mean_call_time[0]
    return [100.0 * (1.0 - v / (K * v1)) for K, v in enumerate(mean_call_time, start=1)]


def estimate(traces, cost, b, n_commit, window=8):
    """Pooled committed tokens per second of budget b, and the call count."""
    committed = 0
    time_us = 0.0
    n_calls = 0
    for ref, prod in traces:
        calls, comm = C.run_session(list(ref), list(prod), lambda i: len(prod), b=b,
                                    window=window, target_len=n_commit)
        committed += len(comm)
        time_us += sum(cost[k] for k, *_ in calls)
        n_calls += len(calls)
    return committed / (time_us * 1e-6), n_calls


def select(traces, cost, b_max, n_commit, window=8):
    """The budget in 0..b_max with the highest pooled estimate (the smallest
    on ties), and every estimate."""
    est = [estimate(traces, cost, b, n_commit, window) for b in range(b_max + 1)]
    rates = [r for r, _ in est]
    best = max(range(b_max + 1), key=lambda b: (rates[b], -b))
    return best, est
