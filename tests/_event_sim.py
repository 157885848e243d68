"""An event-driven stage simulator: a second, independent CPU formulation of
the 1F1B and Eager-1F1B pipelines used only to pin the oracle.

Instead of building the DAG of Sec. 4.1 and taking its longest path, this
simulates each stage as a worker with a queue.  A stage keeps at most W_s
micro-batches in flight (activations held): N-s+1 under 1F1B and 2(N-s)+1
under Eager 1F1B (1-based s, at most M); it runs a forward whenever it has
room and forwards remain, else a backward.  An op starts when its stage is
free and its input (activation from stage s-1, gradient from stage s+1) has
arrived; the gradient all-reduce of stage s starts when its last backward
ends.  The iteration ends when every all-reduce has ended.
"""


def stage_program(S, M, s, eager=False):
    """Op sequence of stage s (0-based) from the in-flight rule."""
    W = min(2 * (S - 1 - s) + 1 if eager else S - s, M)
    prog, in_flight, nf, nb = [], 0, 0, 0
    while nb < M:
        if nf < M and in_flight < W:
            prog.append(("F", nf))
            nf += 1
            in_flight += 1
        else:
            prog.append(("B", nb))
            nb += 1
            in_flight -= 1
    return prog


def simulate(S, M, F, B, pf, pb, d, eager=False):
    """F, B, d: per-stage times; pf[s]: activation transfer s->s+1;
    pb[s]: gradient transfer s+1->s.  Returns (T, fin_F, fin_B)."""
    progs = [stage_program(S, M, s, eager) for s in range(S)]
    pos = [0] * S
    free = [0] * S
    fin_F = [[None] * M for _ in range(S)]
    fin_B = [[None] * M for _ in range(S)]
    remaining = 2 * S * M
    while remaining:
        progressed = False
        for s in range(S):
            while pos[s] < len(progs[s]):
                kind, m = progs[s][pos[s]]
                if kind == "F":
                    if s == 0:
                        ready = 0
                    elif fin_F[s - 1][m] is None:
                        break
                    else:
                        ready = fin_F[s - 1][m] + pf[s - 1]
                    start = max(free[s], ready)
                    fin_F[s][m] = start + F[s]
                    free[s] = fin_F[s][m]
                else:
                    if s == S - 1:
                        ready = 0
                    elif fin_B[s + 1][m] is None:
                        break
                    else:
                        ready = fin_B[s + 1][m] + pb[s]
                    start = max(free[s], ready)
                    fin_B[s][m] = start + B[s]
                    free[s] = fin_B[s][m]
                pos[s] += 1
                remaining -= 1
                progressed = True
        if not progressed:
            raise RuntimeError("deadlock")
    T = max(fin_B[s][M - 1] + d[s] for s in range(S))
    return T, fin_F, fin_B
