"""Which row kernel the launchers should pick for a contiguous [T, V] batch
(row stride V, base address 16-byte aligned), as occ_last_kernel() names it:
the vector kernel when rows start on 16-byte boundaries, the peeled vector
kernel when they do not but a row holds at least 16 vectors, else the
element-load kernel; for K1, rows of up to 32 KB run one warp per row.  The
fused kernel and K2 run their tensor-memory tiers on aligned or peeled rows
(CTAs of 128 threads up to 64 KB rows, 256 up to 112 KB, 512 beyond) whose
head and 16 tensor-memory blocks (of NT vectors) lie in whole
rounds of the walk (4 blocks per round in the fused kernel, 3 with its
diagnostics, 8 in K2, 6 in K2's peeled 512-thread rows; heads of 9
blocks at 512 threads, none at 256, none / 8 blocks at 128)."""


def _tmem(kind, nvec, rb, diag, peel):
    nt = 128 if rb <= 64 * 1024 else 256 if rb <= 112 * 1024 else 512
    if kind == "fused":
        head, u = (9 if nt == 512 else 0), (3 if diag else 4)
    elif kind == "k2":
        head, u = {512: 9, 256: 0, 128: 8}[nt], (6 if peel and nt == 512 else 8)
    else:
        return False
    return nvec // (u * nt) * u >= head + 16


def expected_kernel(kind, V, elem_size, diag=True):
    vec = 16 // elem_size
    names = {"k1": ("k1_logprob_vec", "k1_logprob_scalar"),
             "k2": ("k2_loss_l2", "k2_loss_stream"),
             "fused": ("k2_fused_l2", "k2_fused_stream")}[kind]
    first = names[0]
    if kind == "k1" and (V // vec) * 16 <= 32 * 1024:  # K1 rows up to 32 KB: one warp each
        first = "k1_logprob_warp"
    rb = (V // vec) * 16
    if (V * elem_size) % 16 == 0:
        return first + ("/tmem" if _tmem(kind, V // vec, rb, diag, False) else "")
    if V < 16 * vec:
        return names[1]
    # peeled rows lose up to vec - 1 elements to their scalar lead
    return first + "/peel" + ("/tmem" if _tmem(kind, (V - vec + 1) // vec, rb, diag, True) else "")
