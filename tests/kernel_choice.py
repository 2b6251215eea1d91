"""Which row kernel the launchers should pick for a contiguous [T, V] batch
(row stride V, base address 16-byte aligned), as occ_last_kernel() names it:
the vector kernel when rows start on 16-byte boundaries, the peeled vector
kernel when they do not but a row holds at least 16 vectors, else the
element-load kernel."""


def expected_kernel(kind, V, elem_size):
    vec = 16 // elem_size
    names = {"k1": ("k1_logprob_vec", "k1_logprob_scalar"),
             "k2": ("k2_loss_l2", "k2_loss_stream"),
             "fused": ("k2_fused_l2", "k2_fused_stream")}[kind]
    if (V * elem_size) % 16 == 0:
        return names[0]
    return names[0] + "/peel" if V >= 16 * vec else names[1]
