"""Device limits of one GB300 (sm_103), as the CUDA runtime reports them, for host-only
tests of the lite space (no GPU needed)."""


def gb300_limits():
    import paper_2309_08978_gb300 as nj
    L = nj.nnjit_device_limits()
    L.sm_count = 152
    L.smem_per_sm = 233472            # 228 KB
    L.smem_per_block_optin = 232448   # 227 KB
    L.regs_per_sm = 65536
    L.max_threads_per_sm = 2048
    L.max_blocks_per_sm = 32
    L.tmem_cols_per_sm = 512
    L.l2_bytes = 132120576
    L.cc_major = 10
    L.cc_minor = 3
    return L
