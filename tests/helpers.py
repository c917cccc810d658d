"""Test harness glue: torch tensors -> the raw numpy arrays the oracle reads."""

from workloads.rawio import dtype_tag, raw_numpy  # noqa: F401


def oracle_on_workload(wl, blocks=None, taus=None):
    """Run the float64 oracle on a workloads.Workload (host tensors)."""
    import oracle

    cfg = wl.cfg
    if cfg.weight_dtype == "nvfp4":
        w_raw, w_tag = (raw_numpy(wl.weight), raw_numpy(wl.weight_block_scale)), "nvfp4"
    else:
        w_raw, w_tag = raw_numpy(wl.weight), dtype_tag(wl.weight)
    return oracle.commit_step(
        raw_numpy(wl.hidden), dtype_tag(wl.hidden),
        w_raw, w_tag,
        None if wl.weight_scale is None else raw_numpy(wl.weight_scale),
        raw_numpy(wl.pos_masked), raw_numpy(wl.block_flags),
        cfg.n_seq, cfg.n_slots, cfg.block_len, wl.mask_token_id,
        wl.tau if taus is None else taus, blocks=blocks)
