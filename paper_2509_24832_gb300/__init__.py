"""GB300-native (sm_103a) fuzzy token matching for SemShareKV (arXiv 2509.24832).

The path: rotary position encoding of the embedding rows of a target and a reference prompt
(Sec. 3.3.1, Eq. 1), random-hyperplane LSH sign codes (Sec. 3.3, App. A.2), the Hamming
nearest reference token of every target token (Sec. 3.3), and the rearrangement of the
reference K/V cache into the target's order (Sec. 3.3, Sec. 3.3.2); before it, the retrieval of
the stored prompt to reuse by LSH-distance similarity (Sec. 3.2, App. A.3); after it, the
Key-Value deviation against the recomputed first layer and the high-deviation tokens (App. A.4,
Insight 1).

The compute lives in libsemshare.so (C ABI: include/semshare.h); this package is its thin
ctypes binding with the same names.  Build the library with `paper_2509_24832_gb300.build`."""
from ._native import (  # noqa: F401
    CHECKED,
    FLAG_CHECK,
    FLAG_INDEX,
    HD_PERCENT,
    FLAG_TIMEOUT,
    KERNEL_HAMMING_TC,
    KERNEL_HASH,
    KERNEL_HASH_2SM,
    KERNEL_SELFTEST,
    KVLayout,
    LIB_PATH,
    Prepared,
    MATCH_STATIC_MAX_TARGETS,
    RETAIN_MAX_LAYERS,
    RETRIEVE_MAX_CANDIDATES,
    SIMILARITY_MAX_DIST,
    SIMILARITY_THRESHOLD,
    Retrieval,
    SemshareError,
    check_flag,
    flag_status,
    hd_count,
    hash_workspace,
    kv_layout,
    load,
    new_err_flag,
    retain_counts,
    semshare_abi_version,
    semshare_check_selftest,
    semshare_checked_build,
    check_record,
    semshare_fetch_rows,
    semshare_fetch_workspace_size,
    semshare_gather_kv,
    semshare_gather_kv_retained,
    semshare_hash,
    semshare_hash_pair,
    semshare_hash_pair_workspace_size,
    semshare_hash_workspace_size,
    semshare_kv_deviation,
    semshare_match,
    semshare_match_static,
    semshare_match_tc,
    semshare_match_tc_selected,
    semshare_match_tc_selected_workspace_size,
    semshare_match_tc_workspace_size,
    semshare_match_workspace_size,
    semshare_retrieve,
    semshare_retrieve_workspace_size,
    semshare_rope_table,
    semshare_select_hd,
    status_string,
)
