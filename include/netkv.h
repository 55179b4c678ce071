/*
 * netkv.h -- C ABI of the NetKV decode-instance scoring library (sm_103a).
 *
 * NetKV (arXiv 2606.03910) places each prefilled request on the decode instance
 * that minimises a cost made of the KV-cache transfer time over the network
 * (Sec. III-D, Eq. 3 and Eq. 4), the prefix-cache locality (Sec. III-B, Eq. 2)
 * and the compute load (Sec. IV-A), by a per-request greedy over the decode pool
 * (Algorithm 1, Sec. V-A).  This library runs that scoring path on one GPU:
 *
 *   netkv_topology_create   the four-tier instance tree (Sec. III-A, III-E)
 *   netkv_oracle_build      network cost oracle C[s][p][d] from per-link utilisation
 *                           snapshots, and the per-instance level bottlenecks UB
 *                           (netkv_oracle_build_directed: per link and direction;
 *                           netkv_oracle_build_tiers: the paper's per-tier maps)
 *   netkv_cache_build       decode caches K_d as an inverted index (block hash -> the
 *                           decodes of a 64-decode group that cache it)
 *   netkv_prefix_match      block-level prefix hit M[r][d] (Sec. III-B)
 *   netkv_schedule_streams  the greedy of Algorithm 1 over independent streams
 *   netkv_schedule_streams_inflight  the same with self-contention (Eq. 4's n_inflight)
 *   netkv_schedule_streams_load      the same with the paper's queue/decode-step model
 *   netkv_schedule_streams_evolving  the same with LRU-managed caches that change with
 *                                    every dispatch (Sec. VI-B), set by netkv_lru_init
 *
 * Conventions for every call:
 *   - Pointers named d_* are device pointers owned by the caller; the library never
 *     frees them and keeps no reference after the call returns.  Other pointers are
 *     host pointers read during the call only.
 *   - Work is enqueued on `stream` (NULL = the legacy default stream) and runs
 *     asynchronously; the call returns once the work is enqueued.
 *   - The return value reports errors found on the host (bad sizes, NULL pointers,
 *     unaligned buffers, failed CUDA launches) before anything is enqueued, except
 *     NETKV_ECUDA, which may follow a partial enqueue.
 *   - Errors found while the kernels run are OR-ed into *d_status (a device int the
 *     caller zeroes once and reads after synchronising) as NETKV_DEV_* bits.  No kernel
 *     traps; a flagged kernel still completes, with the affected outputs defined as
 *     stated per call.
 *   - No global mutable state: calls on different streams and threads may overlap as
 *     long as they do not write the same buffers.  A topology handle is immutable
 *     after creation and may be shared.
 */
#ifndef NETKV_H
#define NETKV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* netkv_stream_t; /* identical to cudaStream_t */

typedef enum {
  NETKV_OK = 0,
  NETKV_EINVAL = 1, /* argument out of range, NULL where required, misaligned buffer */
  NETKV_ENOMEM = 2, /* host or device allocation for a topology handle failed */
  NETKV_ECUDA = 3,  /* a CUDA runtime call or kernel launch failed */
  NETKV_ELIMIT = 4  /* request count above the fixed capacity of netkv_prefix_match_static */
} netkv_status;

/* Bits OR-ed into *d_status by the kernels. */
#define NETKV_DEV_EDOMAIN 1 /* utilisation outside [0,1) or NaN; zero-length request;
                               hash value 0 in a chain or key list; M[r][d] > len/16 */
#define NETKV_DEV_EFULL 2   /* a hash table had no free slot, a probe ran the whole table,
                               or a cache index is inconsistent */
#define NETKV_DEV_ERANGE 4  /* a request, prefill rank or snapshot index out of range */

/* ------------------------------------------------------------------ topology
 * The cluster is a four-level tree (Sec. III-A): fanout[0] instances per node,
 * fanout[1] nodes per leaf (rack / ToR), fanout[2] leaves per pod, fanout[3] pods
 * under the spine.  Instances are numbered depth-first, pod-major: instance i sits
 * in node i/f0, leaf i/(f0 f1), pod i/(f0 f1 f2).  The locality tier tau(p,d) of a
 * pair is 0 (same node), 1 (same leaf), 2 (same pod) or 3 (Sec. III-A).
 *
 * Links (the entries of a utilisation snapshot) are numbered in blocks by level:
 *   level 0  instance-node links  [0, N)                     link of instance i = i
 *   level 1  node-leaf links      [N, N + N/f0)              link of node n = N + n
 *   level 2  leaf-pod links       next N/(f0 f1)             by leaf
 *   level 3  pod-spine links      next f3                    by pod
 * The path between p and d uses the links of levels 0..tau(p,d) above p and above d.
 * A snapshot row holds n_links >= used links floats; entries past the used links are
 * padding and are never read.
 *
 * Prefill ranks number the instances with role 0 in instance order, decode ranks the
 * instances with role 1; every other argument indexes instances by these ranks.
 */
typedef struct netkv_topology* netkv_topology_t;

typedef struct {
  uint32_t fanout[4];     /* instances/node, nodes/leaf, leaves/pod, pods; each >= 1 */
  const uint8_t* role;    /* host [N], N = product of fanouts: 0 prefill, 1 decode */
  double tier_bw_Bps[4];  /* B_k: bandwidth of a level-k link, bytes/s, > 0 (Sec. III-A) */
  double tier_lat_s[4];   /* L_k: base latency of a tier-k transfer, seconds, >= 0 */
  uint32_t n_links;       /* utilisation row length (>= used links) */
} netkv_topology_desc;

/* Validates desc, builds the instance tables and copies them to the current device.
 * N must be below 2^31 and P, D >= 1.  Synchronous; allocates the handle and its
 * device mirror (freed by netkv_topology_destroy). */
netkv_status netkv_topology_create(const netkv_topology_desc* desc, netkv_topology_t* out);
netkv_status netkv_topology_destroy(netkv_topology_t topo);
/* Any output pointer may be NULL. */
netkv_status netkv_topology_query(netkv_topology_t topo, uint32_t* n_instances, uint32_t* P,
                                  uint32_t* D, uint32_t* used_links);

/* ------------------------------------------------------------------ oracle
 * Network cost oracle (Sec. III-D, Sec. III-E) with per-link congestion: for snapshot
 * s, prefill rank p and decode rank d,
 *     Bbot(s,p,d) = min over links e on the path of  B_level(e) * (1 - u[s][e])
 *     C[s][p][d]  = kv_bytes / Bbot(s,p,d) + L_tau(p,d)
 * i.e. Eq. 3 with Eq. 4's residual bandwidth taken at the bottleneck link and the
 * self-contention count at zero.  fp32 arithmetic; C is correctly-rounded division
 * of fp32 operands followed by an fp32 add.
 *
 *   d_util  [n_snap][n_links] fp32 utilisations in [0,1)
 *   d_C     [n_snap][P][D] fp32 output, row-major (d fastest), or NULL
 *   d_UB    [n_snap][N][4] fp32 output, or NULL: the level bottlenecks
 *           UB[s][i][k] = min over h <= k of B_h * (1 - u[s][link of i at level h]),
 *           so that Bbot(s,p,d) = min(UB[s][p][tau], UB[s][d][tau]) (instances by index)
 *   d_status device int, see NETKV_DEV_*.  Utilisations outside [0,1) set EDOMAIN and
 *           the affected outputs are whatever the formula gives.
 * At least one of d_C, d_UB must be non-NULL.  kv_bytes > 0.
 */
netkv_status netkv_oracle_build(netkv_topology_t topo, const float* d_util, uint32_t n_snap,
                                double kv_bytes, float* d_C, float* d_UB, int* d_status,
                                netkv_stream_t stream);

/* The same with directed links (the per-link generalisation of Eq. 4's c_tau, one
 * utilisation per link and direction): a transfer from prefill p to decode d climbs p's
 * links at their upward utilisation and descends d's at their downward utilisation,
 *     C[s][p][d] = kv_bytes / min(UB[s][p][tau], UB[s][d][tau]) + L_tau
 * with UB of a prefill instance computed from d_util_up and of a decode instance from
 * d_util_down (both [n_snap][n_links], same layout and domain as d_util above).  UB
 * keeps its layout, so netkv_schedule_streams consumes it unchanged.  With equal rows
 * the results are those of netkv_oracle_build.
 */
netkv_status netkv_oracle_build_directed(netkv_topology_t topo, const float* d_util_up,
                                         const float* d_util_down, uint32_t n_snap,
                                         double kv_bytes, float* d_C, float* d_UB,
                                         int* d_status, netkv_stream_t stream);

/* The paper-literal per-tier oracle (Sec. III-E: the tier, bandwidth, congestion and
 * latency maps; Eq. 4 with n_inflight = 0): d_c is [n_snap][4] per-tier congestion
 * c_tau in [0, 1), and a pair's bandwidth is B_tau * (1 - c_tau) with no minimum over the
 * lower levels of its path:
 *     C[s][p][d] = kv_bytes / (B_tau (1 - c[s][tau])) + L_tau
 * UB[s][i][k] = B_k (1 - c[s][k]) for every instance, so that netkv_schedule_streams
 * scores with the same maps.  Other arguments and errors as netkv_oracle_build.
 */
netkv_status netkv_oracle_build_tiers(netkv_topology_t topo, const float* d_c, uint32_t n_snap,
                                      double kv_bytes, float* d_C, float* d_UB, int* d_status,
                                      netkv_stream_t stream);

/* ------------------------------------------------------------------ caches
 * Decode caches K_d (Sec. III-C), the sets of block hashes each decode instance holds.
 * Decodes are taken in groups of 64 (decode ranks 64q .. 64q+63 form group q); each
 * (table set g, group q) has one index, index number g * G + q with G = ceil(D / 64), of
 * 2^log2_capacity hash slots, then 2^log2_capacity run keys, then 2^log2_capacity run
 * masks, padded to a multiple of 256 bytes:
 *   run keys     uint64: the group's distinct cached hashes in list order (decode by
 *                decode, first appearance);
 *   run masks    W bytes each, W = 1, 2, 4 or 8 for D <= 8, <= 16, <= 32 or more: bit
 *                (d mod 64) says that decode d caches the run key at that position;
 *   hash slots   {uint64 hash, uint64 run position}, open addressing with linear probing
 *                from a multiplicative hash; hash 0 marks an empty slot (block hash 0 is
 *                reserved).
 * Lists that give each cached prefix in chain order (as caches are filled) let the match
 * follow runs instead of probing block by block; any order gives the same results.
 * Keep the group's distinct hashes below about half of 2^log2_capacity.
 *
 *   d_index    device buffer of netkv_cache_index_bytes(n_sets, D, log2_capacity) bytes,
 *              16-byte aligned; cleared, then filled by netkv_cache_build
 *   d_keys     keys of (set g, decode d), list t = g * D + d, are
 *              d_keys[d_key_off[t] .. d_key_off[t+1])
 *   d_key_off  [n_sets * D + 1] uint64, non-decreasing
 * Duplicate keys are stored once.  A zero key sets EDOMAIN and is skipped; an index with
 * more distinct keys than slots sets EFULL (the excess keys are dropped).
 * 1 <= log2_capacity <= 31.
 */
size_t netkv_cache_index_bytes(uint32_t n_sets, uint32_t D, uint32_t log2_capacity);
netkv_status netkv_cache_build(void* d_index, uint32_t n_sets, uint32_t D,
                               uint32_t log2_capacity, const uint64_t* d_keys,
                               const uint64_t* d_key_off, int* d_status, netkv_stream_t stream);

/* ------------------------------------------------------------------ prefix match
 * Block-level prefix hit (Sec. III-B): M[r][d] = number of leading blocks of request
 * r's block-hash chain that are all present in decode d's cache; the cache hit in
 * tokens is lambda = 16 * M (B_tok = 16).  The scan stops at the first missing block.
 *
 *   d_index      cache index built by netkv_cache_build (same n_sets, D, log2_capacity)
 *   d_chains     uint64 block hashes; chain r = d_chains[d_chain_off[r] .. d_chain_off[r+1])
 *   d_chain_off  [R+1] uint64; every chain has at most 65535 blocks
 *   d_set_off    [n_sets+1] uint32 request offsets: table set g serves requests
 *                [d_set_off[g], d_set_off[g+1]); may be NULL when n_sets == 1
 *   d_workspace  NULL, or a device buffer of at least
 *                netkv_prefix_match_workspace_size(R) bytes, 256-byte aligned, owned by
 *                the caller and overwritten by the call.  With a workspace, requests are
 *                grouped by (table set, first block hash); each group's longest chain is
 *                matched in full and the others reuse its answers over their common
 *                prefix (exactly: the result is identical to the NULL-workspace call).
 *                Calls that overlap on the GPU need distinct workspaces.
 *   d_M          [R][D] uint16 output
 * A zero hash in a chain sets EDOMAIN and counts as a miss.  A chain longer than 65535
 * blocks sets EDOMAIN and its M saturates at 65535.  R < 2^31.
 */
size_t netkv_prefix_match_workspace_size(uint32_t R);
netkv_status netkv_prefix_match(const void* d_index, uint32_t D, uint32_t log2_capacity,
                                uint32_t n_sets, const uint64_t* d_chains,
                                const uint64_t* d_chain_off, uint32_t R,
                                const uint32_t* d_set_off, void* d_workspace,
                                size_t workspace_bytes, uint16_t* d_M, int* d_status,
                                netkv_stream_t stream);

/* Prefix match without allocation.  The paper has no counterpart: this entry point
 * serves callers that cannot allocate device memory at scoring time, for example a
 * scheduler plugin that runs inside a serving engine whose memory pool owns the whole
 * GPU, or code that must not call cudaMalloc on its request path.  It computes exactly
 * what netkv_prefix_match computes with a workspace, using instead a fixed 32 MiB
 * device array compiled into the library (every GPU that loads the library keeps it
 * until the process exits).
 *   - Arguments are those of netkv_prefix_match without the workspace.
 *   - R above NETKV_PREFIX_MATCH_STATIC_MAX_R returns NETKV_ELIMIT and enqueues nothing.
 *   - Every call made outside a stream capture looks up the array's device address
 *     with the device current (so a device reset, which may move the array, is
 *     followed); a call inside a capture uses the last address looked up on that
 *     device.  Make the first call on a device before any stream capture.
 *   - Allocates nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 *     The array is cleared where it must start at zero on every call.
 *   - All calls on a device share the one array: calls that overlap on the GPU (on
 *     different streams, or from several threads) race and must be serialised by the
 *     caller.
 */
#define NETKV_PREFIX_MATCH_STATIC_MAX_R 524288u
netkv_status netkv_prefix_match_static(const void* d_index, uint32_t D,
                                       uint32_t log2_capacity, uint32_t n_sets,
                                       const uint64_t* d_chains, const uint64_t* d_chain_off,
                                       uint32_t R, const uint32_t* d_set_off, uint16_t* d_M,
                                       int* d_status, netkv_stream_t stream);

/* ------------------------------------------------------------------ greedy
 * Per-stream weights and constants (device memory, one per stream).  Layout is fixed:
 * 4 floats, then two 8-byte integers (32 bytes).
 */
typedef struct {
  float w_net;             /* weight of the transfer time T_xfer, 1/s */
  float w_prefix;          /* weight of the missed fraction (l - lambda)/l */
  float w_load;            /* weight of the load term theta * load[d] */
  float theta_s_per_token; /* seconds of queueing per active token on a decode */
  int64_t cap_tokens;      /* capacity: d is feasible iff load[d] + l <= cap (Sec. IV-A) */
  uint64_t bytes_per_token;/* KV bytes per token per GPU pair (Eq. 1 / TP) */
} netkv_weights;

/* Algorithm 1 (Sec. V-A) over n_streams independent streams, each a sequence of
 * events processed in order.  For an arrival of request r (prefill rank p_r, length
 * l_r tokens, telemetry snapshot k_r), every decode rank d gets
 *     s_eff  = (l_r - 16 M[r][d]) * bytes_per_token                (Eq. 2, exact integer)
 *     T_xfer = s_eff / min(UB[k_r][p][tau], UB[k_r][d][tau]) + L_tau  (Eq. 3, Eq. 4)
 *     miss   = (l_r - 16 M[r][d]) / l_r
 *     score  = w_net * T_xfer + w_prefix * miss + w_load * (theta * load[d])
 * over the feasible set load[d] + l_r <= cap (line 1); the request goes to the feasible
 * d of minimum score, the lowest d among equal scores (line 13), or is rejected (-1)
 * when nothing is feasible (line 2); then load[d*] += l_r.  A departure event of a
 * dispatched request subtracts its l from the decode that took it.
 *
 *   d_w          [n_streams] netkv_weights
 *   d_len        [R] request length in tokens (>= 1)
 *   d_prefill    [R] prefill rank of the request (< P)
 *   d_snap       [R] snapshot index (< n_snap) into d_UB
 *   d_M          [R][D] prefix hits from netkv_prefix_match
 *   d_UB         [n_snap][N][4] level bottlenecks from netkv_oracle_build
 *   d_events     uint32 codes: bit 31 set = departure, bits 0..30 = request index r;
 *                stream j's events are d_events[d_event_off[j] .. d_event_off[j+1])
 *   d_event_off  [n_streams+1] uint64
 *   d_load_init  [n_streams][D] int64 initial loads, or NULL for zero (resume support)
 *   d_dec        [R] int32 output: decision of each arrival handled (others untouched)
 *   d_best       [R] fp32 output: minimum score (+inf when rejected)
 *   d_second     [R] fp32 output: minimum over the other feasible candidates (+inf if none)
 *   d_load_final [n_streams][D] int64 output: loads after the last event
 *   d_workspace  NULL, or a device buffer, 256-byte aligned, owned by the caller and
 *                overwritten by the call, of at least R * D * 4 bytes rounded up to 256.
 *                With a workspace the decision-independent part of every arrival's scores
 *                (w_net * T_xfer + w_prefix * miss) is computed first for all arrivals in
 *                parallel and the sequential walk only adds the load term; without one
 *                the walk computes every term itself.  For pools of 1,025 .. 4,096 decodes
 *                a workspace of netkv_schedule_workspace_size(R, D) bytes also holds, per
 *                arrival, the pool's 32 smallest (base score, rank) pairs and a bound on
 *                the rest: the walk then rescores only those and falls
 *                back to the arrival's full row when the bound does not certify the argmin
 *                (the same decisions and scores, bit for bit).  A workspace of only the
 *                rows runs the walk over every candidate.  Overlapping calls need distinct
 *                workspaces.
 * Every request index must occur in at most one stream, and its departure after its
 * arrival.  Out-of-range indices set ERANGE and the event is skipped.  The topology
 * may have at most 4096 decode instances.
 */
size_t netkv_schedule_workspace_size(uint32_t R, uint32_t D);
netkv_status netkv_schedule_streams(netkv_topology_t topo, uint32_t n_streams,
                                    const netkv_weights* d_w, uint32_t R, const uint32_t* d_len,
                                    const uint32_t* d_prefill, const uint32_t* d_snap,
                                    const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
                                    const uint32_t* d_events, const uint64_t* d_event_off,
                                    const int64_t* d_load_init, int32_t* d_dec, float* d_best,
                                    float* d_second, int64_t* d_load_final, void* d_workspace,
                                    size_t workspace_bytes, int* d_status, netkv_stream_t stream);

/* netkv_schedule_streams with the level bottlenecks taken from the telemetry itself: d_util
 * [n_snap][n_links] fp32 utilisation rows (as for netkv_oracle_build) replace d_UB, and the
 * base-score pass computes each candidate's min(UB[k][p][tau], UB[k][d][tau]) from the
 * utilisations of the links of p and d in row k, with the arithmetic of netkv_oracle_build.
 * So the results equal those of netkv_oracle_build(d_UB) followed by
 * netkv_schedule_streams with a workspace, without writing UB.  The workspace is required
 * (EINVAL when NULL or smaller than R * D * 4 bytes rounded up to 256; the candidate lists
 * need netkv_schedule_workspace_size(R, D), as for netkv_schedule_streams); other arguments
 * and errors as netkv_schedule_streams, plus EDOMAIN for a utilisation outside [0, 1). */
netkv_status netkv_schedule_streams_util(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const uint16_t* d_M,
    const float* d_util, uint32_t n_snap, const uint32_t* d_events, const uint64_t* d_event_off,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int64_t* d_load_final, void* d_workspace, size_t workspace_bytes, int* d_status,
    netkv_stream_t stream);

/* Algorithm 1 with self-contention (Eq. 4's n_inflight term, Algorithm 1 lines 5 and 14,
 * Sec. V-C).  As netkv_schedule_streams without a workspace, and in addition each
 * stream keeps a counter n[p][tau] per prefill rank and tier (zero at the start of the
 * call) of its own transfers in flight:
 *     B_eff  = min(UB[k_r][p][tau], UB[k_r][d][tau]) / (1 + n[p_r][tau])  (Eq. 4)
 *     T_xfer = s_eff / B_eff + L_tau                                     (Eq. 3)
 * A dispatch to d* raises n[p_r][tau(p_r, d*)] by one unless it is already at
 * inflight_cap, and its transfer completes at arrival_us[r] + xfer_us[r], where
 * xfer_us[r] is its T_xfer rounded to whole microseconds; a completion lowers the
 * counter by one unless it is zero.  Completions due at or before an arrival's time
 * are applied before that arrival is scored.  inflight_cap = 0 keeps every counter at
 * zero: the result is then that of netkv_schedule_streams (without a workspace when
 * d_workspace is NULL).
 *
 *   d_arrival_us [R] int64 arrival time of each request in microseconds; a stream's
 *                arrivals must be in time order, as its events are
 *   inflight_cap 0 .. 255 (the paper's default is 16)
 *   d_xfer_us    [R] int32 output: T_xfer of the chosen candidate in whole microseconds
 *                (at most 2^31 - 1), -1 for a rejected arrival
 *   d_workspace  NULL, or at least netkv_schedule_inflight_workspace_size(R, D) bytes,
 *                256-byte aligned: the decision-independent score part and s_eff / Bbot of
 *                every (arrival, decode) are then computed first in parallel, and the walk
 *                adds w_net * (s_eff / Bbot) * n and the load term; with inflight_cap = 0
 *                the result is then netkv_schedule_streams' with a workspace.
 * Other arguments as for netkv_schedule_streams.  Limits: fewer than 16,384 prefill
 * ranks; the counters (4 bytes per prefill rank) and the pending completions of a
 * stream live in shared memory, 4,096 pending completions per stream for pools of more
 * than 16 decodes and 256 for smaller ones (packed several streams to a warp); a
 * completion that does not fit sets EFULL and is dropped (its counter is not lowered).
 * Host errors: EINVAL for a cap above 255, too many prefill ranks or missing buffers.
 */
size_t netkv_schedule_inflight_workspace_size(uint32_t R, uint32_t D);
netkv_status netkv_schedule_streams_inflight(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap,
    const int64_t* d_arrival_us, const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
    const uint32_t* d_events, const uint64_t* d_event_off, uint32_t inflight_cap,
    const int64_t* d_load_init, int32_t* d_dec, float* d_best, float* d_second,
    int32_t* d_xfer_us, int64_t* d_load_final, void* d_workspace, size_t workspace_bytes,
    int* d_status, netkv_stream_t stream);

/* The paper's compute-load model (Sec. III-C decode state, Sec. IV-B component models). */
typedef struct {
  float t_a_s, t_b_s;     /* iteration time t_iter(beta) = t_a + t_b * beta, seconds (>= 0) */
  int32_t beta_max;       /* batch slots per decode (the paper uses 64), >= 1 */
  int32_t reserved;       /* set to 0 */
  int64_t m_min_bytes;    /* memory each decode holds back (>= 0) */
  int64_t m0_bytes;       /* free memory of every decode at the start when d_m_init is NULL */
} netkv_load_model;       /* 32 bytes */

/* Algorithm 1 with the paper's compute-load model instead of the token load.  Decode d
 * holds n_d requests (dispatched, not departed) and m_d free bytes; with the batch
 * beta = min(n_d, beta_max) and the queue q = n_d - beta,
 *     T_queue  = max(0, q - (beta_max - beta)) * t_iter(beta)         (Sec. IV-B)
 *     T_decode = t_iter(beta + 1)
 *     score    = w_net * T_xfer + w_prefix * miss + w_load * (T_queue + T_decode)
 * over the feasible set m_d >= s_eff(d) + m_min (the objective's feasible set, Sec. IV-A),
 * s_eff exact in bytes.  A dispatch to d* adds one request to it and takes s_eff(d*)
 * bytes; the request's departure gives both back.  T_xfer and miss as in
 * netkv_schedule_streams (without a workspace); the weights' theta and cap_tokens are
 * not used.
 *
 *   model      host pointer to the model's constants
 *   d_m_init   [n_streams][D] int64 free bytes at the start, or NULL for m0_bytes
 *   d_n_init   [n_streams][D] int32 requests held at the start, or NULL for 0
 *   d_m_final  [n_streams][D] int64 output: free bytes after the last event
 *   d_n_final  [n_streams][D] int32 output: requests held after the last event
 * Other arguments and errors as netkv_schedule_streams; EINVAL for a missing model,
 * beta_max < 1 or negative constants.
 */
netkv_status netkv_schedule_streams_load(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w,
    const netkv_load_model* model, uint32_t R, const uint32_t* d_len, const uint32_t* d_prefill,
    const uint32_t* d_snap, const uint16_t* d_M, const float* d_UB, uint32_t n_snap,
    const uint32_t* d_events, const uint64_t* d_event_off, const int64_t* d_m_init,
    const int32_t* d_n_init, int32_t* d_dec, float* d_best, float* d_second, int64_t* d_m_final,
    int32_t* d_n_final, int* d_status, netkv_stream_t stream);

/* ------------------------------------------------------------------ evolving caches
 * The decode caches of the simulator of Sec. VI-B, LRU-managed KV-block caches that change
 * with every dispatch.  Each (stream, decode) pair has its own cache, number
 * c = stream * D + d, holding at most cap_blocks block hashes in recency order:
 *   - netkv_lru_init sets every cache from a key list given from the most to the least
 *     recently used block;
 *   - in netkv_schedule_streams_evolving, a dispatch of request r to d* uses every block
 *     of r's chain on cache (stream, d*), from the last block to the first, so that
 *     block 0 becomes the most recently used one (a cached prefix loses its tail first);
 *     present blocks are refreshed, absent ones inserted, and then the least recently
 *     used blocks beyond cap_blocks are evicted.  Departures leave the caches unchanged.
 * The caches live in a caller-owned state buffer of netkv_lru_state_bytes(n_caches, cfg)
 * bytes (16-byte aligned) that the greedy updates in place, so a later call continues
 * from the caches an earlier call left.  Per cache it holds a hash table of
 * 2^log2_slots 16-byte slots and a recency log of 2^log2_ring 8-byte entries: 12 MiB for
 * 2^19 of each, enough for caches of 200,000 blocks.
 */
typedef struct {
  uint64_t cap_blocks; /* blocks a cache keeps (>= 1); the least recently used beyond go */
  uint32_t log2_slots; /* hash slots per cache: (3/4) 2^log2_slots >= cap_blocks + 65535 */
  uint32_t log2_ring;  /* recency-log entries per cache: 2^log2_ring >= cap_blocks + 65536 */
} netkv_lru_config;   /* 16 bytes */

/* Bytes of state for n_caches caches; 0 for an invalid configuration. */
size_t netkv_lru_state_bytes(uint64_t n_caches, const netkv_lru_config* cfg);

/* Sets caches [0, n_caches) of d_state (state_bytes bytes, at least
 * netkv_lru_state_bytes(n_caches, cfg)) from key lists: cache c holds
 * d_keys[d_key_off[c] .. d_key_off[c+1]), most recently used first (d_key_off has
 * n_caches + 1 uint64 entries).  d_keys = NULL sets every cache empty.  A list longer than
 * cap_blocks sets ERANGE and keeps its first cap_blocks entries; a zero key sets EDOMAIN
 * and is skipped; repeated keys count once, at their first (most recent) entry.
 * Host errors: EINVAL for a bad configuration or buffer. */
netkv_status netkv_lru_init(void* d_state, size_t state_bytes, uint64_t n_caches,
                            const netkv_lru_config* cfg, const uint64_t* d_keys,
                            const uint64_t* d_key_off, int* d_status, netkv_stream_t stream);

/* Every cache's blocks from the most to the least recently used:
 * d_keys_out [n_caches][cap_blocks] (cache c's list starts at c * cap_blocks) and
 * d_len_out [n_caches] its length.  Reads the state only. */
netkv_status netkv_lru_export(const void* d_state, size_t state_bytes, uint64_t n_caches,
                              const netkv_lru_config* cfg, uint64_t* d_keys_out,
                              uint64_t* d_len_out, int* d_status, netkv_stream_t stream);

/* Algorithm 1 (Sec. V-A) with evolving caches.  As netkv_schedule_streams without a
 * workspace (scores, feasibility, argmin, loads, departures), except that the prefix hits
 * are not an input: each arrival's hits on every decode are taken against the stream's
 * caches in d_state as they are at that arrival (the first-miss scan of Sec. III-B), and
 * a dispatch updates the chosen decode's cache as described above.
 *
 *   d_chains, d_chain_off  request chains as for netkv_prefix_match ([R+1] offsets;
 *                          a chain longer than 65535 blocks sets EDOMAIN and is cut)
 *   d_state                caches of n_streams * D decodes from netkv_lru_init (or an
 *                          earlier call), with the same cfg; updated in place
 *   state_bytes            size of d_state, at least netkv_lru_state_bytes(n_streams * D,
 *                          cfg) (EINVAL otherwise)
 *   d_M                    [R][D] uint16 output: the hits each arrival was scored with
 * Other arguments as netkv_schedule_streams.  A zero hash in a chain sets EDOMAIN, counts as
 * a miss and is not cached.  The decode pool may have at most 1024 instances.  Calls that
 * overlap on the GPU need distinct state buffers.
 */
netkv_status netkv_schedule_streams_evolving(
    netkv_topology_t topo, uint32_t n_streams, const netkv_weights* d_w, uint32_t R,
    const uint32_t* d_len, const uint32_t* d_prefill, const uint32_t* d_snap, const float* d_UB,
    uint32_t n_snap, const uint64_t* d_chains, const uint64_t* d_chain_off,
    const uint32_t* d_events, const uint64_t* d_event_off, void* d_state, size_t state_bytes,
    const netkv_lru_config* cfg, const int64_t* d_load_init, int32_t* d_dec, float* d_best,
    float* d_second, uint16_t* d_M, int64_t* d_load_final, int* d_status, netkv_stream_t stream);

/* ------------------------------------------------------------------ transfers
 * Asynchronous copy of `bytes` bytes by a kernel (SM loads and stores).  Either side may
 * be device memory or pinned host memory reachable through unified addressing (memory
 * from cudaHostAlloc / cudaMallocHost); on NVLink-C2C systems this moves a step's inputs
 * host->device faster than the copy engines.  Both pointers 16-byte aligned; the
 * regions must not overlap.  Used by the host-buffer step; not part of the paper's path.
 */
netkv_status netkv_copy_async(void* dst, const void* src, size_t bytes, netkv_stream_t stream);

/* Library version, for the bindings' load check. */
uint32_t netkv_version(void);

#ifdef __cplusplus
}
#endif
#endif /* NETKV_H */
