/*
 * gmgsim.h — C ABI of the GB300 what-if placement simulator.
 *
 * The library evaluates K candidate operator placements of one Global
 * Mapping Graph (GMG) by event-driven simulation, as the Global Simulator of
 * SliceScheduler does for each candidate partition of a scheduling round
 * (paper Sec. 3.3 "Global Simulator", Sec. 3.4 and Algorithm 1).  Every
 * candidate is simulated by one warp of a CUDA kernel compiled for sm_103a.
 *
 * Semantics (all integers; times in microseconds, sizes in bytes):
 *   xfer(d, e, b) = 0 if d == e, else ceil(b / bw[d][e]) + lat[d][e]
 *                                     (transfer estimator, Sec. 3.3.1)
 *   r_i = max(release_i, max over predecessors p of f_p + xfer(dev_p, dev_i, bytes_p))
 *                                     (ready time, Sec. 3.3.2)
 *   each accelerator runs one op at a time; an idle accelerator starts the
 *   ready op with the smallest (r_i, i); it is busy until avail0[d] first
 *                                     (queue rule, Sec. 3.3.2 / 3.5.1)
 *   s_i = start, f_i = s_i + dur_i    (event-driven simulation, Sec. 3.3.3)
 *   HBM: op i's output is allocated on dev_i at s_i; a receive copy on every
 *   other accelerator running a successor at f_i; a copy is freed at the
 *   latest finish of i's listed consumers on that accelerator, not before it
 *   arrived (source copy: not before all outgoing transfers arrived and i
 *   finished).  Frees before allocs at equal times.  A placement whose live
 *   bytes exceed an accelerator's capacity is infeasible (Sec. 3.3.2,
 *   Sec. 3.5.2, Sec. 3.4.2).
 *   score = sum of f_i over scored ops (INT64_MAX if infeasible); best =
 *   lexicographic argmin of (score, k) over feasible candidates (Algorithm 1).
 *
 * Ownership: the caller (e.g. PyTorch) allocates every device buffer and the
 * stream.  The library never allocates device memory; handles borrow the
 * workspaces given to them, which must outlive the handles.  Host pointers in
 * gmg_desc_t are read during gmg_create only.
 *
 * Errors: every int-returning call returns GMG_OK (0) or a negative GMG_E*
 * code and never aborts.  Per-candidate problems (bad device id, bad move
 * list, capacity of the event queue or the iteration cap) are written to
 * status[k]; such candidates are never selected.  Kernel launches are
 * asynchronous on the given stream; launch errors return GMG_ECUDA.
 *
 * Threading: a gmg_t / gmg_base_t is immutable after creation and may be
 * used from several streams at once; concurrent calls need their own scratch
 * and output buffers.
 */
#ifndef GMGSIM_H_
#define GMGSIM_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without including the CUDA headers. */
typedef struct CUstream_st* gmg_stream_t;

/* Return codes. */
#define GMG_OK 0
#define GMG_EINVAL (-1)   /* malformed argument or graph */
#define GMG_ENOTTOPO (-2) /* a predecessor id is not smaller than its op id */
#define GMG_ERANGE (-3)   /* times or byte totals could overflow the int64 / packed-key ranges */
#define GMG_EWS (-4)      /* workspace or scratch buffer too small or misaligned */
#define GMG_ECUDA (-5)    /* a CUDA runtime call failed */
#define GMG_ENOMEM (-6)   /* host allocation failed */

/* Per-candidate status codes (status[k]). */
#define GMG_SIM_OK 0
#define GMG_SIM_BADDEV 1     /* a placement entry is >= n_dev */
#define GMG_SIM_MOVE_RANGE 2 /* a move's op is outside [0, n_ops) or its device >= n_dev */
#define GMG_SIM_MOVE_DUP 3   /* an op appears twice in one move list */
#define GMG_SIM_BADBASE 4    /* the base placement of an incremental batch is invalid */
#define GMG_SIM_QUEUE 5      /* the per-candidate event queue overflowed (raise queue_cap) */
#define GMG_SIM_LOOP 6       /* the event loop exceeded its iteration cap */

/*
 * The GMG: a topologically numbered operator DAG (Sec. 3.2 "Graph structure")
 * with pre-evaluated integer estimates and the accelerator set.
 * Layout: plain host arrays; CSR lists are (offsets of length n_ops+1,
 * indices).  NULL for an optional array selects its default.
 */
typedef struct {
  int32_t n_ops;   /* N >= 0 */
  int32_t n_edges; /* E = pred_off[N] */
  int32_t n_dev;   /* D in [1, 256] */
  int32_t n_req;   /* R >= 0 */
  const int32_t* pred_off; /* [N+1] predecessors of op i: pred_idx[pred_off[i]..pred_off[i+1]) */
  const int32_t* pred_idx; /* [E] each < i (topological), no duplicates per op */
  const int32_t* cons_off; /* [N+1] optional: consumers whose completion releases op i's output */
  const int32_t* cons_idx; /* each a successor of i, no duplicates; NULL lists = all successors */
  const int64_t* dur_us;     /* [N] >= 1 (ignored, may be NULL, when n_types >= 2) */
  const int64_t* out_bytes;  /* [N] >= 0 */
  const int64_t* release_us; /* [N] >= 0, optional (0) */
  const int32_t* req_id;     /* [N] in [-1, R), optional (-1 = no request) */
  const uint8_t* scored;     /* [N] 0/1, optional (all 1) */
  const int64_t* deadline_us; /* [R] optional (INT64_MAX = none) */
  const int64_t* cap_bytes;   /* [D] >= 0, optional (INT64_MAX) */
  const int64_t* base_bytes;  /* [D] in [0, cap], optional (0): resident throughout */
  const int64_t* avail0_us;   /* [D] >= 0, optional (0): accelerator busy until then */
  const int64_t* bw_B_per_us; /* [D*D] row = source; >= 1 off the diagonal (diagonal ignored) */
  const int64_t* lat_us;      /* [D*D] >= 0 off the diagonal */
  /* Heterogeneous accelerators: the operator estimator of Sec. 3.3.1 keeps one
   * estimate per (accelerator type, operator), so an op's duration depends on
   * the type of the accelerator it is placed on.  n_types <= 1: one type, every
   * op takes dur_us[i] everywhere and the two arrays below are not read. */
  int32_t n_types;             /* T in [0, 256] */
  const uint8_t* dev_type;     /* [D] each < T */
  const int64_t* dur_by_type;  /* [N*T] row-major by op: dur of op i on type t at [i*T + t], >= 1 */
  /* Communication links, read only by arbitrated transfers (sim_opts_t.
   * transfer_mode): transfers over ordered pairs with the same id compete for
   * that link (Sec. 3.5.2).  Optional (NULL: every ordered pair has a link of
   * its own, so only the endpoints are shared).  Off-diagonal ids in
   * [0, D*D); the diagonal is ignored. */
  const int32_t* link_id;      /* [D*D] row = source */
} gmg_desc_t;

typedef struct gmg gmg_t;           /* opaque; host metadata + borrowed device workspace */
typedef struct gmg_base gmg_base_t; /* opaque; base schedule snapshot for incremental runs */

/* sim_opts_t.gmg_staging: where sim_batch's warps read the GMG's hot fields
 * (durations, transfer sizes, flags, releases, both CSR lists) when they start
 * ops and test successors.  GMG_STAGING_SHARED: each CTA (one per SM, up to 28
 * warps) first copies a compact 16-byte record per op, the releases and both
 * lists into shared memory with bulk copies; needs one accelerator type,
 * uniform links, every time below 2^31, at most 32 accelerators and the copy
 * within the CTA's shared memory, else GMG_EINVAL.  GMG_STAGING_L1: 4-warp
 * CTAs read the 64-byte op records through the read-only L1 path.
 * GMG_STAGING_DEFAULT stages wherever staging applies (measured faster on the
 * prefill workload) and takes the L1 path elsewhere; sim_batch_noalloc always
 * takes the L1 path (and refuses GMG_STAGING_SHARED). */
#define GMG_STAGING_DEFAULT 0
#define GMG_STAGING_SHARED 1
#define GMG_STAGING_L1 2

/* sim_opts_t.transfer_mode */
#define GMG_TRANSFER_LATENCY 0    /* a transfer starts when its producer finishes (Sec. 3.3.2) */
#define GMG_TRANSFER_ARBITRATED 1 /* transfers wait for the arbiter (Sec. 3.5.2); sim_batch only */

typedef struct {
  int32_t score_mode;       /* select_best: 0 = score, 1 = (sla_miss, score) */
  int32_t n_trace;          /* number of candidates whose per-op schedule is written */
  const int32_t* d_trace_k; /* device [n_trace]: candidate indices to trace (distinct) */
  int32_t queue_cap;        /* per-candidate event-queue entries; 0 = library default */
  int32_t warps_per_block;  /* 0 = library default (tuning knob) */
  int32_t transfer_mode;    /* GMG_TRANSFER_*; 0 = GMG_TRANSFER_LATENCY */
  int32_t gmg_staging;      /* GMG_STAGING_*; sim_batch with pure-latency transfers only */
  int32_t reserved[2];      /* must be 0 */
} sim_opts_t;

/* Caller-owned device output arrays for K candidates. */
typedef struct {
  int64_t* makespan;  /* [K] max f_i (0 for an empty graph) */
  int64_t* score;     /* [K] sum of f_i over scored ops; INT64_MAX if infeasible or status != 0 */
  int32_t* status;    /* [K] GMG_SIM_* */
  int32_t* viol_flag; /* [K] 1 if some live total exceeded the capacity */
  int32_t* viol_op;   /* [K] op of the first violating allocation, -1 if none */
  int32_t* viol_dev;  /* [K] its accelerator, -1 if none */
  int64_t* viol_time; /* [K] its time, -1 if none */
  int64_t* peak;      /* [K*D] per-accelerator peak live bytes (base included) */
  int32_t* sla_miss;  /* [K] requests whose completion is past their deadline */
  int64_t* events;    /* [K] operators simulated: N, or the re-simulated suffix for incremental */
  int64_t* req_done;  /* [K*R] optional (NULL): per-request completion time */
  int64_t* trace_start;  /* [n_trace*N] optional: start of every op of each traced candidate */
  int64_t* trace_finish; /* [n_trace*N] optional: finish of every op */
} sim_out_t;

/* Static information about a created GMG (for callers and tests). */
typedef struct {
  int32_t n_ops, n_edges, n_dev, n_req;
  int32_t n_roots;       /* ops without predecessors */
  int32_t id_bits;       /* bits of an op id in the packed event key */
  int32_t time_bits;     /* bits of a time in the packed event key */
  int32_t uniform_links; /* 1 if every off-diagonal link has the same bw and latency */
  int64_t time_bound;    /* proven upper bound of every simulated time */
  int64_t default_queue_cap;
  int32_t batched_sweep; /* 1 if the simulation kernels start READY ops in batches (graphs on
                            more than 32 accelerators whose keys have room for a duration class) */
  int32_t t32;           /* 1 if the kernels carry times as 32-bit integers (time_bound < 2^31) */
  int32_t stageable;     /* 1 if sim_batch can stage this graph's hot fields in shared memory on
                            the current device (one accelerator type, uniform links, 32-bit times,
                            at most 32 accelerators, and the copy fits beside one warp's areas);
                            the default then stages, with pure-latency transfers */
  int32_t reserved_;
} gmg_info_t;

/* ---------------------------------------------------------------------- */

/* Bytes of device workspace gmg_create needs for this description; 0 if the
 * description is too malformed to size (gmg_create then reports why). */
size_t gmg_workspace_bytes(const gmg_desc_t* desc);

/* Validate `desc` on the host, build the device layout (CSR, op records,
 * link tables, sorted roots) and copy it into d_ws (>= gmg_workspace_bytes,
 * 256-byte aligned) on `stream`; synchronizes the stream before returning.
 * Returns GMG_EINVAL / GMG_ENOTTOPO / GMG_ERANGE for invalid graphs,
 * GMG_EWS for a short workspace.  *out receives the handle. */
int gmg_create(const gmg_desc_t* desc, void* d_ws, size_t ws_bytes, gmg_stream_t stream,
               gmg_t** out);

/* Free the host metadata of a handle (the device workspace stays the caller's). */
void gmg_destroy(gmg_t* g);

int gmg_get_info(const gmg_t* g, gmg_info_t* info);

/* Bytes of device scratch sim_batch needs for K candidates with these
 * options (depends on the current device's SM count). */
size_t sim_scratch_bytes(const gmg_t* g, int32_t K, const sim_opts_t* opts);

/* Simulate K full placements (paper Sec. 3.3.3 for each candidate p of
 * Algorithm 1).  d_place: device uint8 [K][ld], row k = device of every op,
 * ld >= n_ops, ld % 16 == 0, 16-byte aligned.  Writes every field of *d_out
 * for every candidate.  d_scratch >= sim_scratch_bytes, 256-byte aligned.
 *
 * opts->transfer_mode = GMG_TRANSFER_ARBITRATED simulates the arbitrated
 * transfers of Sec. 3.5.2 ("Tensor Transfer Arbitration") instead of pure
 * latency: a producer's completion raises one transfer intent per distinct
 * remote accelerator of its successors; after every intent or transfer
 * completion at time t, the pending intents are visited in (intent time,
 * producer id, destination id) order and each one whose sending endpoint
 * (its source accelerator), receiving endpoint (its destination) and link
 * (gmg_desc_t.link_id) are free of every active transfer starts at t.  It
 * lasts the transfer estimate; its receive buffer is allocated when it
 * starts; the successors' input arrives when it completes.  The paper does
 * not fix the choice among conflicting intents: this FIFO-greedy order is
 * the library's.  Needs accelerator ids that fit the packed event key and
 * op ids < 2^27 (n_dev <= 32) or < 2^24 (33 to 256 accelerators), else
 * GMG_ERANGE.
 * base_create and base_workspace_bytes accept only GMG_TRANSFER_LATENCY
 * (GMG_EINVAL, or 0 bytes, otherwise).  sim_incremental with
 * GMG_TRANSFER_ARBITRATED takes such a base but uses only its placement and
 * status: every candidate's moved placement is simulated in full (events =
 * n_ops), since the base's resume points hold no transfer state. */
int sim_batch(const gmg_t* g, const uint8_t* d_place, int32_t K, int32_t ld,
              const sim_opts_t* opts, const sim_out_t* d_out, void* d_scratch,
              size_t scratch_bytes, gmg_stream_t stream);

/* Size of the library's own scratch buffer used by sim_batch_noalloc. */
#define GMG_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

/* sim_batch without a caller scratch buffer (the paper has no counterpart;
 * this is a deployment convenience).  Some callers cannot allocate device
 * memory when they evaluate placements: a scheduler loop that runs under a
 * fixed device-memory budget, code embedded in another framework that owns
 * the allocator, or a host that must not allocate after start-up.  This call
 * takes only the placements and the output arrays; the per-warp scratch is a
 * GMG_NOALLOC_SCRATCH_BYTES buffer compiled into the library, present on every
 * GPU that loads the library until the process exits.  It never calls
 * cudaMalloc or cudaFree.  Results are identical to sim_batch; with large
 * graphs fewer warps run at once because fewer scratch slots fit.
 *   - Returns GMG_EWS if one warp's scratch for this graph does not fit in
 *     the buffer (about 16 bytes per op plus queue spill space), other
 *     arguments and errors as sim_batch.
 *   - The first call on each device looks up the buffer's device address
 *     (with that device current) and keeps it for the life of the process;
 *     make that first call before any stream capture, and do not call this
 *     entry point again after a cudaDeviceReset of that device (the reset
 *     unloads the library's module, so the kept address no longer holds).
 *   - All calls share the buffer and find the previous call's data in it;
 *     nothing needs clearing (the kernel initialises what it reads), but two
 *     calls that could run at the same time on the GPU race: order them. */
int sim_batch_noalloc(const gmg_t* g, const uint8_t* d_place, int32_t K, int32_t ld,
                      const sim_opts_t* opts, const sim_out_t* d_out, gmg_stream_t stream);

/* Bytes of device workspace base_create needs. */
size_t base_workspace_bytes(const gmg_t* g, const sim_opts_t* opts);

/* Simulate the base placement (device uint8 [n_ops]) once and record what
 * incremental candidates resume from: per-op ready and finish times and
 * snapshots of the simulator state at time boundaries (the GMG snapshot of
 * Sec. 3.3.2 from which a simulator can be rebuilt at any instant).
 * Asynchronous on `stream`; *out receives the handle.
 *   - opts->transfer_mode GMG_TRANSFER_ARBITRATED (at most 32 accelerators,
 *     a graph with link ids): the base is simulated with the arbiter of
 *     Sec. 3.5.2 and each snapshot also keeps the arbiter's state (input
 *     counters, holds, intent FIFOs, pair queues, endpoint and link sets);
 *     such a base serves arbitrated candidates only.  On more accelerators
 *     the call returns GMG_EINVAL; take a pure-latency base there (arbitrated
 *     candidates against it are simulated in full).
 *   - GMG_STAGING_SHARED in opts->gmg_staging is refused (GMG_EINVAL). */
int base_create(const gmg_t* g, const uint8_t* d_base_place, const sim_opts_t* opts,
                void* d_base_ws, size_t ws_bytes, gmg_stream_t stream, gmg_base_t** out);

void base_destroy(gmg_base_t* b);

/* Bytes of device scratch sim_incremental needs for K candidates (with
 * arbitrated opts: enough for either kind of base). */
size_t inc_scratch_bytes(const gmg_t* g, int32_t K, const sim_opts_t* opts);

/* K candidates, each a list of moves (op, device) against the base
 * placement (Sec. 3.4.2: small-batch incremental scheduling).  Results equal
 * sim_batch on the moved placement; only the suffix of the timeline that the
 * moves can change is re-simulated, from T0 = min over effective moves x of
 * (min base finish of x's predecessors, or x's release).  Move lists are CSR
 * on the device: ops d_move_op[d_move_off[k]..d_move_off[k+1]) go to
 * d_move_dev[...].  events[k] = ops whose base ready time is >= T0.
 *   - With GMG_TRANSFER_ARBITRATED and an arbitrated base, candidates resume
 *     from the base's arbiter snapshots the same way; with a pure-latency
 *     base, each moved placement is simulated in full (events[k] = n_ops).
 *     An arbitrated base with pure-latency opts returns GMG_EINVAL.
 *   - The first 256 bytes of d_scratch hold a candidate counter that the call
 *     zeroes on `stream` before its launch (warps take resumed candidates one
 *     at a time); calls sharing one scratch buffer must be ordered. */
int sim_incremental(const gmg_t* g, const gmg_base_t* b, const int32_t* d_move_off,
                    const int32_t* d_move_op, const uint8_t* d_move_dev, int32_t K,
                    const sim_opts_t* opts, const sim_out_t* d_out, void* d_scratch,
                    size_t scratch_bytes, gmg_stream_t stream);

/* Bytes of device scratch select_best needs for K candidates. */
size_t select_best_tmp_bytes(int32_t K);

/* Algorithm 1 "BestRecordedCandidateResult": d_best[0] = argmin k of
 * (score, k) (score_mode 0) or (sla_miss, score, k) (mode 1) over candidates
 * with status 0 and viol_flag 0, or -1 if none; d_best[1] = its score
 * (INT64_MAX if none).  Reads status, viol_flag, score, sla_miss of d_out.
 * Two launches: per-block argmin, then a final argmin. */
int select_best(const sim_out_t* d_out, int32_t K, int32_t score_mode, int64_t* d_best,
                void* d_tmp, size_t tmp_bytes, gmg_stream_t stream);

/* Human-readable text of a GMG_E* code or (for codes >= 0) a GMG_SIM_* status. */
const char* gmg_strerror(int code);

/* Exact ceil(n / d) as computed on the device for links (0 <= n < 2^53,
 * 1 <= d < 2^62), exported so host tests can check the multiply-shift form. */
int64_t gmg_ceil_div_host(int64_t n, int64_t d);

#ifdef __cplusplus
}
#endif

#endif /* GMGSIM_H_ */
