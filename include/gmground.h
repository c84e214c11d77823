/*
 * One round of incremental simulation-based scheduling (Algorithm 1, Sec. 3.4)
 * on the GPU: the steps that produce the candidate placements the what-if
 * simulation (gmgsim.h) evaluates, and the write-back of the chosen one.
 *
 *   round_select      frontiers (Sec. 3.4.1) and the issued-operator budget;
 *                     the highest-priority operator of the unscheduled
 *                     frontier; CollectConnectedGraph(op, budget)
 *   round_candidates  one placement row per pre-defined accelerator
 *                     partition, batch ops mapped by their graph template's
 *                     fixed mapping (Sec. 3.4.2)
 *   (sim_batch + select_best evaluate the rows, gmgsim.h)
 *   round_commit      write the chosen placement back and mark the batch
 *                     issued
 *
 * Op states (uint8 per op): 0 unscheduled, 1 issued, 2 done.  The caller keeps
 * the scheduled set closed under predecessors (an op is issued or done only
 * if all its predecessors are).
 *   scheduled frontier   issued/done ops with at least one unscheduled successor
 *   unscheduled frontier unscheduled ops whose predecessors are all issued/done
 * Priority: int64 per op, smaller = more urgent (for example the deadline of
 * its request); ties go to the smaller op id.
 *
 * Batch collection (CollectConnectedGraph): starting from the chosen op, ops
 * are taken in increasing op id from a candidate set seeded with it; taking op
 * x adds every unscheduled successor of x whose predecessors are all
 * scheduled or already taken or waiting, so every batch op can run once its
 * batch predecessors have.  At most min(max_batch, budget - issued) ops.
 *
 * The what-if simulation of a round covers every op of the GMG: ops outside
 * the batch keep the placement given in d_place (scheduled ops their actual
 * placement, unscheduled ones the caller's provisional placement).
 *
 * All pointers are device pointers; calls are asynchronous on `stream` and
 * need no host synchronisation between them (sizes produced on the device are
 * read on the device).  Return 0 or a negative GMG_E* code.
 */
#ifndef GMGROUND_H
#define GMGROUND_H

#include <stddef.h>
#include <stdint.h>

#include "gmgsim.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Round status in info[5]. */
#define GMG_ROUND_BATCH 0      /* a batch was collected */
#define GMG_ROUND_BUDGET 1     /* issued ops >= budget: nothing to schedule */
#define GMG_ROUND_EMPTY 2      /* the unscheduled frontier is empty */
#define GMG_ROUND_NO_FEASIBLE 3 /* (round_commit) no candidate was feasible */

/* Scratch of round_select for this GMG (per-op marks and the candidate
 * queue).  Zero it once (cudaMemset) before the first round; afterwards every
 * round_select call on it takes an epoch different from all earlier ones
 * since the zeroing (1, 2, 3, ...), which avoids clearing per round. */
size_t round_scratch_bytes(const gmg_t* g);

/* Frontiers, budget, chosen op and batch.
 *   d_state [N] uint8, d_prio [N] int64
 *   d_batch [max_batch] int32 out: batch op ids in collection order
 *   d_info  [8] int64 out: [0] batch size, [1] chosen op (-1 if none),
 *           [2] unscheduled frontier size, [3] issued ops, [4] scheduled
 *           frontier size, [5] GMG_ROUND_* status, [6..7] 0 */
int round_select(const gmg_t* g, const uint8_t* d_state, const int64_t* d_prio, int32_t budget,
                 int32_t max_batch, uint32_t epoch, void* d_scratch, size_t scratch_bytes, int32_t* d_batch,
                 int64_t* d_info, gmg_stream_t stream);

/* Candidate rows, one per partition p in [0, n_part) (d_batch / d_info /
 * max_batch as given to round_select):
 *   d_rows [n_part * ld] uint8 out: row p = d_place with every batch op x set to
 *     d_part_dev[d_part_off[p] + s], s = d_map[(d_tmpl[x] * n_part + p) * n_roles + d_role[x]];
 *     an s outside [0, size of partition p) writes 255 (the simulation then
 *     reports a bad device and select_best skips the candidate)
 *   d_place [N] (row of ld >= N, ld % 16 == 0), d_part_off [n_part + 1],
 *   d_part_dev [d_part_off[n_part]], d_tmpl / d_role [N] int32 (role < n_roles),
 *   d_map [n_tmpl * n_part * n_roles] int32. */
int round_candidates(const gmg_t* g, const uint8_t* d_place, int32_t ld, const int32_t* d_batch,
                     int32_t max_batch, const int64_t* d_info, int32_t n_part, const int32_t* d_part_off, const uint8_t* d_part_dev,
                     const int32_t* d_tmpl, const int32_t* d_role, const int32_t* d_map, int32_t n_roles,
                     uint8_t* d_rows, gmg_stream_t stream);

/* Write-back: with d_best = select_best's {k, score}, set every batch op's
 * placement to row k's entry and its state to issued (1).  If k < 0, nothing
 * changes and info[5] becomes GMG_ROUND_NO_FEASIBLE. */
int round_commit(const int32_t* d_batch, int32_t max_batch, int64_t* d_info, const int64_t* d_best,
                 const uint8_t* d_rows, int32_t ld, uint8_t* d_place, uint8_t* d_state, gmg_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* GMGROUND_H */
