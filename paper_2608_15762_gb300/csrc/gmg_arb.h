// Launch parameters of the arbitrated-transfer simulation (sim_batch with
// transfer_mode = GMG_TRANSFER_ARBITRATED).  Private to the library: shared
// by the host translation unit (gmgsim_host.cu) and gmgsim_arb.cu.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "gmg_layout.h"

namespace gsim {

// An arbitrated base snapshot keeps, beside the simulation state of every
// checkpoint (DevBase), the arbiter's state at that instant in one arena per
// checkpoint: the per-op input counters, latest arrivals, holds, remote sets,
// FIFO links and hold times, the arrived intents, the pair queues, every
// lane's sending transfer and FIFO head, and the endpoint and link sets.
struct ArbCk {
  uint8_t* arena;         // [nck][bytes]
  int64_t bytes;          // per checkpoint
  int64_t off_cnt, off_rmax, off_refs, off_rmask, off_nextop, off_hold;  // per op (times as int64)
  int64_t off_xent, off_xnext;  // [xcap]
  int64_t off_qhead, off_qtail; // [D*D]
  int64_t off_lanes;      // [32][7] int64: pm, xd, xdp, xde, fh, ft, fa
  int64_t off_warp;       // int64 nx, xev, sendm, recvm; then uint32 lbits[32]
};

struct ArbParams {
  SimParams P;            // the full simulation's parameters (slot offsets inside P too)
  const uint16_t* link;   // [D*D] link id of each ordered accelerator pair (< D*D)
  int32_t shared_links;   // 1 if two ordered pairs share a link id (else the sender check covers links)
  int32_t xcap;           // transfers per candidate (sum over ops of min(successors, D-1))
  int32_t heads_shared;   // 1: the pair queue heads live in shared memory (D <= 16)
  int32_t smem_arb;       // shared bytes of the arbitration state per warp
  int64_t smem_std;       // shared bytes of the simulation state of all warps of a block
  // byte offsets inside a warp's scratch slot
  int64_t off_cnt;        // int32 [N]  inputs present
  int64_t off_rmax;       // time  [N]  latest input arrival so far
  int64_t off_refs;       // int32 [N]  holds left on an op's own output copy
  int64_t off_rmask;      // uint32 [N] remote accelerators of an op's successors
  int64_t off_nextop;     // int32 [N]  next started op of the same accelerator with remote successors
  int64_t off_xent;       // uint32 [xcap]  arrived intent: producer << 5 | destination
  int64_t off_xnext;      // int32 [xcap]  next intent of the same pair (-1: last)
  int64_t off_qhead;      // int32 [D*D]  first pending intent of each pair (-1: none), when not shared
  int64_t off_qtail;      // int32 [D*D]
  const int32_t* pre_status;  // [K] optional: a nonzero entry is the candidate's status, not simulated
  ArbCk ck;               // arbitrated base snapshot (base and resumed incremental launches)
};

// Incremental candidates under arbitrated transfers: row k = the base row with
// candidate k's moves applied (rows [K][ld]); status[k] = the move list's
// GMG_SIM_* code (GMG_SIM_BADBASE for every candidate if *base_status is not OK).
cudaError_t launch_expand_moves(const uint8_t* base_row, const int32_t* base_status, int32_t ld, int32_t n,
                                int32_t D, const int32_t* off, const int32_t* op, const uint8_t* dev, int32_t K,
                                uint8_t* rows, int32_t* status, cudaStream_t st);

// Kernel entry of one instance (for occupancy queries) and the launcher.
const void* arb_kernel_ptr(bool t32, bool types);
cudaError_t launch_arb(bool t32, bool types, const ArbParams& A, int grid, int block, size_t smem,
                       cudaStream_t st);

// The arbitrated base snapshot (one warp) and the incremental candidates
// resumed from it (at most 32 accelerators).
const void* arb_base_kernel_ptr(bool types);
const void* arb_inc_kernel_ptr(bool t32, bool types);
cudaError_t launch_arb_base(bool types, const ArbParams& A, size_t smem, cudaStream_t st);
cudaError_t launch_arb_inc(bool t32, bool types, const ArbParams& A, int grid, int block, size_t smem,
                           cudaStream_t st);

}  // namespace gsim
