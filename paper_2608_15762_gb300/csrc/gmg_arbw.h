// Launch parameters of the arbitrated-transfer simulation for 33 to 256
// accelerators (gmgsim_arbw.cu).  Private to the library: shared by the host
// translation unit (gmgsim_host.cu) and gmgsim_arbw.cu.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "gmg_layout.h"

namespace gsim {

struct ArbWParams {
  SimParams P;            // the full simulation's parameters (slot offsets inside P too)
  const uint16_t* link;   // [D*D] link id of each ordered accelerator pair (< D*D)
  const int32_t* pre_status;  // [K] optional: a nonzero entry is the candidate's status, not simulated
  int32_t shared_links;   // 1 if two ordered pairs share a link id
  int32_t xcap;           // transfers per candidate (sum over ops of min(successors, D-1))
  int32_t words;          // W = ceil(D / 32): words of an accelerator bit set
  int32_t smem_arb;       // shared bytes of the arbitration state per warp
  int64_t smem_std;       // shared bytes of the simulation state of all warps of a block
  // byte offsets inside a warp's scratch slot
  int64_t off_cnt;        // int32 [N]  inputs present
  int64_t off_rmax;       // time  [N]  latest input arrival so far
  int64_t off_refs;       // int32 [N]  holds left on an op's own output copy
  int64_t off_nextop;     // int32 [N]  next started op of the same accelerator with remote successors
  int64_t off_xent;       // uint32 [xcap]  arrived intent: producer << 8 | destination
  int64_t off_xnext;      // int32 [xcap]  next intent of the same pair (-1: last)
  int64_t off_qhead;      // int32 [D*D]  first pending intent of each pair (-1: none)
  int64_t off_qtail;      // int32 [D*D]
  int64_t off_xd;         // time [D]   completion of the transfer each accelerator is sending (never: none)
  int64_t off_xp;         // uint32 [D] its producer
  int64_t off_xe;         // int32 [D]  its destination
  int64_t off_fh;         // int32 [D]  head of each accelerator's FIFO of coming intents (-1: empty)
  int64_t off_ft;         // int32 [D]  its tail
  int64_t off_fa;         // time [D]   finish time of the head (never: empty)
  int64_t off_pm;         // uint32 [D*W] destinations with a pending intent, per source
  int64_t off_lb;         // uint32 [ceil(D*D/32)] busy links
};

const void* arbw_kernel_ptr(bool t32, bool types);
cudaError_t launch_arbw(bool t32, bool types, const ArbWParams& A, int grid, int block, size_t smem,
                        cudaStream_t st);

}  // namespace gsim
