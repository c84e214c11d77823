// Device layout of a GMG and launch parameters shared by the library's host
// code (gmgsim_host.cu) and its kernels (gmgsim_kernels.cu).  Private to the
// library: not part of the C ABI.
#pragma once

#include <stdint.h>

#include "../../include/gmgsim.h"

namespace gsim {

// One 64-byte record per operator, in four 16-byte pieces grouped by use:
// [dur, bytes] | [release, predecessor list] (readiness checks) | [xq,
// successor list] (starting the op) | [consumer list, request, flags].
struct alignas(64) OpRec {
  int64_t dur;       // duration (us), >= 1
  int64_t bytes;     // output size (B)
  int64_t release;   // arrival of the op itself (us)
  uint32_t pred_off; // predecessors: pred[pred_off .. +npred); bit 31 set if this op
  uint32_t npred;    //   is a listed consumer of that predecessor's output
  int64_t xq;        // ceil(bytes / bw) when every link has the same bandwidth
  uint32_t succ_off; // successors: succ[succ_off .. +nsucc), ascending
  uint32_t nsucc;
  uint32_t cons_off; // listed consumers of this op's output: cons[cons_off .. +ncons)
  uint32_t ncons;    //   (equals the successor list when kAllCons is set)
  int32_t req;       // request id or -1
  uint32_t flags;    // kScored | kReqSink | kAllCons
};
static_assert(sizeof(OpRec) == 64, "OpRec must be 64 bytes");

constexpr uint32_t kScored = 1u;   // counts in the score
constexpr uint32_t kReqSink = 2u;  // no successor in its own request: may end the request
constexpr uint32_t kAllCons = 4u;  // consumers = successors
constexpr uint32_t kHoldBit = 0x80000000u;
constexpr uint32_t kSibNone = 0xffffffffu;  // the only listed consumer
constexpr uint32_t kSibMany = 0xfffffffeu;  // three or more listed consumers
constexpr uint32_t kSibLater = 0x40000000u; // flag: the other consumer is a descendant
constexpr uint32_t kIdMask = 0x7fffffffu;

// Exact ceil(n / bw) by multiply-shift (Granlund & Montgomery 1994,
// "Division by invariant integers using multiplication", Thm 4.2): with
// l = ceil(log2 bw), s = 53 + l and m = ceil(2^s / bw), floor(n / bw) =
// floor(m * n / 2^s) for every 0 <= n < 2^53.
struct LinkRec {
  uint64_t magic;
  int64_t bw;
  int64_t lat;
  int32_t shift;
  int32_t pad;
};
static_assert(sizeof(LinkRec) == 32, "LinkRec must be 32 bytes");

#if defined(__CUDACC__)
#define GMG_HD __host__ __device__ __forceinline__
#else
#define GMG_HD inline
#endif

GMG_HD uint64_t mulhi_u64(uint64_t a, uint64_t b) {
#if defined(__CUDA_ARCH__)
  return __umul64hi(a, b);
#else
  return (uint64_t)(((unsigned __int128)a * (unsigned __int128)b) >> 64);
#endif
}

GMG_HD int64_t ceil_div_link(int64_t n, const LinkRec& L) {
  const uint64_t un = (uint64_t)n;
  const uint64_t hi = mulhi_u64(un, L.magic);
  const uint64_t lo = un * L.magic;
  const int s = L.shift;
  const uint64_t q = s >= 64 ? (hi >> (s - 64)) : ((hi << (64 - s)) | (lo >> s));
  return (int64_t)q + ((int64_t)q * L.bw != n ? 1 : 0);
}

// Pointers into the caller's device workspace.
struct DevGmg {
  const OpRec* ops;
  const uint32_t* succ;
  const uint32_t* pred;
  const uint2* predsib;       // per predecessor entry: {pred | hold bit, the other listed
                              // consumer of that predecessor (kSibNone / kSibMany)}
  const uint32_t* cons;
  const uint64_t* root_keys;  // READY keys of ops without predecessors, ascending
  const uint64_t* root_keys_q;// the same keys with the duration class below them (batched sweep)
  const int64_t* cap;
  const int64_t* base;
  const int64_t* avail0;
  const int64_t* deadline;
  const LinkRec* links;       // D*D, NULL when links are uniform
  int64_t lat0;               // uniform latency
  int64_t max_iter;           // event-loop iteration cap per candidate
  int32_t n, D, R, nroots;
  int32_t ib;                 // op-id bits of a packed key
  int32_t tb;                 // time bits needed (every time < 2^tb)
  int32_t dev_key;            // 1 if an accelerator id fits above (time, class, op) in 64 bits
  int32_t t32;                // 1 if every time is below 2^31 (the kernels then use int32 times)
  int32_t ntypes;             // accelerator types; >= 2: durations from durt by dtype
  const int64_t* durt;        // [N*ntypes] duration of op i on type t at i*ntypes + t
  const uint8_t* dtype;       // [D] type of each accelerator
  int32_t uniform;
  int32_t batch;              // 1: the kernels take READY keys in batches (keys carry kQB class bits)
  // The hot fields in the compact form a CTA stages into shared memory
  // (sim_full_staged_kernel); present when stage_ok.
  const uint4* st_hot;        // [N] {dur, xq | flags << 29, succ_off | nsucc << 24, pred_off | npred << 24}
  const int32_t* st_rel;      // [N] release
  int32_t stage_ok;           // 1: 32-bit times, one type, uniform links, lists and sizes fit the fields
  int32_t n_edges;
  const uint8_t* ws;          // the whole device copy (every array above), for L2 prefetches
  int64_t ws_bytes;
};

// Bytes of the staged copy in shared memory: an mbarrier, then the four
// arrays, each padded to 16 bytes (bulk copies move multiples of 16 bytes).
#if defined(__CUDACC__)
__host__ __device__
#endif
inline int64_t stage_smem_bytes(int64_t n, int64_t E) {
  return 16 + 16 * n + (4 * n + 15) / 16 * 16 + 2 * ((4 * E + 15) / 16 * 16);
}

// Resident 4-warp blocks per SM the batched kernels are compiled for (their
// register budget; compile-time overridable for tuning sweeps).
#ifndef GMG_BATCH_BLOCKS_PER_SM
#define GMG_BATCH_BLOCKS_PER_SM 7
#endif
constexpr int kBatchBlocksPerSM = GMG_BATCH_BLOCKS_PER_SM;

// The staged-GMG kernel's largest CTA (one per SM; 72 registers a thread).
constexpr int kStageMaxWarps = 28;

// Batched sweep: a READY key is followed by kQB bits holding floor(log2) of a
// lower bound of the op's duration (31 at most).
constexpr int kQB = 5;

// Packed event key: time << (ib + 2) | class << ib | op.  Classes at equal
// times: READY (an op's last input arrived) < FREE < ALLOC.
constexpr uint32_t kReady = 0, kFree = 1, kAlloc = 2;

// Candidate simulation modes.
enum Mode : int { kFull = 0, kInc = 1, kBase = 2 };

// Output pointers (device) as in sim_out_t.
struct DevOut {
  int64_t* makespan;
  int64_t* score;
  int32_t* status;
  int32_t* viol_flag;
  int32_t* viol_op;
  int32_t* viol_dev;
  int64_t* viol_time;
  int64_t* peak;
  int32_t* sla_miss;
  int64_t* events;
  int64_t* req_done;
  int64_t* trace_start;
  int64_t* trace_finish;
};

// Base snapshot (incremental resume points) in the base workspace.
struct DevBase {
  uint8_t* row;          // [ld] base placement
  int64_t* rb;           // [N] base ready time
  int64_t* fb;           // [N] base finish time
  int32_t* status;       // [1]
  // base results (outputs of the base placement)
  int64_t* res_scalars;  // [8]: makespan, score, viol_flag, viol_op, viol_dev, viol_time, sla_miss, n_ck
  int64_t* res_peak;     // [D]
  int64_t* res_creq;     // [R]
  // checkpoints c = 0 .. nck-1
  int64_t* ck_time;      // [nck]  T_c (INT64_MAX = not recorded)
  int64_t* ck_scalars;   // [nck*8]: qsize, rootptr, score, makespan, vflag, vt, vop<<32|vdev, log size
  int64_t* ck_dev;       // [nck*3*D]: free, live, peak
  int64_t* ck_creq;      // [nck*R]
  uint64_t* ck_qkey;     // [nck*ckq] READY heap
  uint64_t* ck_mkey;     // [nck*ckm] HBM event log entries
  uint8_t* ck_mdev;      // [nck*ckm] their accelerators (when not inside the entries)
  int32_t nck;
  int32_t ckq;           // READY entries per checkpoint
  int32_t ckm;           // HBM events per checkpoint
  int32_t ld;
  int32_t stride_pops;   // READY pops between checkpoints
};

struct SimParams {
  DevGmg g;
  DevOut out;
  DevBase base;
  const uint8_t* place;  // kFull: [K][ld]; kBase: base row
  int64_t ld;
  int32_t K;
  int32_t qs;            // READY heap slots in shared memory per warp (32m+1, >= 33)
  int32_t qcap;          // READY heap slots per warp
  int32_t ms;            // HBM event log slots in shared memory per warp
  int32_t mcap;          // HBM event log slots per warp
  int32_t sortcap;       // sort area entries per warp (power of two, >= max(32, n_dev))
  int32_t drain_trigger; // batched sweep: ops started before an HBM-event generation
  int32_t opcap;         // ops started between HBM-event generations (one at a time), or the
                         // capacity of the list of started ops (batched: drain_trigger + 32)
  int32_t n_trace;
  const int32_t* trace_k;
  const int32_t* move_off;
  const int32_t* move_op;
  const uint8_t* move_dev;
  uint8_t* scratch;
  int64_t slot_bytes;    // scratch bytes per warp slot
  int32_t dev_bytes;     // shared bytes of accelerator state per warp
  int32_t stage_bytes;   // shared bytes of the staged GMG copy (sim_full_staged_kernel), else 0
  int32_t no_side;       // 1: no side bytes in shared memory (the accelerator is inside the log entry)
  int32_t pad_;
  // byte offsets inside a slot (off_pk < 0: the peaks are in shared memory)
  int64_t off_f, off_hold, off_bits, off_creq, off_qk, off_mk, off_md, off_row, off_pk;
  // Incremental candidates: the next candidate a warp takes (zeroed before
  // the launch).  Resumed candidates differ widely in length, so warps take
  // them one at a time instead of a fixed stride.
  uint32_t* next_k;
};

// Scratch bytes in front of the slots of a resumed incremental launch (the
// candidate counter).
constexpr size_t kCounterBytes = 256;

}  // namespace gsim
