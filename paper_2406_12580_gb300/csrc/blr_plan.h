// Tiling plan and workspace layout of the BD-LRU scan kernels (host and device).
//
// The (B, L, D) problem is cut into tiles of `tsteps` consecutive time steps x
// `CH` consecutive channels of one batch row. A thread block scans one tile at
// a time (persistent blocks, static schedule):
//   lane (cv, tcl) of warp w owns channels [cv*VEC, cv*VEC + VEC) of the tile
//   and the kTc steps starting at w*kWarpSteps + tcl*kTc.
// Tiles of the same (batch row, channel group) are chained along time with a
// single-pass decoupled look-back over per-tile, per-channel records: each
// tile publishes its aggregate (A = prod alpha, U = its scan from a zero
// state), then its inclusive prefix (the state after its last step). The recurrence is the
// first-order linear scan of Sec. 3.3, whose operator on affine maps is
// (a2, u2) . (a1, u1) = (a2 a1, a2 u1 + u2).
#pragma once

#include <stddef.h>
#include <stdint.h>

namespace blr {

constexpr int kNvl = 8;                    // lanes along channels (8 x 4 channels per row)
constexpr int kNtl = 4;                    // lanes along time within a warp
constexpr int kTc = 4;                     // time steps per lane
constexpr int kWarpSteps = kNtl * kTc;     // time steps per warp
constexpr int kMaxWarps = 4;               // warps (time sub-tiles) per tile
constexpr int kStripes = 8;                // dlambda float64 partial-sum stripes
constexpr size_t kAlign = 256;             // alignment of every workspace region

// Error bits recorded in FwdHeader::err.
constexpr uint32_t kErrTimeout = 1u;
constexpr uint32_t kErrWorkspace = 2u;
// Per-tile records validate themselves: they are filled with this all-ones
// pattern (a negative NaN with a full payload, which float arithmetic never
// produces) before a scan, and a record is published by one 32- or 64-bit store.
constexpr uint32_t kEmpty = 0xffffffffu;
constexpr int kLookWindow = 4;     // predecessors read per round trip of the look-back

// Upper bound of every inter-block wait.
constexpr uint64_t kWaitTimeoutNs = 1000000000ull;  // 1 s
constexpr uint32_t kMaxWaitIters = 1u << 23;

struct FwdHeader {     // cleared before every forward (by its prep kernel)
  uint32_t spare;
  uint32_t exited;     // blocks that left the tile loop
  uint32_t err;        // error bits (forward and backward timeouts, workspace misuse)
  uint32_t tag;        // hash of the problem, written when the forward completed
  uint32_t complete;   // 1 once every forward tile is done
  uint32_t pad[3];
};

struct BwdHeader {     // cleared before every backward
  uint32_t spare;
  uint32_t exited;
  uint32_t selftest_flag;  // a flag nothing sets (blr_selftest_wait_timeout)
  uint32_t pad[5];
};

// Channels per lane: 4 (a 16-byte float32 or an 8-byte bfloat16 vector), so a
// lane holds 16 elements and a tile covers 8 x 4 = 32 channels.
inline int fwd_vec(int) { return 4; }
inline int bwd_vec(int) { return 4; }

// Problems with at least this many chains of 128-byte row segments (32
// float32 or 64 bfloat16 channels of one batch row) use the serial kernels:
// one warp walks one chain through the whole sequence. The others use the
// tiled look-back kernels. The choice depends only on the problem's shape.
constexpr int64_t kSeqMinChains = 256;
constexpr int64_t kSeqTallRowsMinL = 1024;

// Problems with fewer chains, bfloat16 I/O and sequences of at least kSegMinL
// steps use the segmented serial kernels when they hold at least
// kSegMinElems elements or L >= kSegLongL: each chain is cut into `nseg` time
// segments of `seg_len` steps (a multiple of every box height), a reduce pass
// computes each segment's affine map (A = prod alpha, U = its scan from a zero
// state; for the backward W, its adjoint scan from a zero carry), and the
// serial kernels then walk every segment from the carry that the maps of the
// segments before it (after it, backward) compose. About kSegTargetWarps warps
// run, 16 on each of 152 SMs; a segment is at least kSegMinLen steps.
// Measured on GB300 against the tiled kernels: 1.45x on 8 x 32768 x 512
// bfloat16 fwd + bwd, slower on smaller problems (fewer warps, each walking
// at least kSegMinLen steps) and on float32 (there the reduce pass's second
// read of the inputs costs more than the tiled kernels lose).
// The forward of those problems runs a chained single-pass kernel instead of
// the reduction and the serial pass (the backward keeps the segmented
// kernels): tiles of kChainTile steps x one chain, kChainWarps compute warps a
// tile (a warp slice of kChainSlice steps), chained along time by a decoupled
// look-back over per-(tile, channel) records.
constexpr int kChainWarps = 16;
constexpr int kChainSlice = 8;
constexpr int kChainTile = kChainWarps * kChainSlice;

constexpr int64_t kSegMinL = 2048;
constexpr int64_t kSegMinElems = (int64_t)8 << 20;
constexpr int64_t kSegLongL = 16384;
constexpr int64_t kSegTargetWarps = 2432;
constexpr int64_t kSegMinLen = 128;
constexpr int64_t kSegAlign = 32;

struct Plan {
  int64_t B, L, D;
  int io;           // 0 = float32, 1 = bfloat16
  float c;
  int seq;          // 1: serial kernels, 0: tiled look-back kernels
  int sv;           // serial: channels per lane (row segment of 32 * sv channels)
  int rb;           // serial: steps between the forward's kept states
  int sr, srb;      // serial: rows per TMA box, forward and backward (multiples of rb)
  int64_t n_chain;  // serial: chains = B * ceil(D / (32 * sv))
  int64_t n_carry;  // serial: kept states per chain = ceil(L / rb) - 1
  int64_t nseg;     // segmented serial kernels: segments per chain (0: not used)
  int64_t seg_len;  // segmented: steps per segment (the last may be shorter)
  int64_t n_tc;     // chained forward (when nseg > 0): time blocks of kChainTile steps
  int nwarps;       // warps per block = time sub-tiles per tile
  int64_t tsteps;   // time steps per tile = nwarps * kWarpSteps
  int64_t n_t;      // time tiles
  int ch_f, ch_b;   // channels per tile (forward, backward)
  int64_t n_cg_f, n_cg_b;       // channel groups per batch row
  int64_t n_c_f, n_c_b;         // channel groups in total (B * n_cg)
  int64_t n_tiles_f, n_tiles_b; // n_t * n_c
  uint32_t tag;
  // Workspace byte offsets. Records hold one entry per (time tile, channel):
  // agg = (A, U) of the tile as one 64-bit word, pre = the state after it.
  // Segmented kernels: kept states as the serial kernels' (off_skept) and one
  // map per (segment, batch row, channel) as a float pair (off_sagg: the
  // forward's (A, U) within a gated forward call, the backward's (A, W)).
  // Chained forward: its records, the state after each tile (off_cinc, 32-bit)
  // then the tile's map (off_cagg, 64-bit), filled with ones together before
  // each call.
  // The tiled forward records end at off_frec_end.
  size_t off_fhdr, off_bhdr, off_dlam, off_k, off_skept, off_sagg, off_cinc, off_cagg, off_cend;
  size_t off_fagg, off_fpre, off_frec_end, off_bagg, off_bpre, bytes;
};

inline size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

inline uint32_t fnv1a(uint32_t h, uint64_t v) {
  for (int i = 0; i < 8; ++i) {
    h ^= (uint32_t)(v & 0xff);
    h *= 16777619u;
    v >>= 8;
  }
  return h;
}

// Fills `p` for a validated problem (B, L, D >= 1, D % 8 == 0).
inline void make_plan(int64_t B, int64_t L, int64_t D, int io, float c, Plan* p) {
  p->B = B;
  p->L = L;
  p->D = D;
  p->io = io;
  p->c = c;
  // Time tiling: as few tiles of up to kMaxWarps warps as cover L, balanced.
  const int64_t max_steps = (int64_t)kMaxWarps * kWarpSteps;
  const int64_t n_t0 = (L + max_steps - 1) / max_steps;
  const int64_t per = (L + n_t0 - 1) / n_t0;
  p->nwarps = (int)((per + kWarpSteps - 1) / kWarpSteps);
  p->tsteps = (int64_t)p->nwarps * kWarpSteps;
  p->n_t = (L + p->tsteps - 1) / p->tsteps;
  p->ch_f = kNvl * fwd_vec(io);
  p->ch_b = kNvl * bwd_vec(io);
  p->n_cg_f = (D + p->ch_f - 1) / p->ch_f;
  p->n_cg_b = (D + p->ch_b - 1) / p->ch_b;
  p->n_c_f = B * p->n_cg_f;
  p->n_c_b = B * p->n_cg_b;
  p->n_tiles_f = p->n_t * p->n_c_f;
  p->n_tiles_b = p->n_t * p->n_c_b;
  uint32_t h = 2166136261u;
  h = fnv1a(h, (uint64_t)B);
  h = fnv1a(h, (uint64_t)L);
  h = fnv1a(h, (uint64_t)D);
  h = fnv1a(h, (uint64_t)io);
  uint32_t cbits;
  __builtin_memcpy(&cbits, &c, 4);
  h = fnv1a(h, cbits);
  p->tag = h | 1u;  // never 0, the value of a cleared header
  p->sv = io == 0 ? 1 : 2;
  p->rb = io == 0 ? 16 : 8;
  // Long float32 sequences stream the forward in 32-row boxes (fewer, larger
  // TMA loads per chain); shorter ones in 16-row boxes, which reach the first
  // rows sooner.
  p->sr = (io == 0 && L >= kSeqTallRowsMinL) ? 32 : 16;
  p->srb = io == 0 ? 16 : 8;
  p->n_chain = B * ((D + 32 * p->sv - 1) / (32 * p->sv));
  p->n_carry = (L + p->rb - 1) / p->rb - 1;
  p->seq = p->n_chain >= kSeqMinChains ? 1 : 0;
  p->nseg = 0;
  p->seg_len = 0;
  p->n_tc = 0;
  if (!p->seq && io == 1 && L >= kSegMinL && (B * L * D >= kSegMinElems || L >= kSegLongL)) {
    int64_t n = (kSegTargetWarps + p->n_chain - 1) / p->n_chain;
    int64_t len = (L + n - 1) / n;
    if (len < kSegMinLen) len = kSegMinLen;
    len = (len + kSegAlign - 1) / kSegAlign * kSegAlign;
    p->seg_len = len;
    p->nseg = (L + len - 1) / len;
    p->n_tc = (L + kChainTile - 1) / kChainTile;
  }
  // The forward's states after each time tile (or every rb steps of a serial
  // chain, but the last) are kept for the backward; the tiled kernels also
  // need aggregates and backward records.
  const int64_t kept = p->seq ? p->n_carry : p->n_t;
  const size_t rec = (size_t)kept * (size_t)B * (size_t)D;
  const size_t rec_t = p->seq ? 0 : rec;
  size_t o = 0;
  p->off_fhdr = o;
  o = align_up(o + sizeof(FwdHeader), kAlign);
  p->off_bhdr = o;
  o = align_up(o + sizeof(BwdHeader), kAlign);
  p->off_dlam = o;
  o = align_up(o + 8 * (size_t)kStripes * (size_t)D, kAlign);
  p->off_k = o;
  o = align_up(o + 4 * (size_t)D, kAlign);
  p->off_fpre = o;  // forward records: pre then agg, emptied together
  // The segmented kernels' kept states and maps lie over the tiled forward
  // records: a forward of either family retags the workspace (the tiled one's
  // preparation clears the tag first), and each backward checks its own tag.
  const size_t kept_s = p->nseg ? (size_t)p->n_carry * (size_t)B * (size_t)D : 0;
  const size_t maps_s = (size_t)p->nseg * (size_t)B * (size_t)D;
  const size_t crec = (size_t)p->n_tc * (size_t)B * (size_t)D;
  p->off_skept = o;
  p->off_sagg = align_up(p->off_skept + 4 * kept_s, kAlign);
  p->off_cinc = align_up(p->off_sagg + 8 * maps_s, kAlign);
  p->off_cagg = align_up(p->off_cinc + 4 * crec, kAlign);
  p->off_cend = align_up(p->off_cagg + 8 * crec, kAlign);
  const size_t seg_end = p->off_cend;
  o = align_up(o + 4 * rec, kAlign);
  p->off_fagg = o;
  o = align_up(o + 8 * rec_t, kAlign);
  p->off_frec_end = o;
  if (o < seg_end) o = seg_end;
  p->off_bagg = o;  // backward records
  o = align_up(o + 8 * rec_t, kAlign);
  p->off_bpre = o;
  o = align_up(o + 4 * rec_t, kAlign);
  p->bytes = o;
}

}  // namespace blr
