// Tiling plan and workspace layout of the BD-LRU scan kernels (host and device).
//
// The (B, L, D) problem is cut into tiles of `ttile` time steps x `dblk`
// channels of one batch row. One thread block scans one tile: thread (tx, ty)
// owns channels [tx*vec, tx*vec + vec) of the block and the `tc` consecutive
// time steps starting at ty*tc. Tiles of the same (batch row, channel block)
// are chained along time with a single-pass decoupled look-back: each block
// publishes its tile's aggregate (A = prod alpha, U = the tile's scan from a
// zero state), then its inclusive prefix (the state at its last step) once the
// carry from earlier tiles is known. The recurrence is the first-order linear
// scan of Sec. 3.3, whose operator is (a2, u2) . (a1, u1) = (a2 a1, a2 u1 + u2).
#pragma once

#include <stddef.h>
#include <stdint.h>

namespace blr {

constexpr int kMaxDblk = 64;       // channels per thread block
constexpr int kMaxNt = 32;         // time chunks (threads along time) per block
constexpr int kTc = 4;             // time steps per thread chunk
constexpr int kTargetTile = 64;    // preferred time steps per tile
constexpr int kStripes = 8;        // dlambda float64 partial-sum stripes
constexpr size_t kAlign = 256;     // alignment of every workspace region

// Error bits recorded in FwdHeader::err.
constexpr uint32_t kErrTimeout = 1u;
constexpr uint32_t kErrWorkspace = 2u;
// Tile status flags of the look-back.
constexpr uint32_t kFlagAggregate = 1u;
constexpr uint32_t kFlagPrefix = 2u;

// Upper bound of every inter-block wait.
constexpr uint64_t kWaitTimeoutNs = 1000000000ull;  // 1 s
constexpr uint32_t kMaxWaitIters = 1u << 23;

struct FwdHeader {     // zeroed before every forward
  uint32_t ticket;     // tile tickets handed out (launch order of tiles)
  uint32_t done;       // forward tiles completed
  uint32_t err;        // error bits (timeouts of forward and backward, workspace misuse)
  uint32_t tag;        // hash of the problem the carries belong to
};

struct BwdHeader {     // zeroed before every backward
  uint32_t ticket;
  uint32_t done;
  uint32_t selftest_flag;  // a flag nothing sets (blr_selftest_wait_timeout)
  uint32_t pad;
};

struct Plan {
  int64_t B, L, D;
  int io;           // 0 = float32, 1 = bfloat16
  float c;
  int vec;          // channels per thread (one 16-byte vector)
  int tc;           // time steps per thread chunk
  int dblk;         // channels per tile
  int nv;           // threads along channels = dblk / vec
  int nt;           // threads along time
  int64_t ttile;    // time steps per tile = tc * nt
  int64_t n_dblk;   // channel blocks per batch row
  int64_t n_c;      // channel blocks in total = B * n_dblk
  int64_t n_t;      // time tiles
  int64_t n_tiles;  // n_c * n_t
  uint32_t tag;
  // workspace byte offsets
  size_t off_fhdr, off_fflags, off_bhdr, off_dlam, off_bflags;
  size_t off_fagg, off_fpre, off_bagg, off_bpre, bytes;
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
  p->vec = (io == 0) ? 4 : 8;
  p->tc = kTc;
  p->dblk = (int)(D < kMaxDblk ? D : kMaxDblk);
  p->nv = p->dblk / p->vec;
  int64_t n_t = (L + kTargetTile - 1) / kTargetTile;
  int64_t per = (L + n_t - 1) / n_t;                  // balanced tile length
  int nt = (int)((per + p->tc - 1) / p->tc);
  while (p->nv * nt < 32) ++nt;                         // at least one full warp
  p->nt = nt;
  p->ttile = (int64_t)nt * p->tc;
  p->n_t = (L + p->ttile - 1) / p->ttile;
  p->n_dblk = (D + p->dblk - 1) / p->dblk;
  p->n_c = B * p->n_dblk;
  p->n_tiles = p->n_c * p->n_t;
  uint32_t h = 2166136261u;
  h = fnv1a(h, (uint64_t)B);
  h = fnv1a(h, (uint64_t)L);
  h = fnv1a(h, (uint64_t)D);
  h = fnv1a(h, (uint64_t)io);
  uint32_t cbits;
  __builtin_memcpy(&cbits, &c, 4);
  h = fnv1a(h, cbits);
  p->tag = h | 1u;  // never 0, the value of a cleared header
  size_t o = 0;
  p->off_fhdr = o;
  o = align_up(o + sizeof(FwdHeader), kAlign);
  p->off_fflags = o;
  o = align_up(o + 4 * (size_t)p->n_tiles, kAlign);
  p->off_bhdr = o;
  o = align_up(o + sizeof(BwdHeader), kAlign);
  p->off_dlam = o;
  o = align_up(o + 8 * (size_t)kStripes * (size_t)D, kAlign);
  p->off_bflags = o;
  o = align_up(o + 4 * (size_t)p->n_tiles, kAlign);
  const size_t rec = (size_t)p->n_tiles * (size_t)p->dblk;
  p->off_fagg = o;
  o = align_up(o + 8 * rec, kAlign);
  p->off_fpre = o;
  o = align_up(o + 4 * rec, kAlign);
  p->off_bagg = o;
  o = align_up(o + 8 * rec, kAlign);
  p->off_bpre = o;
  o = align_up(o + 4 * rec, kAlign);
  p->bytes = o;
}

}  // namespace blr
