// Shared pieces of the d = 128 / 80 backward main kernels (csrc/attn_bwd_d128.cu, one CTA
// per key tile; csrc/attn_bwd_d128_persist.cu, CTAs walking key tiles): shared-memory and
// TMEM layout, barrier block, work items.
#pragma once
#include "common.cuh"

namespace ddattn {

template <int D_>
struct BwdBig {
  static constexpr int D = D_, BN = 128, BQ = 128;
  static constexpr int NCH = (D + 31) / 32;              // 32-column chunks of dQ^T / dK / dV
  static constexpr int BLK = 128 * 128;                  // [128 rows][64] bf16, 128B swizzle
  static constexpr int TILE = 2 * BLK;                   // [128 rows][128] bf16
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + TILE;
  static constexpr int OFF_Q = OFF_V + TILE;             // 2 stages
  static constexpr int OFF_DO = OFF_Q + 2 * TILE;        // 2 stages (dO, then dS^T)
  static constexpr int OFF_STG = OFF_DO + 2 * TILE;      // dQ staging
  static constexpr int STG_BYTES = 2 * 4 * 32 * 32 * 4; // two [32 x 32] fp32 slices per drain warp
  static constexpr int OFF_LSE = OFF_STG + STG_BYTES;    // [2][128] fp32
  static constexpr int OFF_DEL = OFF_LSE + 2 * BQ * 4;   // [2][128] fp32
  static constexpr int OFF_BAR = OFF_DEL + 2 * BQ * 4;
  // No alignment slack: the dynamic shared-memory base is 1024-aligned on this GPU (0x400 in
  // every launch shape probed); the kernels check it at entry and record an error otherwise.
  static constexpr int SMEM_BYTES = OFF_BAR + 256;
  static constexpr uint32_t TM_R = 0, TM_DV = 256, TM_DK = 384;  // R[k] at TM_R + 128 k
  static constexpr int THREADS = 512;
  // setmaxnreg splits (4 warps low, 12 high): the per-tile kernel's, and the persistent
  // kernel's, whose per-item state needs more registers in the producer / MMA group.
  static constexpr int REGS_LOW = 32, REGS_HIGH = 160;
  static constexpr int REGS_LOW_P = 48, REGS_HIGH_P = 152;
};
static_assert(4 * 32 * BwdBig<128>::REGS_LOW + 12 * 32 * BwdBig<128>::REGS_HIGH <= 512 * 128, "register split");
static_assert(4 * 32 * BwdBig<128>::REGS_LOW_P + 12 * 32 * BwdBig<128>::REGS_HIGH_P <= 512 * 128, "register split");

struct Bwd128Bars {
  uint64_t kv_full;
  uint64_t q_full[2], q_empty[2];
  uint64_t s_full, dp_full, p_full, dp_read, dss_full, dv_done, dq_full, r_free;
  uint64_t mma_done;
  // the persistent kernel's item hand-offs
  uint64_t kv_empty;          // the item's MMAs are done: K / V may be replaced
  uint64_t dv_free, dk_free;  // the item's dV / dK have left TMEM: the next item may accumulate
  uint64_t mma_drain;
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(Bwd128Bars) <= 256, "barrier block");
static_assert(BwdBig<128>::SMEM_BYTES <= 232448, "shared memory per block");

// The layout's 1024-byte alignment (128B-swizzled tiles) holds only if the dynamic
// shared-memory base is 1024-aligned. If it is not, the kernel records
// kStatusLayout and every thread returns before touching shared memory.
__device__ __forceinline__ bool smem_base_ok(const uint8_t* smem_raw, int* status) {
  if ((smem_u32(smem_raw) & 1023u) == 0) return true;
  if (threadIdx.x == 0 && status) atomicCAS(status, 0, kStatusLayout);
  return false;
}

// A work item: one 128-key tile of one (sequence, head) and its live query tiles, from the
// diagonal to the end of the tile's last document. Items are numbered key tile fastest.
struct BwdItem {
  int n, h, b, kv0, m_lo, nq;
  long long seq0, vec0;
};
template <int BN, int BQ>
__device__ __forceinline__ BwdItem bwd_item(const BwdParams& p, int it) {
  BwdItem I;
  I.n = it % p.nkt;
  I.h = (it / p.nkt) % p.H;
  I.b = it / (p.nkt * p.H);
  I.seq0 = (long long)I.b * p.L;
  I.kv0 = I.n * BN;
  const int kv_last = min(I.kv0 + BN - 1, p.L - 1);
  const int de_last = (int)(doc_end(p.offsets, p.n_offsets, I.seq0 + kv_last, I.seq0 + p.L) - I.seq0);
  I.m_lo = I.kv0 / BQ;
  I.nq = (de_last - 1) / BQ - I.m_lo + 1;
  I.vec0 = ((long long)I.b * p.H + I.h) * p.L128;  // row 0 of this (b, h) in the padded vectors
  return I;
}

// How the CTAs of the walking backward kernel get their items (a template parameter, so
// that each kernel instance holds only its own walk's code).
enum BwdWalk { kWalkStatic = 0, kWalkOwned = 1 };

// The w-th item of this CTA's walk (w = 0, 1, ...), or -1 past its end. Two orders:
//   * per key tile: items c, c + G, c + 2G, ... (c = blockIdx.x, G = gridDim.x coprime with
//     the key-tile count), so the CTAs share the (sequence, head) pairs' dQ rows and reduce
//     their partials into one fp32 accumulator that the post kernel converts;
//   * dQ owned (kWalkOwned): CTA c owns the (sequence, head) pairs c, c + G, ... and walks
//     each one's key tiles from the last to the first. All partials of a query tile then
//     come from one CTA, the first of them from the key tile on its diagonal (step 0 of that
//     item: no key tile after it reaches back to the tile, and every earlier one reaches it
//     only after), and the last from the key tile that holds the document start of the
//     tile's first row.
template <int WALK>
__device__ __forceinline__ int bwd_walk_item(const BwdParams& p, int w) {
  if (WALK != kWalkOwned) {
    const long long it = blockIdx.x + (long long)w * gridDim.x;
    return it < (long long)p.nkt * p.H * p.B ? (int)it : -1;
  }
  const long long bh = blockIdx.x + (long long)(w / p.nkt) * gridDim.x;
  if (bh >= (long long)p.B * p.H) return -1;
  return (int)(bh * p.nkt + (p.nkt - 1 - w % p.nkt));
}

// Key tile (relative to the sequence) of the last dQ contributor of query tile qt in the
// dQ-owned walk: the tile holding the document start of the query tile's first row.
__device__ __forceinline__ int bwd_last_contributor(const BwdParams& p, long long seq0, int qt) {
  return (int)((doc_start(p.offsets, p.n_offsets, seq0 + (long long)qt * 128, seq0) - seq0) / 128);
}

}  // namespace ddattn
