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

// ---- dV / dK epilogues
// A thread holds one row of an accumulator (its TMEM lane), and rows lie H d elements apart in
// memory, so storing from the thread that holds the row would have each store instruction of a
// warp touch 32 lines. Both epilogues rearrange the bf16 rows first so that every store
// instruction writes whole 128-byte lines.

// 8 x 8 transpose of 16-byte parts within each group of 8 lanes (butterfly over lane bits 4,
// 2, 1): lane 8G + i enters with parts x[0..7] of row i of its group and leaves with part i of
// its group's rows 0..7 (x[k]: row k).
__device__ __forceinline__ void transpose8x8_u4(uint4 (&x)[8], int lane) {
#pragma unroll
  for (int b = 4; b >= 1; b >>= 1) {
    const bool hi = (lane & b) != 0;
#pragma unroll
    for (int j = 0; j < 8; j++) {
      if (j & b) continue;
      const uint4 send = hi ? x[j] : x[j ^ b];
      uint4 recv;
      recv.x = __shfl_xor_sync(0xffffffffu, send.x, b);
      recv.y = __shfl_xor_sync(0xffffffffu, send.y, b);
      recv.z = __shfl_xor_sync(0xffffffffu, send.z, b);
      recv.w = __shfl_xor_sync(0xffffffffu, send.w, b);
      if (hi) x[j] = recv;
      else x[j ^ b] = recv;
    }
  }
}

// dV of one P / dS warp: rows row0 + lane (its TMEM lanes; tl_dv addresses column qh of them)
// x columns qh .. qh + 63 inside d. The two TMEM loads become eight 16-byte bf16 parts of the
// row; release() runs once they are in registers (the accumulator may then be reused); after
// the transpose, store k writes row k of each group of 8 lanes: four whole rows of 64 columns.
template <int D, typename Release>
__device__ __forceinline__ void dv_epilogue(const BwdParams& p, uint32_t tl_dv, int qh, long long seq0, int h,
                                            int row0, int lane, Release release) {
  uint4 x[8];
#pragma unroll
  for (int c = 0; c < 2; c++) {
    if (D - (qh + c * 32) > 0) {  // d = 80: the second group's second chunk is past d
      uint32_t v[32];
      tmem_ld32(tl_dv + c * 32, v);
      tmem_ld_wait(v);
#pragma unroll
      for (int q = 0; q < 4; q++)
        x[4 * c + q] = make_uint4(pack_bf16x2(__uint_as_float(v[8 * q]), __uint_as_float(v[8 * q + 1])),
                                  pack_bf16x2(__uint_as_float(v[8 * q + 2]), __uint_as_float(v[8 * q + 3])),
                                  pack_bf16x2(__uint_as_float(v[8 * q + 4]), __uint_as_float(v[8 * q + 5])),
                                  pack_bf16x2(__uint_as_float(v[8 * q + 6]), __uint_as_float(v[8 * q + 7])));
    } else {
#pragma unroll
      for (int q = 0; q < 4; q++) x[4 * c + q] = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  release();
  transpose8x8_u4(x, lane);
  const int part = lane & 7;
  const bool in_d = qh + 8 * part < D;
#pragma unroll
  for (int k = 0; k < 8; k++) {
    const int row = row0 + 8 * (lane >> 3) + k;
    if (in_d && row < p.L) *reinterpret_cast<uint4*>(p.dv + ((seq0 + row) * p.H + h) * D + qh + 8 * part) = x[k];
  }
}

// dK of one drain warp: rows row0 + lane (its TMEM lanes; tl_dk addresses column 0 of them) x d
// columns, dk = scale * acc, rotated back (R^T) with RoPE, as bf16 16-byte parts staged in the
// warp's 8 KB of shared memory at stg (part t of row r at r * 256 + ((t ^ (r & 7)) * 16):
// conflict-free writes by row and reads by line); release() runs once TMEM is read; then
// consecutive lanes copy consecutive parts, so each store instruction writes two whole rows.
template <int D, int NCH, typename Release>
__device__ __forceinline__ void dk_epilogue(const BwdParams& p, uint32_t tl_dk, uint32_t stg, long long seq0, int h,
                                            int row0, int lane, Release release) {
  const int kv = row0 + lane;
  const int m = kv < p.L ? kv : p.L - 1;  // RoPE position (rows past L are computed, not stored)
#pragma unroll 1
  for (int c = 0; c < NCH; c++) {
    const int n = D - c * 32 < 32 ? D - c * 32 : 32;  // columns of this chunk inside d
    uint32_t v[32];
    tmem_ld32(tl_dk + c * 32, v);
    tmem_ld_wait(v);
    float f[32];
#pragma unroll
    for (int e = 0; e < 32; e++) f[e] = __uint_as_float(v[e]) * p.scale;
    if (p.rope_tab) {  // R^T per pair from the warp-coalesced (cos, sin) table
#pragma unroll
      for (int u = 0; u < 8; u++) {
        if (4 * u >= n) break;
        const float4 cs = p.rope_tab[rope_tab_index(m, D, c * 8 + u)];
        rope_unrotate_pair(f[4 * u], f[4 * u + 1], cs.x, cs.y);
        rope_unrotate_pair(f[4 * u + 2], f[4 * u + 3], cs.z, cs.w);
      }
    }
#pragma unroll
    for (int q = 0; q < 4; q++) {
      if (8 * q >= n) break;
      const int t = 4 * c + q;
      st_shared_v4(stg + lane * 256 + ((t ^ (lane & 7)) << 4), pack_bf16x2(f[8 * q], f[8 * q + 1]),
                   pack_bf16x2(f[8 * q + 2], f[8 * q + 3]), pack_bf16x2(f[8 * q + 4], f[8 * q + 5]),
                   pack_bf16x2(f[8 * q + 6], f[8 * q + 7]));
    }
  }
  release();
  __syncwarp();
  constexpr int PARTS = D / 8;  // 16-byte parts per row: 16 (d = 128), 10 (d = 80)
#pragma unroll 4
  for (int i = lane; i < 32 * PARTS; i += 32) {
    const int r = i / PARTS, t = i - r * PARTS;
    if (row0 + r < p.L)
      *reinterpret_cast<uint4*>(p.dk + ((seq0 + row0 + r) * p.H + h) * D + t * 8) =
          lds_u4(stg + r * 256 + ((t ^ (r & 7)) << 4));
  }
  __syncwarp();  // the staging may be written again
}

// Row-wise forms of the two epilogues: each thread stores its own row (32 lines per store
// instruction of a warp, but no exchange between threads). Measured per main kernel (H = 16,
// d = 128, 65536 tokens), the transposed dV of dv_epilogue is 9% faster in the dQ-owned walk
// (L = 256, where the stores bind), but 4-7% slower in the walk over key tiles at L = 512 and
// 1024: there the P / dS warps' extra exchange before the next item's first P^T is on the
// critical path; the staged dK of dk_epilogue was within +-2% in the walks. The kernel with
// one CTA per key tile (L > 2048 and document-masked chunks) takes both rearranged forms
// (concat-and-chunk step -1.2%).
template <int D, typename Release>
__device__ __forceinline__ void dv_epilogue_rows(const BwdParams& p, uint32_t tl_dv, int qh, long long seq0, int h,
                                                 int kv, Release release) {
  __nv_bfloat16* dst = p.dv + ((seq0 + (kv < p.L ? kv : p.L - 1)) * p.H + h) * D + qh;
#pragma unroll 1
  for (int c = 0; c < 2; c++) {
    const int nvalid = D - (qh + c * 32);  // columns of this chunk inside d (d = 80: 32, 32, 16, none)
    if (nvalid <= 0) break;
    uint32_t v[32];
    tmem_ld32(tl_dv + c * 32, v);
    tmem_ld_wait(v);
    if (kv < p.L) {
      float f[32];
#pragma unroll
      for (int e = 0; e < 32; e++) f[e] = __uint_as_float(v[e]);
      store_row(dst + c * 32, f, nvalid < 32 ? nvalid : 32);
    }
  }
  release();
}

template <int D, int NCH, typename Release>
__device__ __forceinline__ void dk_epilogue_rows(const BwdParams& p, uint32_t tl_dk, long long seq0, int h, int kv,
                                                 Release release) {
  __nv_bfloat16* dst = p.dk + ((seq0 + (kv < p.L ? kv : p.L - 1)) * p.H + h) * D;
#pragma unroll 1
  for (int c = 0; c < NCH; c++) {
    uint32_t v[32];
    tmem_ld32(tl_dk + c * 32, v);
    tmem_ld_wait(v);
    // With RoPE, R^T per pair from the warp-coalesced (cos, sin) table.
    if (kv < p.L)
      store_dk_row32(dst + c * 32, v, p.scale, p.rope_tab, kv, D, c * 8, D - c * 32 < 32 ? D - c * 32 : 32);
  }
  release();
}

}  // namespace ddattn
