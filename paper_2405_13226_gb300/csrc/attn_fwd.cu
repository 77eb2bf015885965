// Causal / document-masked attention forward for sm_103a, two query tiles per work item.
//
// A work item is query tiles 2u and 2u + 1 (256 rows) of one (sequence, head); one CTA
// per SM walks items (see attn_fwd_kernel), so that an item's loads overlap the previous
// item's last softmax steps and epilogue and no CTA launch separates them (at L = 256
// a one-item CTA spent ~2.6 of its ~9.2 us waiting for its first loads and ~0.9 on exit
// and relaunch). Each key / value tile is loaded once for both tiles of an item. The two tiles have their
// own softmax warpgroup, S buffer and O accumulator in TMEM, and the single
// MMA-issuing thread alternates between them:
//   ... PV_0(j-1), S_0(j), PV_1(j-1), S_1(j), PV_0(j), S_0(j+1) ...
// so that while one warpgroup computes the softmax of its tile the tensor core
// works on the other tile's O += P V and next S = Q K^T. Per tile the chain
// softmax -> PV -> S stays serial (P lives over the first 64 columns of the S
// buffer that the next S overwrites; tcgen05.mma of one thread execute in issue
// order, so S_t(j) is issued right behind PV_t(j-1) without waiting for it), but
// the two chains interleave on the tensor core.
//
// Commits: each tcgen05.commit costs the tensor pipe a drain (~200 cycles
// measured, against ~64 per M = N = 128, K = 16 MMA), so there are two per key
// tile, s_full[t] after S_t(j). A commit covers every earlier MMA of the
// thread, so s_full[t] of key tile j also means that PV_t(j-1) is done: the
// softmax then rescales O_t without another wait, and the softmax thread 0 of
// the last tile to read key tile j (value tile j - 1) relays that to the K (V)
// producer with a plain arrive on k_empty (v_empty) of its ring stage. The
// producers cannot wait on s_full themselves: with two ring stages the tensor
// core may complete two phases of it before a producer looks, and a parity wait
// cannot tell those apart. pv_done[t] is committed once per item, after the
// tile's last PV, for the epilogue.
//
// Warp roles (three warpgroups):
//   WG0, WG1  softmax of tile 0 / tile 1: thread r owns query row r of its tile
//             = TMEM lane r. Mask (diagonal / document-edge tiles only), online
//             max and sum in the log2 domain with a lazy rescale of O (only when
//             the running max grows by more than 8: P <= 256 stays exact enough
//             in bf16 / fp32), P as bf16 pairs over the S buffer.
//   WG2       warp 8: K ring producer and TMEM owner; warp 9: V ring producer;
//             warp 10: the MMA issuer; warp 11: Q producer (both tiles of each
//             item). WG2 gives registers back (setmaxnreg.dec) to the softmax
//             groups (setmaxnreg.inc).
// MMA issue: the whole of warp 10 runs the issue loop (waits, descriptor
// arithmetic) and one lane chosen by elect.sync issues each group of MMAs and
// its commit. The same loop run by lane 0 alone inside a divergent branch issued
// 17% slower at L = 8192: that warp shares its SM sub-partition with two busy
// softmax warps, and the divergent form costs more instructions per MMA.
// TMEM (512 columns): S_t at columns 128 t, O_t at 256 + 128 t.
// Key tiles: tile t covers [lo_t, 2u + t] (lo_t: the key tile of the document
// start of its first row); the item walks the union [lo_0, 2u + 1] and each
// tile skips the key tiles outside its own range.
#include "common.cuh"

namespace ddattn {

template <int D>
struct FwdCfg {
  static constexpr int BM = 128, BN = 128, KST = 2, VST = 2;  // the stage-free logic assumes 2 / 2
  static constexpr int DB = (D + 63) / 64;   // 64-column swizzle blocks per row
  static constexpr int DCH = (D + 31) / 32;  // 32-column TMEM chunks of O
  static constexpr int Q_BLK = BM * 128;
  static constexpr int KV_BLK = BN * 128;
  static constexpr int Q_BYTES = DB * Q_BLK;
  static constexpr int KV_BYTES = DB * KV_BLK;
  static constexpr int OFF_Q = 0;  // two tiles
  static constexpr int OFF_K = OFF_Q + 2 * Q_BYTES;
  static constexpr int OFF_V = OFF_K + KST * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + VST * KV_BYTES;
  static constexpr int OFF_OST = OFF_BAR + 1024;  // RoPE forms: O staging, 4 KB per softmax warp (32 x 64)
  static constexpr int SMEM_BYTES = OFF_BAR + 512 + 1024;
  static constexpr int SMEM_BYTES_ROPE = OFF_OST + 8 * 4096 + 1024;
  static constexpr int PF = 4;  // K / V tiles prefetched into L2 ahead of the ring
  static constexpr uint32_t TMEM_S = 0, TMEM_O = 256, TMEM_COLS = 512;
  static constexpr int THREADS = 384;  // the RoPE forms add a rotation warpgroup: 512
  // setmaxnreg split (the spill-free one for each head dim under ptxas 13.0); REGS_ROT: the
  // rotation warpgroup of the RoPE forms
  static constexpr int REGS_LOW = D == 128 ? 80 : 72, REGS_HIGH = D == 128 ? 184 : 192;
  static constexpr int REGS_ROT = D == 128 ? 64 : 56;
};
// The split must fit in the launch's 384 threads x 168 registers (512 x 128 with RoPE).
static_assert(128 * FwdCfg<128>::REGS_LOW + 256 * FwdCfg<128>::REGS_HIGH <= 384 * 168, "register split");
static_assert(128 * FwdCfg<64>::REGS_LOW + 256 * FwdCfg<64>::REGS_HIGH <= 384 * 168, "register split");
static_assert(128 * (FwdCfg<128>::REGS_LOW + FwdCfg<128>::REGS_ROT) + 256 * FwdCfg<128>::REGS_HIGH <= 512 * 128,
              "register split");
static_assert(128 * (FwdCfg<64>::REGS_LOW + FwdCfg<64>::REGS_ROT) + 256 * FwdCfg<64>::REGS_HIGH <= 512 * 128,
              "register split");

// RoPE forms of the forward kernel: none (q, k given rotated, or no RoPE); Q tiles rotated in
// shared memory as they land (k given rotated); Q and K tiles rotated as they land.
enum FwdRope { kRopeNone = 0, kRopeQ = 1, kRopeQK = 2 };
__host__ __device__ constexpr int fwd_threads(int rope) { return rope ? 512 : 384; }


// The item ring: warp 11 claims each next item and publishes its index to the roles that
// read it: the K and V producer lanes, the 32 lanes of the MMA warp and the 256 softmax
// threads, each of which arrives on item_empty after reading.
// The RoPE forms add the 128 rotation threads.
constexpr int kItemRing = 4;
__host__ __device__ constexpr int fwd_item_readers(int rope) { return 1 + 1 + 32 + 256 + (rope ? 128 : 0); }

struct FwdBars {
  uint64_t item_full[kItemRing], item_empty[kItemRing];
  int item[kItemRing];  // -1: no more items
  uint64_t q_full[2], q_empty[2];
  uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2];
  uint64_t s_full[2], p_full[2], pv_done[2];
  uint64_t mma_drain;
  uint64_t q_rot[2], k_rot[2];  // RoPE forms: Q_t / the K stage has been rotated in shared memory
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(FwdBars) <= 512, "barrier block");
static_assert(FwdCfg<128>::KST == 2 && FwdCfg<128>::VST == 2, "ring barriers");

// A work item: query tiles 2u and 2u + 1 of one (sequence, head). Items are numbered pair
// fastest, heaviest pair (largest u) first.
struct FwdItem {
  int u, h, b;
  long long seq0;
  bool has1;              // an odd tile count leaves the last pair one tile
  int lo0, lo1, hi0, hi1; // key-tile range [lo_t, hi_t] of tile t; lo_0 <= lo_1 (documents start in order)
  int J0, NJ;             // the key tiles the item walks: J0 .. J0 + NJ - 1
};
__device__ __forceinline__ FwdItem fwd_item(const FwdParams& p, int it) {
  constexpr int BM = 128, BN = 128;
  const int nqp = (p.nqt + 1) >> 1;
  FwdItem I;
  I.u = nqp - 1 - it % nqp;
  I.h = (it / nqp) % p.H;
  I.b = it / (nqp * p.H);
  I.seq0 = (long long)I.b * p.L;
  I.has1 = 2 * I.u + 1 < p.nqt;
  const int r1c = (2 * I.u + 1) * BM < p.L ? (2 * I.u + 1) * BM : p.L - 1;
  I.lo0 = (int)(doc_start(p.offsets, p.n_offsets, I.seq0 + 2 * I.u * BM, I.seq0) - I.seq0) / BN;
  I.lo1 = (int)(doc_start(p.offsets, p.n_offsets, I.seq0 + r1c, I.seq0) - I.seq0) / BN;
  I.hi0 = 2 * I.u;
  I.hi1 = 2 * I.u + 1;
  I.J0 = I.lo0;
  I.NJ = (I.has1 ? I.hi1 : I.hi0) - I.J0 + 1;
  return I;
}

// A CTA per SM walks items, starting with item blockIdx.x; each next item is claimed from a
// global counter (item G + count) when the CTA starts loading the previous one, so items
// spread over the CTAs as they free up, whatever their cost (with document masks it varies
// with the documents). Items are numbered sequence and head slowest, so the CTAs working at
// one time share each sequence's K / V tiles in L2. Over four DM steps (8 x 8192) a static
// assignment (items c, c + G, ...) was 8-10% slower than one CTA per item and claiming
// 0-4%; over the plain buckets claiming was within 0-2% of static. The K / V
// rings, Q buffers and per-tile barrier phases run on across items:
//   * ring position jg counts the key tiles the CTA has loaded; stage jg % 2, parity
//     (jg / 2) % 2, in every role;
//   * Q_t of an item is loaded (by warp 11) once the previous item's last S_t has
//     completed: the softmax thread that sees that S's commit relays it on q_empty[t];
//   * the relays of K / V ring stages are those of one item, plus, after pv_done, the
//     value tile whose last reader no S commit of the item covers: the item's last one,
//     and tile 0's last one when tile 1's document starts at tile 1 (then tile 1 reads
//     none of it);
//   * an item's first PV into O_t needs no barrier of its own: it waits for that item's
//     first p_full[t], which the tile's softmax group arrives only after its epilogue of
//     the previous item has read O_t out.
// A CPU discrete-event model of this protocol (random walks, random document starts,
// random timings) runs in tests/test_fwd_walk_protocol.py.
// The n-th item of a CTA from its item ring, for a role whose whole warp waits (-1: no
// more items, or the CTA was aborted: then ok is false).
__device__ __forceinline__ int fwd_next_item(FwdBars* bars, int n, bool& ok, const Watchdog& wd) {
  const int slot = n & (kItemRing - 1);
  ok = __all_sync(0xffffffffu, ok && mbar_wait(&bars->item_full[slot], (n / kItemRing) & 1, wd));
  if (!ok) return -1;
  const int it = *reinterpret_cast<volatile int*>(&bars->item[slot]);
  mbar_arrive(&bars->item_empty[slot]);
  return it;
}

// RoPE of one 128-row tile in shared memory, in place: row r holds position pos0 + r and
// each pair (x_2j, x_2j+1) becomes (x_2j c - x_2j+1 s, x_2j s + x_2j+1 c), c, s = cos, sin
// of (pos0 + r) theta_j, in fp32, rounded to bf16 (rope_rotate_bf16x2, the arithmetic of
// dd_rope_qk). Rows at or past L are TMA zero fill and stay as they are. With gdst set
// the rotated rows below L are also written to global memory (gdst: element 0 of row pos0,
// rows `rs` elements apart). Thread t of the 128 takes the 16-byte chunk c = t % 16
// (columns 8c .. 8c + 7: pairs 4c .. 4c + 3) of rows g, g + 8, ..., g + 120 (g = t / 16),
// which share one swizzled chunk position (the 128B swizzle XORs the chunk index with
// row % 8 = g). Its (cos, sin) start from the table row of position pos0 + g (the values
// dd_rope_qk uses) and advance eight positions per row by the angle-sum step with
// (C, S) = (cos, sin) of 8 theta_j (table row 8): after up to 15 steps they are within a
// few 1e-7 of the table's, so a rotated value can differ from dd_rope_qk's in its last bit
// where the fp32 result lies that close to a bf16 rounding boundary (rare).
template <int D>
__device__ __forceinline__ void rope_step8(const FwdParams& p, int t, float (&stc)[4], float (&sts)[4]) {
  const int c = t & 15;
#pragma unroll
  for (int e = 0; e < 4; e++) {
    stc[e] = 1.f;
    sts[e] = 0.f;
  }
  if (p.L > 8 && c < D / 8) {  // with L <= 8 no thread steps past its first row
#pragma unroll
    for (int e = 0; e < 4; e++) {
      const float2 v = __ldg(p.rope_rows + 8 * (D / 2) + 4 * c + e);
      stc[e] = v.x;
      sts[e] = v.y;
    }
  }
}
template <int D>
__device__ __forceinline__ void rope_rotate_tile(uint8_t* tile, int pos0, int L, const float2* tab,
                                                 const float (&stc)[4], const float (&sts)[4], __nv_bfloat16* gdst,
                                                 long long rs, int t) {
  const int c = t & 15, g = t >> 4;
  if (c >= D / 8 || pos0 + g >= L) return;
  const uint32_t base = smem_u32(tile) + (uint32_t)(c >> 3) * (128u * 128u) + sw128_offset((uint32_t)g, c & 7);
  const float4* t4 = reinterpret_cast<const float4*>(tab + (long long)(pos0 + g) * (D / 2) + 4 * c);
  const float4 a = __ldg(t4), b = __ldg(t4 + 1);
  float cv[4] = {a.x, a.z, b.x, b.z}, sv[4] = {a.y, a.w, b.y, b.w};
#pragma unroll 2
  for (int k = 0; k < 16; k++) {
    const int r = g + 8 * k;
    if (pos0 + r >= L) break;
    const uint32_t addr = base + (uint32_t)k * 1024u;  // eight rows on: the same swizzle phase
    const float4 x4 = lds_f4(addr);
    uint32_t w[4] = {__float_as_uint(x4.x), __float_as_uint(x4.y), __float_as_uint(x4.z), __float_as_uint(x4.w)};
#pragma unroll
    for (int e = 0; e < 4; e++) {
      w[e] = rope_rotate_bf16x2(__uint_as_float(w[e] << 16), __uint_as_float(w[e] & 0xffff0000u), cv[e], sv[e]);
      const float cn = fmaf(cv[e], stc[e], -sv[e] * sts[e]);
      sv[e] = fmaf(sv[e], stc[e], cv[e] * sts[e]);
      cv[e] = cn;
    }
    st_shared_v4(addr, w[0], w[1], w[2], w[3]);
    if (gdst) *reinterpret_cast<uint4*>(gdst + r * rs + 8 * c) = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

template <int D, int ROPE>
__global__ void __launch_bounds__(fwd_threads(ROPE), 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmO,
                    const FwdParams p) {
  using C = FwdCfg<D>;
  constexpr int KST = C::KST, VST = C::VST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  FwdBars* bars = reinterpret_cast<FwdBars*>(smem + C::OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int nqp = (p.nqt + 1) >> 1;
  const int n_items = nqp * p.H * p.B;
  Watchdog wd{&bars->abort_flag, p.status, p.timeout_ns};

  if (threadIdx.x == 0) {
    bars->abort_flag = 0;
    for (int i = 0; i < kItemRing; i++) {
      mbar_init(&bars->item_full[i], 1);
      mbar_init(&bars->item_empty[i], fwd_item_readers(ROPE));
    }
    for (int t = 0; t < 2; t++) {
      mbar_init(&bars->q_full[t], 1);
      mbar_init(&bars->q_empty[t], 1);
      mbar_init(&bars->s_full[t], 1);
      mbar_init(&bars->p_full[t], 4);  // per-warp arrivals (mbar_arrive_warp)
      mbar_init(&bars->pv_done[t], 1);
    }
    for (int i = 0; i < 2; i++) {
      mbar_init(&bars->k_full[i], 1);
      mbar_init(&bars->k_empty[i], 1);
      mbar_init(&bars->v_full[i], 1);
      mbar_init(&bars->v_empty[i], 1);
      mbar_init(&bars->q_rot[i], 4);
      mbar_init(&bars->k_rot[i], 4);
    }
    mbar_init(&bars->mma_drain, 1);
    fence_mbar_init();
  }
  if (warp == 8) {
    tmem_alloc(&bars->tmem_base, C::TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  const int wg = warp >> 2;

  if (wg == 2) {
  setmaxnreg_dec<C::REGS_LOW>();
  if (warp == 8 || warp == 9) {
    // ---------------- K (warp 8) / V (warp 9) ring producer; jg = ring position
    if (lane == 0) {
      const bool isk = warp == 8;
      const CUtensorMap* tm = isk ? &tmK : &tmV;
      uint8_t* sR = isk ? sK : sV;
      uint64_t* full = isk ? bars->k_full : bars->v_full;
      uint64_t* empty = isk ? bars->k_empty : bars->v_empty;
      prefetch_tmap(tm);
      int jg = 0;
      bool ok = true;
      for (int n = 0; ok; n++) {
        const int slot = n & (kItemRing - 1);
        if (!(ok = mbar_wait(&bars->item_full[slot], (n / kItemRing) & 1, wd))) break;
        const int it = *reinterpret_cast<volatile int*>(&bars->item[slot]);
        mbar_arrive(&bars->item_empty[slot]);
        if (it < 0) break;
        const FwdItem I = fwd_item(p, it);
        for (int j = 0; j < I.NJ; j++, jg++) {
          const int s = jg & 1;
          if (jg >= KST && !(ok = mbar_wait(&empty[s], ((jg >> 1) - 1) & 1, wd))) break;
          mbar_arrive_expect_tx(&full[s], C::KV_BYTES);
          const int kv0 = (I.J0 + j) * C::BN;
          for (int blk = 0; blk < C::DB; blk++)
            tma_load_4d(sR + s * C::KV_BYTES + blk * C::KV_BLK, tm, &full[s], 64 * blk, I.h, kv0, I.b);
          if (j + C::PF < I.NJ)
            for (int blk = 0; blk < C::DB; blk++) tma_prefetch_4d(tm, 64 * blk, I.h, kv0 + C::PF * C::BN, I.b);
        }
      }
      // Every copy lands before the CTA can exit (after an abort nobody else waits for them).
      for (int j = jg - KST < 0 ? 0 : jg - KST; j < jg; j++) mbar_wait_drain(&full[j & 1], (j >> 1) & 1, wd.limit_ns);
    }
  } else if (warp == 11) {
    // ---------------- Q producer: Q_t of an item once the previous one's last S_t is done
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      int nload[2] = {0, 0};
      bool ok = true;
      int it = blockIdx.x;
      for (int n = 0; ok; n++) {
        const int slot = n & (kItemRing - 1);
        if (n >= kItemRing && !(ok = mbar_wait(&bars->item_empty[slot], ((n / kItemRing) - 1) & 1, wd))) break;
        *reinterpret_cast<volatile int*>(&bars->item[slot]) = it < n_items ? it : -1;
        mbar_arrive(&bars->item_full[slot]);  // release: the index is visible to the waiting roles
        if (it >= n_items) break;
        const FwdItem I = fwd_item(p, it);
#pragma unroll
        for (int t = 0; t < 2; t++) {
          if (!ok || !(t == 0 || I.has1)) continue;
          if (nload[t] > 0 && !(ok = mbar_wait(&bars->q_empty[t], (nload[t] - 1) & 1, wd))) break;
          mbar_arrive_expect_tx(&bars->q_full[t], C::Q_BYTES);
          for (int blk = 0; blk < C::DB; blk++)
            tma_load_4d(sQ + t * C::Q_BYTES + blk * C::Q_BLK, &tmQ, &bars->q_full[t], 64 * blk, I.h,
                        (2 * I.u + t) * C::BM, I.b);
          nload[t]++;
        }
        it = (int)gridDim.x + (int)atomicAdd(p.work_ctr, 1u);
      }
#pragma unroll
      for (int t = 0; t < 2; t++)
        if (nload[t] > 0) mbar_wait_drain(&bars->q_full[t], (nload[t] - 1) & 1, wd.limit_ns);
    }
  } else if (warp == 10) {
    // ---------------- MMA issuer: the whole warp runs the loop, one elected lane issues
    {
      const bool leader = elect_one();
      constexpr uint32_t idesc_s = idesc_bf16(128, 128, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16(128, D, false, true);      // P (TMEM) x V (MN-major)
      // Descriptors built once; a K-slice, ring stage or tile is an added (byte offset >> 4).
      const uint64_t dQ0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t dK0 = sdesc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t dV0 = sdesc_sw128(smem_u32(sV), C::KV_BLK, 1024);
      // Running counts (static indices only): PV issued per tile, items per tile; per item:
      // S and PV issued per tile.
      int npv[2] = {0, 0}, nit[2] = {0, 0};
      int jg0 = 0;
      bool ok = true;
      for (int n = 0; ok; n++) {
      const int it = fwd_next_item(bars, n, ok, wd);
      if (it < 0) break;
      const FwdItem I = fwd_item(p, it);
      const bool has1 = I.has1;
      const int lo0 = I.lo0, lo1 = I.lo1, hi0 = I.hi0, hi1 = I.hi1, J0 = I.J0, NJ = I.NJ;
      int ns_i[2] = {0, 0}, npv_i[2] = {0, 0};
      for (int j = 0; j <= NJ && ok; j++) {
        const int kt = J0 + j;
#pragma unroll
        for (int t = 0; t < 2; t++) {
          const bool tile = t == 0 || has1;
          const int lo_t = t ? lo1 : lo0, hi_t = t ? hi1 : hi0;
          // O_t += P_t V_{j-1}
          if (ok && tile && j >= 1 && kt - 1 >= lo_t && kt - 1 <= hi_t) {
            const int jv = jg0 + j - 1;
            ok = __all_sync(0xffffffffu, mbar_wait(&bars->v_full[jv & 1], (jv >> 1) & 1, wd) &&
                                             mbar_wait(&bars->p_full[t], npv[t] & 1, wd));
          }
          if (ok && tile && j >= 1 && kt - 1 >= lo_t && kt - 1 <= hi_t) {
            const int vs = (jg0 + j - 1) & 1;
            tc_fence_after();
            const uint64_t dV = dV0 + ((uint32_t)(vs * C::KV_BYTES) >> 4);
            const uint32_t tP = tmem + C::TMEM_S + t * 128;
            if (leader) {
#pragma unroll
              for (int kk = 0; kk < C::BN / 16; kk++)
                umma_bf16_ts(tmem + C::TMEM_O + t * 128, tP + kk * 8, dV + (uint32_t)((kk * 2048) >> 4), idesc_o,
                             (npv_i[t] > 0 || kk > 0) ? 1u : 0u);
              if (kt - 1 == hi_t) umma_commit(&bars->pv_done[t]);  // the tile's last PV: for the epilogue
            }
            __syncwarp();
            npv[t]++;
            npv_i[t]++;
          }
          // S_t = Q_t K_j^T into the buffer PV_t has just read (issue order keeps them apart)
          if (ok && tile && j < NJ && kt >= lo_t && kt <= hi_t) {
            const int jk = jg0 + j;
            // With RoPE the rotation warpgroup's q_rot / k_rot follow q_full / k_full.
            uint64_t* kb = ROPE == kRopeQK ? &bars->k_rot[jk & 1] : &bars->k_full[jk & 1];
            uint64_t* qb = ROPE ? &bars->q_rot[t] : &bars->q_full[t];
            ok = __all_sync(0xffffffffu, mbar_wait(kb, (jk >> 1) & 1, wd) &&
                                             (ns_i[t] > 0 || mbar_wait(qb, nit[t] & 1, wd)));
          }
          if (ok && tile && j < NJ && kt >= lo_t && kt <= hi_t) {
            const int ks = (jg0 + j) & 1;
            tc_fence_after();
            const uint64_t dQ = dQ0 + ((uint32_t)(t * C::Q_BYTES) >> 4);
            const uint64_t dK = dK0 + ((uint32_t)(ks * C::KV_BYTES) >> 4);
            const uint32_t tS = tmem + C::TMEM_S + t * 128;
            if (leader) {
#pragma unroll
              for (int kk = 0; kk < D / 16; kk++) {
                constexpr int q_blk = C::Q_BLK, kv_blk = C::KV_BLK;
                umma_bf16(tS, dQ + (uint32_t)(((kk >> 2) * q_blk + (kk & 3) * 32) >> 4),
                          dK + (uint32_t)(((kk >> 2) * kv_blk + (kk & 3) * 32) >> 4), idesc_s, kk > 0 ? 1u : 0u);
              }
              umma_commit(&bars->s_full[t]);
            }
            __syncwarp();
            ns_i[t]++;
          }
        }
      }
      nit[0]++;
      if (has1) nit[1]++;
      jg0 += NJ;
      }
      if (leader) umma_commit(&bars->mma_drain);
      __syncwarp();
      mbar_wait_drain(&bars->mma_drain, 0, wd.limit_ns);
    }
  }
  } else if (ROPE && wg == 3) {
  setmaxnreg_dec<C::REGS_ROT>();
  // ---------------- rotation warpgroup (RoPE forms): in the order the MMA thread needs them,
  // Q_0 of an item, its first key tile, Q_1, then its other key tiles (key tiles with
  // kRopeQK only), each rotated in place as soon as its TMA copy has landed and released
  // with q_rot / k_rot (fence.proxy.async first: the tensor core reads these generic-proxy
  // writes). Every Q tile also goes to q_rot in global memory for the backward, and every
  // key tile to k_rot from the one item on whose diagonal it lies (key tile 2u or 2u + 1 of
  // item u).
  {
    const int t = threadIdx.x - 384;
    float stc[4], sts[4];
    rope_step8<D>(p, t, stc, sts);
    const long long rs = (long long)p.H * D;  // elements between rows of q / k
    int nq[2] = {0, 0}, jg = 0;
    bool ok = true;
    for (int n = 0; ok; n++) {
      const int it = fwd_next_item(bars, n, ok, wd);
      if (it < 0) break;
      const FwdItem I = fwd_item(p, it);
      const long long row_base = ((long long)I.b * p.L) * p.H + I.h;  // (b, position 0, h) in rows of d
      // e = 0: Q_0; e = 1: key tile J0; e = 2: Q_1; e >= 3: key tile J0 + e - 2.
      for (int e = 0; e < I.NJ + 2 && ok; e++) {
        if (e == 0 || e == 2) {
          const int tq = e / 2;
          if (tq == 1 && !I.has1) continue;
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_full[tq], nq[tq] & 1, wd)))) break;
          const int pos0 = (2 * I.u + tq) * C::BM;
          rope_rotate_tile<D>(sQ + tq * C::Q_BYTES, pos0, p.L, p.rope_rows, stc, sts,
                              p.q_rot + (row_base + (long long)pos0 * p.H) * D, rs, t);
          fence_proxy_async_smem();
          mbar_arrive_warp(&bars->q_rot[tq]);
          nq[tq]++;
        } else if (ROPE == kRopeQK) {
          const int jj = e == 1 ? 0 : e - 2;
          const int jk = jg + jj;
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->k_full[jk & 1], (jk >> 1) & 1, wd)))) break;
          const int kt = I.J0 + jj;
          const int pos0 = kt * C::BN;
          const bool diag = kt == 2 * I.u || (I.has1 && kt == 2 * I.u + 1);
          rope_rotate_tile<D>(sK + (jk & 1) * C::KV_BYTES, pos0, p.L, p.rope_rows, stc, sts,
                              diag ? p.k_rot + (row_base + (long long)pos0 * p.H) * D : nullptr, rs, t);
          fence_proxy_async_smem();
          mbar_arrive_warp(&bars->k_rot[jk & 1]);
        }
      }
      jg += I.NJ;
    }
  }
  } else {
  setmaxnreg_inc<C::REGS_HIGH>();
  // ---------------- softmax of tile t = wg: thread r <-> query row r <-> TMEM lane r
  const int t = wg;
  const int r = threadIdx.x & 127;
  const uint32_t tl = tmem + ((uint32_t)((warp & 3) * 32) << 16);
  const uint32_t sbuf = tl + C::TMEM_S + t * 128;
  const uint32_t obuf = tl + C::TMEM_O + t * 128;
  const float sl2 = p.scale_log2;
  const uint64_t sl2x2 = f32x2(sl2, sl2);
  int jg0 = 0, nit = 0, ns = 0;  // ring position of the item's first key tile, items of this tile, S seen
  bool ok = true;
  for (int n = 0; ok; n++) {
  const int it = fwd_next_item(bars, n, ok, wd);
  if (it < 0) break;
  const FwdItem I = fwd_item(p, it);
  if (!(t == 0 || I.has1)) {
    jg0 += I.NJ;
    continue;
  }
  const bool has1 = I.has1;
  const int lo1 = I.lo1, J0 = I.J0, h = I.h, b = I.b;
  const long long seq0 = I.seq0;
  const int row0 = (2 * I.u + t) * C::BM;
  const int row = row0 + r;
  const int rowc = row < p.L ? row : p.L - 1;
  const int lo_t = t ? I.lo1 : I.lo0, hi_t = t ? I.hi1 : I.hi0;
  const int nt = hi_t - lo_t + 1;
  const int ds = (int)(doc_start(p.offsets, p.n_offsets, seq0 + rowc, seq0) - seq0);
  float m_run = -INFINITY, l_run = 0.f;
  for (int i = 0; i < nt && ok; i++) {
    const int kv0 = (lo_t + i) * C::BN;
    ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full[t], ns & 1, wd));
    if (!ok) break;
    ns++;
    tc_fence_after();
    if (r == 0) {  // relay: this tile is the last reader of key tile kt / value tile kt - 1
      const int kt = lo_t + i, jk = jg0 + kt - J0;
      if (t == 1 || !(has1 && kt >= lo1)) mbar_arrive(&bars->k_empty[jk & 1]);
      if (i >= 1 && (t == 1 || !(has1 && kt - 1 >= lo1))) mbar_arrive(&bars->v_empty[(jk - 1) & 1]);
      if (i == nt - 1) mbar_arrive(&bars->q_empty[t]);  // the tile's last S is done: Q_t may be replaced
    }
    uint32_t v0[32], v1[32], v2[32], v3[32];
    tmem_ld32(sbuf + 0, v0);
    tmem_ld32(sbuf + 32, v1);
    tmem_ld32(sbuf + 64, v2);
    tmem_ld32(sbuf + 96, v3);
    tmem_ld_wait(v0);
    tmem_ld_wait(v1);
    tmem_ld_wait(v2);
    tmem_ld_wait(v3);
    float sc[128];
#pragma unroll
    for (int c = 0; c < 32; c++) {
      sc[c] = __uint_as_float(v0[c]);
      sc[32 + c] = __uint_as_float(v1[c]);
      sc[64 + c] = __uint_as_float(v2[c]);
      sc[96 + c] = __uint_as_float(v3[c]);
    }
    if (kv0 + C::BN - 1 > row || kv0 < ds) {
#pragma unroll
      for (int c = 0; c < 128; c++) {
        const int kv = kv0 + c;
        if (kv > row || kv < ds) sc[c] = -INFINITY;
      }
    }
    // Row max as eight independent 3-input max chains over 16 columns each, then a tree:
    // the critical path is ~10 dependent instructions instead of a 127-long chain.
    float mq[8];
#pragma unroll
    for (int q = 0; q < 8; q++) {
      float m = fmax3(sc[16 * q], sc[16 * q + 1], sc[16 * q + 2]);
#pragma unroll
      for (int e = 3; e < 15; e += 2) m = fmax3(m, sc[16 * q + e], sc[16 * q + e + 1]);
      mq[q] = fmaxf(m, sc[16 * q + 15]);
    }
    const float mx = fmax3(fmax3(mq[0], mq[1], mq[2]), fmax3(mq[3], mq[4], mq[5]), fmaxf(mq[6], mq[7]));
    const float m_tile = mx * sl2;
    float alpha = 1.f;
    bool rescale = false;
    if (m_tile > m_run + 8.f) {
      alpha = exp2_approx(m_run - m_tile);  // 0 when m_run = -inf
      rescale = (i > 0);
      m_run = m_tile;
    }
    const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
    const uint64_t negm = f32x2(-m_use, -m_use);
    uint64_t rs2[4] = {f32x2(0.f, 0.f), f32x2(0.f, 0.f), f32x2(0.f, 0.f), f32x2(0.f, 0.f)};  // 4 sum chains
    uint32_t pk0[32], pk1[32];
#pragma unroll
    for (int c = 0; c < 64; c++) {
      const uint64_t x = fma_f32x2(f32x2(sc[2 * c], sc[2 * c + 1]), sl2x2, negm);
      const float p0 = exp2_approx(f32x2_lo(x));
      const float p1 = exp2_approx(f32x2_hi(x));
      rs2[c & 3] = add_f32x2(rs2[c & 3], f32x2(p0, p1));
      if (c < 32) pk0[c] = pack_bf16x2(p0, p1);
      else pk1[c - 32] = pack_bf16x2(p0, p1);
    }
    const uint64_t rsum = add_f32x2(add_f32x2(rs2[0], rs2[1]), add_f32x2(rs2[2], rs2[3]));
    l_run = l_run * alpha + (f32x2_lo(rsum) + f32x2_hi(rsum));
    tmem_st32(sbuf + 0, pk0);
    tmem_st32(sbuf + 32, pk1);
    // O_t *= alpha. PV_t of the previous key tile has completed: it was issued
    // before S_t of this one, whose commit (s_full, waited above) covers it.
    if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll 1
      for (int c = 0; c < C::DCH; c++) {
        uint32_t ov[32];
        tmem_ld32(obuf + c * 32, ov);
        tmem_ld_wait(ov);
#pragma unroll
        for (int e = 0; e < 32; e++) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
        tmem_st32(obuf + c * 32, ov);
      }
    }
    tmem_st_wait();
    tc_fence_before();
    mbar_arrive_warp(&bars->p_full[t]);
  }
  // Epilogue: O / l -> bf16, LSE = (m + log2 l) * ln2.
  if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->pv_done[t], nit & 1, wd));
  if (ok) {
    tc_fence_after();
    // The value tile whose last reader no S commit of the item covers: the item's last
    // one (tile 1's, or tile 0's without a tile 1), and tile 0's last one when tile 1's
    // document starts at tile 1 (tile 1 reads none of it).
    if (r == 0 && (t == (has1 ? 1 : 0) || (t == 0 && has1 && lo1 > I.hi0)))
      mbar_arrive(&bars->v_empty[(jg0 + hi_t - J0) & 1]);
    const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
    const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
    // The RoPE forms: O leaves through shared memory and tensor stores; the plain forward keeps
    // each thread's own row stores. Measured per forward (H = 16, d = 128, 65536 tokens), tensor
    // stores made the RoPE forward 12% / 5% faster at L = 256 / 512 (its rotation warpgroup
    // also stores rows), the plain one 3-4% slower at L = 256 / 512 and 1-2% faster from
    // L = 4096 and on the concat-and-chunk step; choosing at run time slowed the plain kernel
    // by 4-6% at L = 512..2048.
    if constexpr (ROPE != kRopeNone) {
      // O / l -> bf16 through this warp's 4 KB staging block: its 32 rows x 64 columns in the O
      // map's 128-byte swizzled layout (16-byte chunk j of row r at r * 128 + ((j ^ (r & 7)) * 16),
      // conflict-free), then one tensor store per 64 columns, which clips rows past L and
      // columns past d and writes whole lines (rows are H d elements apart, so each store
      // instruction of a warp storing its own rows touches 32 lines).
      const uint32_t ost = smem_u32(smem + C::OFF_OST) + (uint32_t)(t * 4 + (warp & 3)) * 4096u;
      const int lr = r & 31;  // the thread's row within its warp's 32
#pragma unroll 1
      for (int hf = 0; hf < C::DB; hf++) {
        if (lane == 0) bulk_wait_read<0>();  // the previous tensor store has read the block
        __syncwarp();
#pragma unroll 1
        for (int cc = 0; cc < 2 && 2 * hf + cc < C::DCH; cc++) {
          uint32_t ov[32];
          tmem_ld32(obuf + (2 * hf + cc) * 32, ov);
          tmem_ld_wait(ov);
#pragma unroll
          for (int q = 0; q < 4; q++) {
            const int j = 4 * cc + q;
            st_shared_v4(ost + lr * 128 + ((j ^ (lr & 7)) << 4),
                         pack_bf16x2(__uint_as_float(ov[8 * q + 0]) * inv_l, __uint_as_float(ov[8 * q + 1]) * inv_l),
                         pack_bf16x2(__uint_as_float(ov[8 * q + 2]) * inv_l, __uint_as_float(ov[8 * q + 3]) * inv_l),
                         pack_bf16x2(__uint_as_float(ov[8 * q + 4]) * inv_l, __uint_as_float(ov[8 * q + 5]) * inv_l),
                         pack_bf16x2(__uint_as_float(ov[8 * q + 6]) * inv_l, __uint_as_float(ov[8 * q + 7]) * inv_l));
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          tma_store_4d(&tmO, smem + C::OFF_OST + (t * 4 + (warp & 3)) * 4096, 64 * hf, h, row0 + 32 * (warp & 3), b);
          bulk_commit();
        }
      }
    } else {
      __nv_bfloat16* orow = p.o + (((long long)b * p.L + rowc) * p.H + h) * D;
#pragma unroll 1
      for (int c = 0; c < C::DCH; c++) {
        uint32_t ov[32];
        tmem_ld32(obuf + c * 32, ov);
        tmem_ld_wait(ov);
        if (row < p.L) {
          uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
          const int nv = (D - c * 32 >= 32) ? 4 : (D - c * 32) / 8;  // 16-byte stores in this chunk
#pragma unroll
          for (int q = 0; q < 4; q++) {
            if (q >= nv) break;
            uint4 w;
            w.x = pack_bf16x2(__uint_as_float(ov[8 * q + 0]) * inv_l, __uint_as_float(ov[8 * q + 1]) * inv_l);
            w.y = pack_bf16x2(__uint_as_float(ov[8 * q + 2]) * inv_l, __uint_as_float(ov[8 * q + 3]) * inv_l);
            w.z = pack_bf16x2(__uint_as_float(ov[8 * q + 4]) * inv_l, __uint_as_float(ov[8 * q + 5]) * inv_l);
            w.w = pack_bf16x2(__uint_as_float(ov[8 * q + 6]) * inv_l, __uint_as_float(ov[8 * q + 7]) * inv_l);
            dst[q] = w;
          }
        }
      }
    }
    if (row < p.L)
      p.lse[((long long)b * p.H + h) * p.L + row] = l_run > 0.f ? (m_use + __log2f(l_run)) * kLn2 : -INFINITY;
  }
  nit++;
  jg0 += I.NJ;
  }
  if (ROPE != kRopeNone && lane == 0) bulk_wait<0>();  // this warp's tensor stores of O have landed
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D, int ROPE>
static cudaError_t launch_fwd_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& to, const FwdParams& p, cudaStream_t stream) {
  using C = FwdCfg<D>;
  static DeviceCache nsm_dev;
  int nsm = 0;
  constexpr int smem_bytes = ROPE != kRopeNone ? C::SMEM_BYTES_ROPE : C::SMEM_BYTES;
  cudaError_t e = kernel_setup(nsm_dev, attn_fwd_kernel<D, ROPE>, smem_bytes, &nsm);
  if (e != cudaSuccess) return e;
  // One CTA per SM (shared memory allows no more) walking items: the first G in order, the
  // rest claimed. G is kept coprime with the pairs per (sequence, head), so the first round
  // of items mixes pair positions (their key-tile counts differ).
  const int nqp = (p.nqt + 1) / 2;
  const long long items = (long long)nqp * p.H * p.B;
  if (items > 2147483647LL - 4096) return cudaErrorInvalidValue;  // item indices (and claims past the end) are int
  long long G = items < nsm ? items : nsm;
  auto gcd = [](long long x, long long y) {
    while (y) {
      const long long t = x % y;
      x = y;
      y = t;
    }
    return x;
  };
  while (G > 1 && gcd(G, nqp) != 1) G--;
  if ((e = cudaMemsetAsync(p.work_ctr, 0, sizeof(unsigned int), stream)) != cudaSuccess) return e;  // the claim counter
  attn_fwd_kernel<D, ROPE><<<(unsigned)G, fwd_threads(ROPE), smem_bytes, stream>>>(tq, tk, tv, to, p);
  return cudaGetLastError();
}

template <int D>
static cudaError_t launch_fwd_rope(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                   const CUtensorMap& to, const FwdParams& p, int rope, cudaStream_t stream) {
  if (rope == kRopeQK) return launch_fwd_d<D, kRopeQK>(tq, tk, tv, to, p, stream);
  if (rope == kRopeQ) return launch_fwd_d<D, kRopeQ>(tq, tk, tv, to, p, stream);
  return launch_fwd_d<D, kRopeNone>(tq, tk, tv, to, p, stream);
}

cudaError_t launch_attn_fwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& to, const FwdParams& p, int rope, cudaStream_t stream) {
  if (d == 64) return launch_fwd_rope<64>(tq, tk, tv, to, p, rope, stream);
  if (d == 80) return launch_fwd_rope<80>(tq, tk, tv, to, p, rope, stream);
  return launch_fwd_rope<128>(tq, tk, tv, to, p, rope, stream);
}

}  // namespace ddattn
