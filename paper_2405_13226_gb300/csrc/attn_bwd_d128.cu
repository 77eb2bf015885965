// Attention backward main kernel for head dims 128 and 80 on sm_103a.
//
// One CTA per 128-key tile of one (sequence, head), walking the live 128-row
// query tiles from the diagonal to the end of the tile's last document (the
// backward counterpart of the forward's tile skipping). Per query step i:
//   S^T  = K Q_i^T            P^T  = exp2(S^T * scale * log2e - LSE_i * log2e)  (masked)
//   dP^T = V dO_i^T           dS^T = P^T (dP^T - D_i)
//   dV  += P^T dO_i           dK  += dS^T Q_i           dQ_i^T = K^T dS^T
// All five contractions are M = 128, N = 128 UMMAs issued by one thread
// (128-row query steps: an N = 64 instruction costs ~80% of an N = 128 one).
//
// TMEM (512 columns): two 128-column regions R[0], R[1] whose roles alternate
// every step (A = R[i % 2], B = R[(i + 1) % 2]):
//   A: S^T (fp32) -> P^T (bf16 pairs: queries 0-63 over columns 0-31, queries
//      64-127 over columns 64-95, the A operand of dV) and dS^T (bf16 pairs over
//      columns 32-63 and 96-127, the A operand of dK) -> dQ^T (fp32, after dV
//      and dK have read P^T and dS^T) -> dP^T of step i + 1
//   B: dP^T (fp32) -> S^T of step i + 1 (as soon as dP^T is in registers)
//   dV [256,384), dK [384,512) accumulate over the steps.
// The tensor core runs dV_i, S_{i+1}, dK_i, dQ^T_i, dP_{i+1}, dV_{i+1}, ... so
// that P of step i + 1 is computed while dK_i, dQ^T_i and dP_{i+1} run.
//
// smem: K, V resident; Q, dO, LSE, D in 2 stages. After dV_i (and dP_i) have
// read dO_i, its buffer receives dS^T_i (bf16, [128 keys][128 queries],
// 128B-swizzled): the B operand of dQ^T_i (MN-major view). dK_i takes dS^T_i
// from TMEM instead (the .ts form: 32 KB less shared-memory operand traffic per
// step, 2-3% faster than reading it back from the dO buffer). The fp32 dQ accumulator is laid out
// [B, H, 4 column chunks, L128, 32] so that each drain warp (which holds 32 of
// the d columns of dQ^T) owns a contiguous [32 queries x 32] block per quarter
// step: it stages that 4 KB block in its own smem slice and adds it with one
// cp.reduce.async.bulk .add.f32, with no barrier shared between warps (a direct
// red.global per element was measured slower: its load/store traffic delays
// the P/dS warps on the same SM).
//
// Warp roles, one warpgroup each (thread r of a group <-> key row r <-> TMEM
// lane r): WG0 / WG1 compute P and dS for query columns 0-63 / 64-127 and write
// the matching half of dV; WG2 drains dQ and writes dK; WG3: warp 12 is the TMA
// producer and TMEM owner, warp 13 issues tcgen05.mma (the whole warp runs the
// issue loop, one elect.sync lane issues each group and its commit: 4% faster at
// L = 8192 than lane 0 alone in a divergent branch). The block launches with
// 128 registers per thread; WG3 gives registers back (setmaxnreg.dec to 32) and
// the other three groups take them (setmaxnreg.inc to 160): 4*32*32 +
// 12*32*160 = 65536, exactly the launch's register file share. With 152 / 56 the
// P / dS code spilled (44 bytes of reloads through the contended L1 / shared-memory
// pipe); 160 / 32 compiles without spills and ran 1.4-3.9% faster.
//
// d = 80 (OpenLM-3B heads) uses the same tiles: each is two 64-column swizzle
// blocks, the second holding columns 64..79 and TMA zero fill beyond. The
// contractions over d (S^T, dP^T) take 5 K-steps instead of 8, dV and dK are
// N = 80 UMMAs, and dQ^T stays M = 128 (its rows 80..127 are zero: K's padded
// columns), drained by the first three warps into a 3-chunk accumulator.
#include "bwd_d128.cuh"

namespace ddattn {

template <int DH>
__global__ void __launch_bounds__(512, 1)
    attn_bwd_main_d128_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                              const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmDO,
                              const BwdParams p) {
  using C = BwdBig<DH>;
  constexpr int D = C::D, BQ = C::BQ;
  constexpr int KD = D / 16;  // K-steps of the contractions over d
  extern __shared__ uint8_t smem_raw[];
  if (!smem_base_ok(smem_raw, p.status)) return;
  uint8_t* smem = smem_raw;
  Bwd128Bars* bars = reinterpret_cast<Bwd128Bars*>(smem + C::OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int n = blockIdx.x, h = blockIdx.y, b = blockIdx.z;
  const long long seq0 = (long long)b * p.L;
  const int kv0 = n * C::BN;
  const int kv_last = min(kv0 + C::BN - 1, p.L - 1);
  // Live query tiles: from the diagonal to the end of the last key's document.
  const int de_last = (int)(doc_end(p.offsets, p.n_offsets, seq0 + kv_last, seq0 + p.L) - seq0);
  const int m_lo = kv0 / BQ;
  const int m_hi = (de_last - 1) / BQ;
  const int nq = m_hi - m_lo + 1;
  Watchdog wd{&bars->abort_flag, p.status, p.timeout_ns};

  if (threadIdx.x == 0) {
    bars->abort_flag = 0;
    mbar_init(&bars->kv_full, 1);
    for (int i = 0; i < 2; i++) {
      mbar_init(&bars->q_full[i], 1);
      mbar_init(&bars->q_empty[i], 1);
    }
    mbar_init(&bars->s_full, 1);
    mbar_init(&bars->dp_full, 1);
    mbar_init(&bars->p_full, 8);  // per-warp arrivals (mbar_arrive_warp)
    mbar_init(&bars->dp_read, 8);
    mbar_init(&bars->dss_full, 8);
    mbar_init(&bars->dv_done, 1);
    mbar_init(&bars->dq_full, 1);
    mbar_init(&bars->r_free, 4);
    mbar_init(&bars->mma_done, 1);
    fence_mbar_init();
  }
  if (warp == 12) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sDO = smem + C::OFF_DO;
  float* sSTG = reinterpret_cast<float*>(smem + C::OFF_STG);
  float* sLSE = reinterpret_cast<float*>(smem + C::OFF_LSE);
  float* sDEL = reinterpret_cast<float*>(smem + C::OFF_DEL);
  const long long vec0 = ((long long)b * p.H + h) * p.L128;  // row 0 of this (b, h) in the padded vectors

  const int wg = warp >> 2;
  if (wg == 3) {
  setmaxnreg_dec<C::REGS_LOW>();
  if (warp == 12) {
    // ---------------- TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      prefetch_tmap(&tmDO);
      mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
      for (int blk = 0; blk < 2; blk++) {
        tma_load_4d(sK + blk * C::BLK, &tmK, &bars->kv_full, 64 * blk, h, kv0, b);
        tma_load_4d(sV + blk * C::BLK, &tmV, &bars->kv_full, 64 * blk, h, kv0, b);
      }
      int issued = 0;
      for (int i = 0; i < nq; i++) {
        const int s = i & 1;
        const int q0 = (m_lo + i) * BQ;
        if (i >= 2 && !mbar_wait(&bars->q_empty[s], ((i >> 1) - 1) & 1, wd)) break;
        mbar_arrive_expect_tx(&bars->q_full[s], 2 * C::TILE + 2 * BQ * 4);
        for (int blk = 0; blk < 2; blk++) {
          tma_load_4d(sQ + s * C::TILE + blk * C::BLK, &tmQ, &bars->q_full[s], 64 * blk, h, q0, b);
          tma_load_4d(sDO + s * C::TILE + blk * C::BLK, &tmDO, &bars->q_full[s], 64 * blk, h, q0, b);
        }
        bulk_load(sLSE + s * BQ, p.lse2_pad + vec0 + q0, BQ * 4, &bars->q_full[s]);
        bulk_load(sDEL + s * BQ, p.delta_pad + vec0 + q0, BQ * 4, &bars->q_full[s]);
        issued = i + 1;
      }
      if (*wd.abort_flag) {  // let in-flight copies land before the CTA exits
        mbar_wait_drain(&bars->kv_full, 0, wd.limit_ns);
        for (int i = issued - 2 < 0 ? 0 : issued - 2; i < issued; i++)
          mbar_wait_drain(&bars->q_full[i & 1], (i >> 1) & 1, wd.limit_ns);
      }
    }
  } else if (warp == 13) {
    // ---------------- MMA issuer: the whole warp runs the loop (descriptor arithmetic
    // stays warp-uniform), one elected lane issues each group of MMAs and its commit.
    {
      const bool leader = elect_one();
      constexpr uint32_t id_s = idesc_bf16(128, 128, false, false);  // K / V rows x Q / dO rows (K-major)
      constexpr uint32_t id_kv = idesc_bf16(128, D, false, true);    // P^T (TMEM) / dS^T (smem) x dO / Q (MN-major)
      constexpr uint32_t id_dq = idesc_bf16(128, 128, true, true);   // K^T (MN-major) x dS^T (MN-major)
      // Descriptors are built once and advanced by adding (byte offset >> 4) to the
      // 14-bit start-address field (all smem offsets here stay below 256 KB).
      const uint64_t dK_k0 = sdesc_sw128(smem_u32(sK), 16, 1024);          // K-major views
      const uint64_t dV_k0 = sdesc_sw128(smem_u32(sV), 16, 1024);
      const uint64_t dQ_k0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t dO_k0 = sdesc_sw128(smem_u32(sDO), 16, 1024);
      const uint64_t dK_mn0 = sdesc_sw128(smem_u32(sK), C::BLK, 1024);     // MN-major views
      const uint64_t dQ_mn0 = sdesc_sw128(smem_u32(sQ), C::BLK, 1024);
      const uint64_t dO_mn0 = sdesc_sw128(smem_u32(sDO), C::BLK, 1024);
      bool ok = __all_sync(0xffffffffu, mbar_wait(&bars->kv_full, 0, wd) && mbar_wait(&bars->q_full[0], 0, wd));
      if (ok) {
        tc_fence_after();
        if (leader) {
#pragma unroll
          for (int ks = 0; ks < KD; ks++) {  // S^T_0 = K Q_0^T into R[0]
            const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
            umma_bf16(tmem + C::TM_R, dK_k0 + off, dQ_k0 + off, id_s, ks > 0 ? 1u : 0u);
          }
          umma_commit(&bars->s_full);
#pragma unroll
          for (int ks = 0; ks < KD; ks++) {  // dP^T_0 = V dO_0^T into R[1]
            const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
            umma_bf16(tmem + C::TM_R + 128, dV_k0 + off, dO_k0 + off, id_s, ks > 0 ? 1u : 0u);
          }
          umma_commit(&bars->dp_full);
        }
        __syncwarp();
      }
      for (int i = 0; ok && i < nq; i++) {
        const int s = i & 1;
        const uint32_t rA = C::TM_R + (uint32_t)(i & 1) * 128, rB = C::TM_R + (uint32_t)((i + 1) & 1) * 128;
        const uint32_t st = (uint32_t)(s * C::TILE) >> 4, st1 = (uint32_t)(((i + 1) & 1) * C::TILE) >> 4;
        // Opaque copies of the base descriptors: keeps the 40 derived
        // descriptors of a step from being hoisted out of the loop (which would
        // hold them all in registers at once).
        const uint64_t dK_k = opaque_u64(dK_k0), dV_k = opaque_u64(dV_k0), dQ_k = opaque_u64(dQ_k0),
                       dO_k = opaque_u64(dO_k0), dK_mn = opaque_u64(dK_mn0), dQ_mn = opaque_u64(dQ_mn0),
                       dO_mn = opaque_u64(dO_mn0);
        // dV += P^T dO  (A: P^T in region A, 8 columns per 16 queries)
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->p_full, i & 1, wd)))) break;
        tc_fence_after();
        if (leader) {
#pragma unroll
          for (int ks = 0; ks < 8; ks++)  // queries 16 ks..: columns 8 ks (+32 for the second group's half)
            umma_bf16_ts(tmem + C::TM_DV, tmem + rA + ks * 8 + (ks >= 4 ? 32 : 0), dO_mn + st + ks * (2048 >> 4),
                         id_kv, (i > 0 || ks > 0) ? 1u : 0u);
          umma_commit(&bars->dv_done);
        }
        __syncwarp();
        // S^T_{i+1} into region B as soon as dP^T_i has been read out of it.
        if (i + 1 < nq) {
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_full[(i + 1) & 1], ((i + 1) >> 1) & 1, wd) &&
                                                  mbar_wait(&bars->dp_read, i & 1, wd))))
            break;
          tc_fence_after();
          if (leader) {
#pragma unroll
            for (int ks = 0; ks < KD; ks++) {
              const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
              umma_bf16(tmem + rB, dK_k + off, dQ_k + st1 + off, id_s, ks > 0 ? 1u : 0u);
            }
            umma_commit(&bars->s_full);
          }
          __syncwarp();
        }
        // dK += dS^T Q  (A: dS^T in TMEM next to P^T in region A)
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->dss_full, i & 1, wd)))) break;
        tc_fence_after();
        if (leader) {
#pragma unroll
          for (int ks = 0; ks < 8; ks++)  // A: dS^T in TMEM, queries 16 ks..: columns 32 + 8 ks (+32 past query 63)
            umma_bf16_ts(tmem + C::TM_DK, tmem + rA + 32 + ks * 8 + (ks >= 4 ? 32 : 0), dQ_mn + st + ks * (2048 >> 4),
                         id_kv, (i > 0 || ks > 0) ? 1u : 0u);
        // dQ^T = K^T dS^T into region A (dV_i has finished reading P^T there:
        // dss_full is only raised after dv_done).
#pragma unroll
          for (int ks = 0; ks < 8; ks++)
            umma_bf16(tmem + rA, dK_mn + ks * (2048 >> 4), dO_mn + st + ks * (2048 >> 4), id_dq, ks > 0 ? 1u : 0u);
          umma_commit(&bars->dq_full);
        }
        if (leader) umma_commit(&bars->q_empty[s]);
        __syncwarp();
        // dP^T_{i+1} into region A once the drain has read dQ^T_i out of it.
        if (i + 1 < nq) {
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->r_free, i & 1, wd)))) break;
          tc_fence_after();
          if (leader) {
#pragma unroll
            for (int ks = 0; ks < KD; ks++) {
              const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
              umma_bf16(tmem + rA, dV_k + off, dO_k + st1 + off, id_s, ks > 0 ? 1u : 0u);
            }
            umma_commit(&bars->dp_full);
          }
          __syncwarp();
        }
      }
      if (leader) umma_commit(&bars->mma_done);
      __syncwarp();
      mbar_wait_drain(&bars->mma_done, 0, wd.limit_ns);
    }
  }
  } else {
  setmaxnreg_inc<C::REGS_HIGH>();
  if (wg < 2) {
    // ---------------- P / dS warps: group wg handles query columns [64 wg, 64 wg + 64)
    const int r = threadIdx.x & 127;
    const int qh = wg * 64;
    const int kv = kv0 + r;
    const int kvc = kv < p.L ? kv : p.L - 1;
    const int de = (int)(doc_end(p.offsets, p.n_offsets, seq0 + kvc, seq0 + p.L) - seq0);
    const uint32_t tl = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const float sl2 = p.scale_log2;
    bool ok = true;
    for (int i = 0; i < nq && ok; i++) {
      const int s = i & 1;
      const int q0 = (m_lo + i) * BQ;
      const uint32_t rA = C::TM_R + (uint32_t)(i & 1) * 128, rB = C::TM_R + (uint32_t)((i + 1) & 1) * 128;
      // LSE of this group's first 32 query columns is loaded before the S^T wait and the
      // other 32 while the S^T loads from TMEM are in flight: these broadcast shared-memory
      // loads queue behind the tensor core's operand reads, so their latency is hidden
      // behind waits rather than paid inside the exp2 loop.
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_full[s], (i >> 1) & 1, wd));
      if (!ok) break;
      const uint32_t lse_a = smem_u32(sLSE + s * BQ + qh), del_a = smem_u32(sDEL + s * BQ + qh);
      float4 la[8], lb[8];
#pragma unroll
      for (int e4 = 0; e4 < 8; e4++) la[e4] = lds_f4(lse_a + 16 * e4);
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full, i & 1, wd));
      if (!ok) break;
      tc_fence_after();
      const bool need_mask = (q0 + qh < kv) || (q0 + qh + 64 > de);
      // P^T of this group's 64 query columns, packed as bf16 pairs.
      uint32_t pk[32];
      {
        uint32_t s0[32], s1[32];
        tmem_ld32(tl + rA + qh, s0);
        tmem_ld32(tl + rA + qh + 32, s1);
#pragma unroll
        for (int e4 = 0; e4 < 8; e4++) lb[e4] = lds_f4(lse_a + 128 + 16 * e4);
        tmem_ld_wait(s0);
        tmem_ld_wait(s1);
#pragma unroll
        for (int c = 0; c < 2; c++) {
#pragma unroll
          for (int e4 = 0; e4 < 8; e4++) {
            const float4 l = c ? lb[e4] : la[e4];
            const uint32_t* sv = c ? s1 : s0;
            float pv[4];
            pv[0] = exp2_approx(fmaf(__uint_as_float(sv[4 * e4 + 0]), sl2, -l.x));
            pv[1] = exp2_approx(fmaf(__uint_as_float(sv[4 * e4 + 1]), sl2, -l.y));
            pv[2] = exp2_approx(fmaf(__uint_as_float(sv[4 * e4 + 2]), sl2, -l.z));
            pv[3] = exp2_approx(fmaf(__uint_as_float(sv[4 * e4 + 3]), sl2, -l.w));
            if (need_mask) {
#pragma unroll
              for (int e = 0; e < 4; e++) {
                const int q = q0 + qh + c * 32 + 4 * e4 + e;
                if (q < kv || q >= de) pv[e] = 0.f;
              }
            }
            pk[c * 16 + 2 * e4] = pack_bf16x2(pv[0], pv[1]);
            pk[c * 16 + 2 * e4 + 1] = pack_bf16x2(pv[2], pv[3]);
          }
        }
      }
      // P^T over the first 32 of this group's own 64 S^T columns of region A
      // (queries 64 wg .. 64 wg + 63 as bf16 pairs; this group has read them).
      tmem_st32(tl + rA + wg * 64, pk);
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive_warp(&bars->p_full);
      // dS^T = P^T (dP^T - D), from the bf16 P^T that dV also uses.
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dp_full, i & 1, wd));
      if (!ok) break;
      tc_fence_after();
      uint32_t dk[32];
      {
        uint32_t d0[32], d1[32];
        tmem_ld32(tl + rB + qh, d0);
        tmem_ld32(tl + rB + qh + 32, d1);
        tmem_ld_wait(d0);
        tmem_ld_wait(d1);
        tc_fence_before();
        mbar_arrive_warp(&bars->dp_read);  // region B may take S^T of the next step
#pragma unroll
        for (int c = 0; c < 2; c++) {
          const uint32_t* dv = c ? d1 : d0;
#pragma unroll
          for (int e4 = 0; e4 < 8; e4++) {
            const float4 dd = lds_f4(del_a + 16 * (c * 8 + e4));
            const int w = c * 16 + 2 * e4;
            // bf16 pair -> two floats (first element in the low half)
            const float p0 = __uint_as_float(pk[w] << 16), p1 = __uint_as_float(pk[w] & 0xffff0000u);
            const float p2 = __uint_as_float(pk[w + 1] << 16), p3 = __uint_as_float(pk[w + 1] & 0xffff0000u);
            dk[w] = pack_bf16x2(p0 * (__uint_as_float(dv[4 * e4 + 0]) - dd.x),
                                p1 * (__uint_as_float(dv[4 * e4 + 1]) - dd.y));
            dk[w + 1] = pack_bf16x2(p2 * (__uint_as_float(dv[4 * e4 + 2]) - dd.z),
                                    p3 * (__uint_as_float(dv[4 * e4 + 3]) - dd.w));
          }
        }
      }
      // dS^T -> TMEM over the second 32 of this group's 64 columns of region A (the A
      // operand of dK += dS^T Q; those S^T columns were read above, P^T is in the first 32)
      // and -> block wg of this stage's dO buffer (the B operand of dQ^T), the latter once
      // dP and dV have finished reading dO.
      tmem_st32(tl + rA + wg * 64 + 32, dk);
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dv_done, i & 1, wd));
      if (!ok) break;
      const uint32_t dsb = smem_u32(sDO) + s * C::TILE + wg * C::BLK;
#pragma unroll
      for (int c = 0; c < 8; c++)
        st_shared_v4(dsb + sw128_offset(r, c), dk[4 * c], dk[4 * c + 1], dk[4 * c + 2], dk[4 * c + 3]);
      fence_proxy_async_smem();
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive_warp(&bars->dss_full);
    }
    // Epilogue: dV rows.
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, 0, wd));
    if (ok) {
      tc_fence_after();
      dv_epilogue<D>(p, tl + C::TM_DV + qh, qh, seq0, h, kv0 + 32 * (warp & 3), lane, [] {});
    }
  } else {
    // ---------------- dQ drain warps 8-11: thread t <-> TMEM lane t <-> column d = t of dQ^T
    const int w = warp & 3;                       // column chunk d = 32 w .. 32 w + 31
    const uint32_t tl = tmem + ((uint32_t)(w * 32) << 16);
    float* stg2 = sSTG + w * (2 * 32 * 32);       // this warp's two [32 q][32] staging slices
    float* acc_w = p.dq_acc + (vec0 * C::NCH + (long long)w * p.L128) * 32;  // chunk w of this (b, h)
    const bool drains = w < C::NCH;               // d = 80: the fourth chunk (rows 96..127 of dQ^T) is zero
    bool ok = true;
    for (int i = 0; i < nq; i++) {
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dq_full, i & 1, wd));
      if (!ok) break;
      tc_fence_after();
      const uint32_t rA = C::TM_R + (uint32_t)(i & 1) * 128;
      uint32_t v[4][32];
#pragma unroll
      for (int c = 0; c < 4; c++) tmem_ld32(tl + rA + c * 32, v[c]);
#pragma unroll
      for (int c = 0; c < 4; c++) tmem_ld_wait(v[c]);
      tc_fence_before();
      mbar_arrive_warp(&bars->r_free);
      const int q0 = (m_lo + i) * BQ;
      if (!drains) continue;
#pragma unroll
      for (int c = 0; c < 4; c++) {
        // Two slices in turn: the reduction two back (same slice) must have read it, the one
        // just issued may still be in flight (5% faster at L = 8192 than one slice).
        float* stg = stg2 + (c & 1) * (32 * 32);
        if (lane == 0) bulk_wait_read<1>();
        __syncwarp();
#pragma unroll
        for (int e = 0; e < 32; e++) stg[e * 32 + lane] = __uint_as_float(v[c][e]);  // row q = 32c + e
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          bulk_reduce_add_f32(acc_w + (long long)(q0 + 32 * c) * 32, stg, 32 * 32 * 4);
          bulk_commit();
        }
      }
    }
    if (lane == 0) bulk_wait<0>();
    // Epilogue: dK rows (scaled; rotated back with RoPE).
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, 0, wd));
    if (ok) {
      tc_fence_after();
      dk_epilogue<D, C::NCH>(p, tl + C::TM_DK, smem_u32(stg2), seq0, h, kv0 + 32 * w, lane, [] {});
    }
  }

  }

  tc_fence_before();
  __syncthreads();
  if (warp == 12) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH>
static cudaError_t launch_big(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                              const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream) {
  using C = BwdBig<DH>;
  static DeviceCache nsm_dev;
  int nsm = 0;
  cudaError_t e = kernel_setup(nsm_dev, attn_bwd_main_d128_kernel<DH>, C::SMEM_BYTES, &nsm);
  if (e != cudaSuccess) return e;
  dim3 grid(p.nkt, p.H, p.B);
  attn_bwd_main_d128_kernel<DH><<<grid, C::THREADS, C::SMEM_BYTES, stream>>>(tq, tk, tv, tdo, p);
  return cudaGetLastError();
}

cudaError_t launch_attn_bwd_main_d128(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                      const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream) {
  // Up to 16 key tiles per sequence (L <= 2048) CTAs walk key tiles (their epilogues and
  // the next tile's loads overlap): -26% at L = 256 ... -2.5% at L = 2048 against one CTA
  // per key tile, which stays faster for longer sequences (+1-4% at 4096 / 8192).
  if (p.nkt <= 16) return launch_attn_bwd_main_d128_persist(d, tq, tk, tv, tdo, p, stream);
  if (d == 80) return launch_big<80>(tq, tk, tv, tdo, p, stream);
  return launch_big<128>(tq, tk, tv, tdo, p, stream);
}

}  // namespace ddattn
