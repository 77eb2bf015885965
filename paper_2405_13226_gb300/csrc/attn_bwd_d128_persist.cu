// Attention backward main kernel for head dims 128 and 80, persistent form for short
// sequences (up to 16 key tiles, L <= 2048).
//
// The per-step work, warp roles, TMEM regions and shared-memory layout are those of
// attn_bwd_main_d128_kernel (csrc/attn_bwd_d128.cu). Here a CTA per SM walks work items
// (128-key tile, head, sequence), items c, c + G, c + 2G ... with G coprime to the key-tile
// count, so that an item's epilogue (dV, dK out of TMEM) and the next item's first loads
// overlap, and the launch gap between CTAs goes. At L = 256 a CTA of the per-tile kernel
// spends ~4.3 of its 11.2 us on exactly those.
//   * Per-step barriers and the two TMEM regions' roles follow the CTA's running step count
//     g across items (q_full / q_empty stage g % 2, the rest parity g % 2).
//   * The producer issues an item's first Q / dO as soon as its stage is free, then waits on
//     kv_empty (committed after the previous item's last MMAs) before replacing K and V.
//   * The item's first S^T / dP^T go into the regions the previous item's last step left
//     (after dp_read / r_free of that step), as within an item.
//   * mma_done is committed per item; the P / dS and drain warps write that item's dV / dK
//     and arrive on dv_free / dk_free, which the next item's first dV / dK MMAs wait for
//     (they overwrite the accumulators).
#include "bwd_d128.cuh"

namespace ddattn {

// dq rows [r0, r0 + 128) of one (sequence, head), columns 32 w .. 32 w + NV - 1 (NV = 32, or
// 16 for the last chunk at d = 80), from the fp32 slot rows acc_w (chunk w, row-major
// [L128][32]): dq = bf16(scale * acc), rotated back (R^T) with RoPE. Lane l converts rows
// r0 + l, r0 + l + 32, ...; a row is 4 NV contiguous bytes of the slot and 2 NV of dq.
template <int D, int NV>
__device__ __forceinline__ void dq_owned_convert(const BwdParams& p, const float* acc_w, long long seq0, int h,
                                                 int r0, int w, int lane) {
#pragma unroll 1
  for (int rr = lane; rr < 128; rr += 32) {
    const int row = r0 + rr;
    if (row >= p.L) break;
    const float4* src = reinterpret_cast<const float4*>(acc_w + (long long)row * 32);
    float f[32];
#pragma unroll
    for (int q = 0; q < NV / 4; q++) {
      const float4 x = src[q];
      f[4 * q] = x.x * p.scale;
      f[4 * q + 1] = x.y * p.scale;
      f[4 * q + 2] = x.z * p.scale;
      f[4 * q + 3] = x.w * p.scale;
    }
    if (p.rope_tab_rows) {  // pairs j = 16 w + u at position row
      const float4* cs = reinterpret_cast<const float4*>(p.rope_tab_rows + (long long)row * (D / 2) + w * 16);
#pragma unroll
      for (int u = 0; u < NV / 4; u++) {
        const float4 c = cs[u];
        rope_unrotate_pair(f[4 * u], f[4 * u + 1], c.x, c.y);
        rope_unrotate_pair(f[4 * u + 2], f[4 * u + 3], c.z, c.w);
      }
    }
    store_row(p.dq + ((seq0 + row) * p.H + h) * D + w * 32, f, NV);
  }
}

template <int DH, int WALK>
__global__ void __launch_bounds__(512, 1)
    attn_bwd_main_d128_persist_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
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

  // CTA c works on the items of bwd_walk_item (G = gridDim.x); per-step barrier phases and
  // TMEM region roles follow the CTA's running step count g across items.
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
    mbar_init(&bars->kv_empty, 1);
    mbar_init(&bars->dv_free, 8);
    mbar_init(&bars->dk_free, 4);
    mbar_init(&bars->mma_drain, 1);
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

  const int wg = warp >> 2;
  if (wg == 3) {
  setmaxnreg_dec<C::REGS_LOW_P>();
  if (warp == 12) {
    // ---------------- TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      prefetch_tmap(&tmDO);
      int q_issued = 0, kv_issued = 0, g0 = 0, ic = 0;
      bool ok = true;
      for (int it; ok && (it = bwd_walk_item<WALK>(p, ic)) >= 0; ic++) {
        const BwdItem I = bwd_item<C::BN, BQ>(p, it);
        for (int i = 0; i < I.nq; i++) {
          const int g = g0 + i, s = g & 1;
          const int q0 = (I.m_lo + i) * BQ;
          if (g >= 2 && !(ok = mbar_wait(&bars->q_empty[s], ((g >> 1) - 1) & 1, wd))) break;
          mbar_arrive_expect_tx(&bars->q_full[s], 2 * C::TILE + 2 * BQ * 4);
          for (int blk = 0; blk < 2; blk++) {
            tma_load_4d(sQ + s * C::TILE + blk * C::BLK, &tmQ, &bars->q_full[s], 64 * blk, I.h, q0, I.b);
            tma_load_4d(sDO + s * C::TILE + blk * C::BLK, &tmDO, &bars->q_full[s], 64 * blk, I.h, q0, I.b);
          }
          bulk_load(sLSE + s * BQ, p.lse2_pad + I.vec0 + q0, BQ * 4, &bars->q_full[s]);
          bulk_load(sDEL + s * BQ, p.delta_pad + I.vec0 + q0, BQ * 4, &bars->q_full[s]);
          q_issued = g + 1;
          if (i == 0) {  // this item's K / V once the previous item's MMAs have read theirs
            if (ic > 0 && !(ok = mbar_wait(&bars->kv_empty, (ic - 1) & 1, wd))) break;
            mbar_arrive_expect_tx(&bars->kv_full, 2 * C::TILE);
            for (int blk = 0; blk < 2; blk++) {
              tma_load_4d(sK + blk * C::BLK, &tmK, &bars->kv_full, 64 * blk, I.h, I.kv0, I.b);
              tma_load_4d(sV + blk * C::BLK, &tmV, &bars->kv_full, 64 * blk, I.h, I.kv0, I.b);
            }
            kv_issued = ic + 1;
          }
        }
        g0 += I.nq;
      }
      // Every copy lands before the CTA can exit (after an abort nobody else waits for them).
      if (kv_issued > 0) mbar_wait_drain(&bars->kv_full, (kv_issued - 1) & 1, wd.limit_ns);
      for (int g = q_issued - 2 < 0 ? 0 : q_issued - 2; g < q_issued; g++)
        mbar_wait_drain(&bars->q_full[g & 1], (g >> 1) & 1, wd.limit_ns);
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
      bool ok = true;
      int g0 = 0, ic = 0;
      for (int it; ok && (it = bwd_walk_item<WALK>(p, ic)) >= 0; ic++) {
        const int nq = bwd_item<C::BN, BQ>(p, it).nq;
        // The item's first S^T and dP^T, into R[g0 % 2] (the previous step's dP^T region,
        // once the P / dS warps have read it) and R[(g0 + 1) % 2] (its dQ^T region, once drained).
        ok = __all_sync(0xffffffffu, mbar_wait(&bars->kv_full, ic & 1, wd) &&
                                         mbar_wait(&bars->q_full[g0 & 1], (g0 >> 1) & 1, wd) &&
                                         (g0 == 0 || (mbar_wait(&bars->dp_read, (g0 - 1) & 1, wd) &&
                                                      mbar_wait(&bars->r_free, (g0 - 1) & 1, wd))));
        if (!ok) break;
        tc_fence_after();
        {
          const uint32_t r0 = C::TM_R + (uint32_t)(g0 & 1) * 128, r1 = C::TM_R + (uint32_t)((g0 + 1) & 1) * 128;
          const uint32_t st0 = (uint32_t)((g0 & 1) * C::TILE) >> 4;
          const uint64_t dK_k = opaque_u64(dK_k0), dV_k = opaque_u64(dV_k0), dQ_k = opaque_u64(dQ_k0),
                         dO_k = opaque_u64(dO_k0);
          if (leader) {
#pragma unroll
            for (int ks = 0; ks < KD; ks++) {
              const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
              umma_bf16(tmem + r0, dK_k + off, dQ_k + st0 + off, id_s, ks > 0 ? 1u : 0u);
            }
            umma_commit(&bars->s_full);
#pragma unroll
            for (int ks = 0; ks < KD; ks++) {
              const uint32_t off = ((ks >> 2) * C::BLK + (ks & 3) * 32) >> 4;
              umma_bf16(tmem + r1, dV_k + off, dO_k + st0 + off, id_s, ks > 0 ? 1u : 0u);
            }
            umma_commit(&bars->dp_full);
          }
          __syncwarp();
        }
        for (int i = 0; ok && i < nq; i++) {
          const int g = g0 + i, s = g & 1;
          const uint32_t rA = C::TM_R + (uint32_t)(g & 1) * 128, rB = C::TM_R + (uint32_t)((g + 1) & 1) * 128;
          const uint32_t st = (uint32_t)(s * C::TILE) >> 4, st1 = (uint32_t)(((g + 1) & 1) * C::TILE) >> 4;
          // Opaque copies of the base descriptors: keeps the 40 derived
          // descriptors of a step from being hoisted out of the loop (which would
          // hold them all in registers at once).
          const uint64_t dK_k = opaque_u64(dK_k0), dV_k = opaque_u64(dV_k0), dQ_k = opaque_u64(dQ_k0),
                         dO_k = opaque_u64(dO_k0), dK_mn = opaque_u64(dK_mn0), dQ_mn = opaque_u64(dQ_mn0),
                         dO_mn = opaque_u64(dO_mn0);
          // dV += P^T dO  (A: P^T in region A, 8 columns per 16 queries)
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->p_full, g & 1, wd) &&
                                                (i > 0 || ic == 0 || mbar_wait(&bars->dv_free, (ic - 1) & 1, wd))))) break;
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
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_full[(g + 1) & 1], ((g + 1) >> 1) & 1, wd) &&
                                                    mbar_wait(&bars->dp_read, g & 1, wd))))
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
          if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->dss_full, g & 1, wd) &&
                                                (i > 0 || ic == 0 || mbar_wait(&bars->dk_free, (ic - 1) & 1, wd))))) break;
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
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(&bars->r_free, g & 1, wd)))) break;
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
        if (!ok) break;
        if (leader) {
          umma_commit(&bars->kv_empty);
          umma_commit(&bars->mma_done);
        }
        __syncwarp();
        g0 += nq;
      }
      if (leader) umma_commit(&bars->mma_drain);  // every MMA of this CTA, before the warp leaves
      __syncwarp();
      mbar_wait_drain(&bars->mma_drain, 0, wd.limit_ns);
    }
  }
  } else {
  setmaxnreg_inc<C::REGS_HIGH_P>();
  if (wg < 2) {
    // ---------------- P / dS warps: group wg handles query columns [64 wg, 64 wg + 64)
    const int r = threadIdx.x & 127;
    const int qh = wg * 64;
    const uint32_t tl = tmem + ((uint32_t)((warp & 3) * 32) << 16);
    const float sl2 = p.scale_log2;
    bool ok = true;
    int g0 = 0, ic = 0;
    for (int it; ok && (it = bwd_walk_item<WALK>(p, ic)) >= 0; ic++) {
    const BwdItem I = bwd_item<C::BN, BQ>(p, it);
    const int h = I.h, m_lo = I.m_lo, nq = I.nq;
    const long long seq0 = I.seq0;
    const int kv = I.kv0 + r;
    const int kvc = kv < p.L ? kv : p.L - 1;
    const int de = (int)(doc_end(p.offsets, p.n_offsets, seq0 + kvc, seq0 + p.L) - seq0);
    for (int i = 0; i < nq && ok; i++) {
      const int g = g0 + i, s = g & 1;
      const int q0 = (m_lo + i) * BQ;
      const uint32_t rA = C::TM_R + (uint32_t)(g & 1) * 128, rB = C::TM_R + (uint32_t)((g + 1) & 1) * 128;
      // LSE of this group's first 32 query columns is loaded before the S^T wait and the
      // other 32 while the S^T loads from TMEM are in flight: these broadcast shared-memory
      // loads queue behind the tensor core's operand reads, so their latency is hidden
      // behind waits rather than paid inside the exp2 loop.
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->q_full[s], (g >> 1) & 1, wd));
      if (!ok) break;
      const uint32_t lse_a = smem_u32(sLSE + s * BQ + qh), del_a = smem_u32(sDEL + s * BQ + qh);
      float4 la[8], lb[8];
#pragma unroll
      for (int e4 = 0; e4 < 8; e4++) la[e4] = lds_f4(lse_a + 16 * e4);
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full, g & 1, wd));
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
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dp_full, g & 1, wd));
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
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dv_done, g & 1, wd));
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
    // Epilogue: dV rows of this item.
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, ic & 1, wd));
    if (ok) {
      tc_fence_after();
      auto release = [&] {
        tc_fence_before();
        mbar_arrive_warp(&bars->dv_free);  // dV of this item has left TMEM
      };
      if (WALK == kWalkOwned) dv_epilogue<D>(p, tl + C::TM_DV + qh, qh, seq0, h, I.kv0 + 32 * (warp & 3), lane, release);
      else dv_epilogue_rows<D>(p, tl + C::TM_DV + qh, qh, seq0, h, kv, release);
    }
    g0 += nq;
    }
  } else {
    // ---------------- dQ drain warps 8-11: thread t <-> TMEM lane t <-> column d = t of dQ^T
    const int w = warp & 3;                       // column chunk d = 32 w .. 32 w + 31
    const uint32_t tl = tmem + ((uint32_t)(w * 32) << 16);
    float* stg2 = sSTG + w * (2 * 32 * 32);       // this warp's two [32 q][32] staging slices
    const bool drains = w < C::NCH;               // d = 80: the fourth chunk (rows 96..127 of dQ^T) is zero
    bool ok = true;
    int g0 = 0, ic = 0;
    for (int it; ok && (it = bwd_walk_item<WALK>(p, ic)) >= 0; ic++) {
    const BwdItem I = bwd_item<C::BN, BQ>(p, it);
    const int h = I.h, m_lo = I.m_lo, nq = I.nq, kv0 = I.kv0;
    const long long seq0 = I.seq0;
    // Chunk w of the fp32 dQ rows: the (b, h) region of the shared accumulator, or, with dQ
    // owned, this CTA's own slot (the region of index blockIdx.x, reused for every pair the
    // CTA owns, so it stays in L2).
    float* acc_w = WALK == kWalkOwned ? p.dq_acc + ((long long)blockIdx.x * C::NCH + w) * p.L128 * 32
                                      : p.dq_acc + (I.vec0 * C::NCH + (long long)w * p.L128) * 32;
    for (int i = 0; i < nq; i++) {
      const int g = g0 + i;
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->dq_full, g & 1, wd));
      if (!ok) break;
      tc_fence_after();
      const uint32_t rA = C::TM_R + (uint32_t)(g & 1) * 128;
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
          float* dst = acc_w + (long long)(q0 + 32 * c) * 32;
          if (WALK == kWalkOwned && i == 0) {
            bulk_store(dst, stg, 32 * 32 * 4);  // the query tile's first partial
          } else {
            // With dQ owned, this block's first partial (a store) is at least 8 groups back:
            // 3 - c after it in its step, 4 in the next item's diagonal step, c before this one.
            if (WALK == kWalkOwned) bulk_wait<7>();
            bulk_reduce_add_f32(dst, stg, 32 * 32 * 4);
          }
          bulk_commit();
        }
      }
    }
    // Epilogue: dK rows of this item (scaled; rotated back with RoPE).
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, ic & 1, wd));
    if (ok) {
      tc_fence_after();
      dk_epilogue_rows<D, C::NCH>(p, tl + C::TM_DK, seq0, h, kv0 + 32 * w + lane, [&] {
        tc_fence_before();
        mbar_arrive_warp(&bars->dk_free);  // dK of this item has left TMEM
      });
    }
    // dQ owned: the query tiles whose last contributor is this key tile are complete once
    // this warp's copies have landed; convert its chunk of their rows to bf16 dq.
    if (WALK == kWalkOwned && ok && drains) {
      uint32_t done = 0;  // bit i: query tile m_lo + i (nq <= 16)
      for (int i = 0; i < nq; i++)
        if (bwd_last_contributor(p, seq0, m_lo + i) == I.n) done |= 1u << i;
      if (done) {
        if (lane == 0) bulk_wait<0>();
        __syncwarp();
        fence_proxy_async_global();
        for (int i = 0; i < nq; i++) {
          if (!(done & (1u << i))) continue;
          if (D - 32 * w >= 32) dq_owned_convert<D, 32>(p, acc_w, seq0, h, (m_lo + i) * BQ, w, lane);
          else dq_owned_convert<D, 16>(p, acc_w, seq0, h, (m_lo + i) * BQ, w, lane);
        }
        __syncwarp();
        fence_proxy_async_global();  // these reads before the next pair's copies into the slot
      }
    }
    g0 += nq;
    }
    if (lane == 0) bulk_wait<0>();  // every reduction of this CTA has landed
  }

  }

  tc_fence_before();
  __syncthreads();
  if (warp == 12) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int DH, int WALK>
static cudaError_t launch_walk(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                               const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream) {
  using C = BwdBig<DH>;
  static DeviceCache nsm_dev;
  int nsm = 0;
  cudaError_t e = kernel_setup(nsm_dev, attn_bwd_main_d128_persist_kernel<DH, WALK>, C::SMEM_BYTES, &nsm);
  if (e != cudaSuccess) return e;
  const long long items = (long long)p.nkt * p.H * p.B;
  if (items > 2147483647LL - 4096) return cudaErrorInvalidValue;  // item indices are int
  long long G = items < nsm ? items : nsm;  // one CTA per SM (shared memory allows no more)
  if (WALK == kWalkOwned) {
    // over the (sequence, head) pairs; CTA c uses slot c
    const long long pairs = (long long)p.B * p.H;
    G = pairs < nsm ? pairs : nsm;
  } else {
    // stride coprime with the key-tile count: every CTA then sees every key-tile position,
    // whose step counts differ
    auto gcd = [](long long x, long long y) {
      while (y) {
        const long long t = x % y;
        x = y;
        y = t;
      }
      return x;
    };
    while (G > 1 && gcd(G, p.nkt) != 1) G--;
  }
  attn_bwd_main_d128_persist_kernel<DH, WALK><<<(unsigned)G, C::THREADS, C::SMEM_BYTES, stream>>>(tq, tk, tv, tdo, p);
  return cudaGetLastError();
}

template <int DH>
static cudaError_t launch_persist(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                  const CUtensorMap& tdo, const BwdParams& p, cudaStream_t stream) {
  if (p.dq_owned) return launch_walk<DH, kWalkOwned>(tq, tk, tv, tdo, p, stream);
  return launch_walk<DH, kWalkStatic>(tq, tk, tv, tdo, p, stream);
}

cudaError_t launch_attn_bwd_main_d128_persist(int d, const CUtensorMap& tq, const CUtensorMap& tk,
                                              const CUtensorMap& tv, const CUtensorMap& tdo, const BwdParams& p,
                                              cudaStream_t stream) {
  if (d == 80) return launch_persist<80>(tq, tk, tv, tdo, p, stream);
  return launch_persist<128>(tq, tk, tv, tdo, p, stream);
}

}  // namespace ddattn
