// Causal / document-masked attention backward for sm_103a.
//
// Three kernels on the caller's stream:
//   attn_bwd_pre   D_i = <dO_i, o_i> and LSE_i*log2(e) into padded per-row
//                  vectors (rows past L: D = 0, LSE = +inf so P = 0), and
//                  zero the fp32 dQ accumulator.
//   attn_bwd_main  (d = 64 here; d = 128 in attn_bwd_d128.cu)
//                  one CTA per 128-key tile of one (sequence, head). It keeps
//                  K, V in smem and dK, dV in TMEM, and walks the live query
//                  tiles (diagonal .. end of the last key's document):
//                    S^T  = K Q^T            (TMEM)  -> P^T = exp2(S^T*scale*log2e - LSE*log2e)
//                    dP^T = V dO^T           (TMEM)  -> dS^T = P^T (dP^T - D)
//                    dV  += P^T dO           (TMEM, A = P^T from smem)
//                    dK  += dS^T Q           (TMEM, A = dS^T from smem)
//                    dQ   = dS K (or its transpose, d = 128)   (TMEM)
//                  dQ is drained by a second warpgroup through smem into one
//                  bulk cp.reduce.async.bulk .add.f32 of the contiguous
//                  [BQ x d] block of the fp32 accumulator.
//   attn_bwd_post  dq = bf16(scale * dQacc), rotated back (R^T) with RoPE.
// With RoPE the pre phase also fills the [L, d/2] (cos, sin) table and the dK
// epilogue rotates dk back with it.
// Warp roles of attn_bwd_main: warps 0-3 compute P/dS (thread r <-> key row r
// <-> TMEM lane r) and write dV; warps 4-7 drain dQ and write dK; warp 8 is
// the TMA producer; warp 9 issues tcgen05.mma.
#include <algorithm>

#include "common.cuh"

namespace ddattn {

template <int D>
struct BwdCfg {
  static constexpr int BN = 128;                        // key rows per CTA
  static constexpr int BQ = (D == 128) ? 64 : 128;      // query rows per step
  static constexpr bool DQ_T = (D == 128);              // TMEM holds dQ^T (lanes = d)
  static constexpr int DB = D / 64;
  static constexpr int KV_BLK = BN * 128;               // [128 rows][64] bf16 block
  static constexpr int KV_BYTES = DB * KV_BLK;
  static constexpr int QB_BLK = BQ * 128;               // [BQ rows][64] bf16 block
  static constexpr int QS_BYTES = DB * QB_BLK;
  static constexpr int PB_BLK = BN * 128;               // [128 key rows][64 q] bf16 block
  static constexpr int P_BYTES = (BQ / 64) * PB_BLK;
  static constexpr int DQS_BYTES = BQ * D * 4;
  static constexpr int OFF_K = 0;
  static constexpr int OFF_V = OFF_K + KV_BYTES;
  static constexpr int OFF_Q = OFF_V + KV_BYTES;
  static constexpr int OFF_DO = OFF_Q + 2 * QS_BYTES;
  static constexpr int OFF_P = OFF_DO + 2 * QS_BYTES;
  static constexpr int OFF_DS = OFF_P + P_BYTES;
  static constexpr int OFF_DQS = OFF_DS + P_BYTES;
  static constexpr int OFF_LSE = OFF_DQS + DQS_BYTES;   // [2][BQ] fp32
  static constexpr int OFF_DEL = OFF_LSE + 2 * BQ * 4;  // [2][BQ] fp32
  static constexpr int OFF_BAR = OFF_DEL + 2 * BQ * 4;
  static constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;
  // TMEM columns
  static constexpr uint32_t TM_S = 0;
  static constexpr uint32_t TM_DP = BQ;
  static constexpr uint32_t TM_DQ = 2 * BQ;
  static constexpr uint32_t TM_DV = (D == 128) ? 256 : 320;
  static constexpr uint32_t TM_DK = 384;
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr int THREADS = 320;
};

struct BwdBars {
  uint64_t kv_full;
  uint64_t q_full[2], q_empty[2];
  uint64_t s_full, sdp_free, p_full, p_free, ds_full, ds_free, dq_full, dq_free;
  uint64_t mma_done;
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(BwdBars) <= 256, "barrier block");

// Columns of one row of the fp32 dQ accumulator: d = 64 keeps [.., L128, 64];
// the d = 80 / 128 kernel uses ceil(d/32) chunks of 32 columns.
template <int D>
__host__ __device__ constexpr int acc_cols() { return D == 64 ? 64 : (D + 31) / 32 * 32; }

// ------------------------------------------------------------------ pre
// D_i = <dO_i, o_i>: one group of G threads per (b, i, h) row, rows in memory
// order; the first d/8 threads of a group load 8 bf16 each (G = d/8 rounded up
// to a power of two, the shuffle width). A warp covers 32/G rows per step and
// keeps U steps of loads in flight before reducing; each step also zeroes the
// same number of the fp32 dQ accumulator's rows (taken as a flat array), so
// reads and writes share the memory bus (measured 0.172 ms for 1.07 GB at
// H = 16, d = 128, 65536 tokens, vs 0.190 with the zeroing as a separate pass).
// LSE*log2e and the padded rows then go over [B, H, L128] in memory order, and
// the accumulator rows beyond B*L*H are zeroed.
template <int D>
__global__ void __launch_bounds__(256) attn_bwd_pre_kernel(const BwdParams p) {
  constexpr int NP = D / 8;                                        // 16-byte parts per row
  constexpr int G = NP <= 8 ? 8 : (NP <= 16 ? 16 : 32);            // threads per row
  constexpr int RPW = 32 / G;                                      // rows per warp step
  constexpr int U = 4;                                             // warp steps in flight
  const long long nrows = (long long)p.B * p.L * p.H;
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long stride = (long long)gridDim.x * blockDim.x;
  const int lane = threadIdx.x & 31, sub = lane / G, part = lane % G;
  const long long warp = tid >> 5, nwarps = stride >> 5;
  // The loop bound is uniform per warp so every shuffle sees all 32 lanes.
  for (long long r0 = warp * (RPW * U); r0 < nrows; r0 += nwarps * (RPW * U)) {
    uint4 a[U], g[U];
#pragma unroll
    for (int u = 0; u < U; u++) {
      const long long row = r0 + u * RPW + sub;
      if (row < nrows && part < NP) {
        a[u] = reinterpret_cast<const uint4*>(p.o + row * D)[part];
        g[u] = reinterpret_cast<const uint4*>(p.dO + row * D)[part];
      } else {
        a[u] = make_uint4(0u, 0u, 0u, 0u);
        g[u] = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    if (!p.dq_owned) {  // zero the accumulator span of these rows (flat), interleaving writes with the reads
      constexpr int AC = acc_cols<D>();
      float4* acc4 = reinterpret_cast<float4*>(p.dq_acc) + r0 * (AC / 4);
      const long long lim = (nrows - r0 < RPW * U ? nrows - r0 : RPW * U) * (AC / 4);
#pragma unroll
      for (int k = 0; k < RPW * U * AC / 4 / 32; k++)
        if (k * 32 + lane < lim) acc4[k * 32 + lane] = make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float acc[U];
#pragma unroll
    for (int u = 0; u < U; u++) {
      const __nv_bfloat162* a2 = reinterpret_cast<const __nv_bfloat162*>(&a[u]);
      const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&g[u]);
      acc[u] = 0.f;
#pragma unroll
      for (int e = 0; e < 4; e++) {
        const float2 x = __bfloat1622float2(a2[e]);
        const float2 y = __bfloat1622float2(g2[e]);
        acc[u] = fmaf(x.x, y.x, acc[u]);
        acc[u] = fmaf(x.y, y.y, acc[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < U; u++)
#pragma unroll
      for (int off = G / 2; off > 0; off >>= 1) acc[u] += __shfl_xor_sync(0xffffffffu, acc[u], off, G);
    if (part == 0) {
#pragma unroll
      for (int u = 0; u < U; u++) {
        const long long row = r0 + u * RPW + sub;
        if (row < nrows) {
          const int h = (int)(row % p.H);
          const long long bi = row / p.H;
          const int i = (int)(bi % p.L);
          const int b = (int)(bi / p.L);
          p.delta_pad[((long long)b * p.H + h) * p.L128 + i] = acc[u];
        }
      }
    }
  }
  // LSE * log2(e) over [B, H, L128]; rows past L: LSE = +inf (P = 0), D = 0.
  const long long nvec = (long long)p.B * p.H * p.L128;
  for (long long t = tid; t < nvec; t += stride) {
    const long long bh = t / p.L128;
    const int i = (int)(t - bh * p.L128);
    if (i < p.L) {
      p.lse2_pad[t] = p.lse[bh * p.L + i] * kLog2e;
    } else {
      p.lse2_pad[t] = INFINITY;
      p.delta_pad[t] = 0.f;
    }
  }
  // zero the rest of the dQ accumulator (past nrows * acc_cols: the padded rows)
  if (p.dq_owned) return;  // the main kernel's first partial of every query tile is a store
  const long long n4 = (long long)p.B * p.H * p.L128 * acc_cols<D>() / 4;
  float4* acc4 = reinterpret_cast<float4*>(p.dq_acc);
  for (long long t = nrows * (acc_cols<D>() / 4) + tid; t < n4; t += stride) acc4[t] = make_float4(0.f, 0.f, 0.f, 0.f);
}

// ------------------------------------------------------------------ post
template <int D>
__global__ void __launch_bounds__(256) attn_bwd_post_kernel(const BwdParams p) {
  constexpr int G = D / 8;
  const long long nrows = (long long)p.B * p.L * p.H;
  const long long stride = (long long)gridDim.x * blockDim.x;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < nrows * G; t += stride) {
    const long long row = t / G;  // (b, i, h) in dq's memory order
    const int part = (int)(t % G);
    const int h = (int)(row % p.H);
    const long long bi = row / p.H;
    const int i = (int)(bi % p.L);
    const int b = (int)(bi / p.L);
    // d = 64: accumulator rows [B, H, L128, 64]; d = 80, 128: [B, H, ceil(d/32) chunks, L128, 32]
    constexpr int NCH = acc_cols<D>() / 32;
    const long long bh = (long long)b * p.H + h;
    const float* srcf = (D != 64) ? p.dq_acc + ((bh * NCH + (part >> 2)) * p.L128 + i) * 32 + (part & 3) * 8
                                  : p.dq_acc + (bh * p.L128 + i) * D + part * 8;
    const float4* src = reinterpret_cast<const float4*>(srcf);
    const float4 x = src[0], y = src[1];
    float f[8] = {x.x * p.scale, x.y * p.scale, x.z * p.scale, x.w * p.scale,
                  y.x * p.scale, y.y * p.scale, y.z * p.scale, y.w * p.scale};
    if (p.rope_tab) {  // dq = R^T dq_rot: pairs j = 4 part .. 4 part + 3 at position i
      const float4* t4 = reinterpret_cast<const float4*>(p.rope_tab_rows + (long long)i * (D / 2) + part * 4);
      const float4 a = t4[0], c = t4[1];
      rope_unrotate_pair(f[0], f[1], a.x, a.y);
      rope_unrotate_pair(f[2], f[3], a.z, a.w);
      rope_unrotate_pair(f[4], f[5], c.x, c.y);
      rope_unrotate_pair(f[6], f[7], c.z, c.w);
    }
    uint4 w;
    w.x = pack_bf16x2(f[0], f[1]);
    w.y = pack_bf16x2(f[2], f[3]);
    w.z = pack_bf16x2(f[4], f[5]);
    w.w = pack_bf16x2(f[6], f[7]);
    reinterpret_cast<uint4*>(p.dq + row * D)[part] = w;
  }
}

// ------------------------------------------------------------------ main
template <int D>
__global__ void __launch_bounds__(320, 1)
    attn_bwd_main_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                         const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmDO,
                         const BwdParams p) {
  using C = BwdCfg<D>;
  constexpr int BQ = C::BQ;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  BwdBars* bars = reinterpret_cast<BwdBars*>(smem + C::OFF_BAR);
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
    mbar_init(&bars->sdp_free, 4);  // per-warp arrivals (mbar_arrive_warp)
    mbar_init(&bars->p_full, 4);
    mbar_init(&bars->p_free, 1);
    mbar_init(&bars->ds_full, 4);
    mbar_init(&bars->ds_free, 1);
    mbar_init(&bars->dq_full, 1);
    mbar_init(&bars->dq_free, 4);
    mbar_init(&bars->mma_done, 1);
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
  uint8_t* sK = smem + C::OFF_K;
  uint8_t* sV = smem + C::OFF_V;
  uint8_t* sQ = smem + C::OFF_Q;
  uint8_t* sDO = smem + C::OFF_DO;
  uint8_t* sP = smem + C::OFF_P;
  uint8_t* sDS = smem + C::OFF_DS;
  float* sDQ = reinterpret_cast<float*>(smem + C::OFF_DQS);
  float* sLSE = reinterpret_cast<float*>(smem + C::OFF_LSE);
  float* sDEL = reinterpret_cast<float*>(smem + C::OFF_DEL);
  const long long vec0 = ((long long)b * p.H + h) * p.L128;  // row 0 of this (b, h) in padded vectors

  if (warp == 8) {
    // ---------------- TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      prefetch_tmap(&tmDO);
      mbar_arrive_expect_tx(&bars->kv_full, 2 * C::KV_BYTES);
      for (int blk = 0; blk < C::DB; blk++) {
        tma_load_4d(sK + blk * C::KV_BLK, &tmK, &bars->kv_full, 64 * blk, h, kv0, b);
        tma_load_4d(sV + blk * C::KV_BLK, &tmV, &bars->kv_full, 64 * blk, h, kv0, b);
      }
      int issued = 0;
      for (int i = 0; i < nq; i++) {
        const int s = i & 1;
        const int q0 = (m_lo + i) * BQ;
        if (i >= 2 && !mbar_wait(&bars->q_empty[s], ((i >> 1) - 1) & 1, wd)) break;
        mbar_arrive_expect_tx(&bars->q_full[s], 2 * C::QS_BYTES + 2 * BQ * 4);
        for (int blk = 0; blk < C::DB; blk++) {
          tma_load_4d(sQ + s * C::QS_BYTES + blk * C::QB_BLK, &tmQ, &bars->q_full[s], 64 * blk, h, q0, b);
          tma_load_4d(sDO + s * C::QS_BYTES + blk * C::QB_BLK, &tmDO, &bars->q_full[s], 64 * blk, h, q0, b);
        }
        bulk_load(sLSE + s * BQ, p.lse2_pad + vec0 + q0, BQ * 4, &bars->q_full[s]);
        bulk_load(sDEL + s * BQ, p.delta_pad + vec0 + q0, BQ * 4, &bars->q_full[s]);
        issued = i + 1;
      }
      if (*wd.abort_flag) {
        mbar_wait_drain(&bars->kv_full, 0, wd.limit_ns);
        for (int i = issued - 2 < 0 ? 0 : issued - 2; i < issued; i++)
          mbar_wait_drain(&bars->q_full[i & 1], (i >> 1) & 1, wd.limit_ns);
      }
    }
  } else if (warp == 9) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_bf16(128, BQ, false, false);   // K / V rows x Q / dO rows
      constexpr uint32_t id_kv = idesc_bf16(128, D, false, true);    // P^T / dS^T (K-major) x dO / Q (MN-major)
      constexpr uint32_t id_dq = idesc_bf16(128, 64, true, true);    // both operands MN-major
      const uint32_t aK = smem_u32(sK), aV = smem_u32(sV), aQ = smem_u32(sQ), aDO = smem_u32(sDO);
      const uint32_t aP = smem_u32(sP), aDS = smem_u32(sDS);
      if (mbar_wait(&bars->kv_full, 0, wd)) {
        for (int i = 0; i < nq; i++) {
          const int s = i & 1;
          if (!mbar_wait(&bars->q_full[s], (i >> 1) & 1, wd)) break;
          if (i >= 1 && !mbar_wait(&bars->sdp_free, (i - 1) & 1, wd)) break;
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < D / 16; ks++) {
            const uint32_t ka = (ks >> 2) * C::KV_BLK + (ks & 3) * 32;
            const uint32_t qa = s * C::QS_BYTES + (ks >> 2) * C::QB_BLK + (ks & 3) * 32;
            umma_bf16(tmem + C::TM_S, sdesc_sw128(aK + ka, 16, 1024), sdesc_sw128(aQ + qa, 16, 1024), id_s,
                      ks > 0 ? 1u : 0u);
          }
#pragma unroll
          for (int ks = 0; ks < D / 16; ks++) {
            const uint32_t ka = (ks >> 2) * C::KV_BLK + (ks & 3) * 32;
            const uint32_t qa = s * C::QS_BYTES + (ks >> 2) * C::QB_BLK + (ks & 3) * 32;
            umma_bf16(tmem + C::TM_DP, sdesc_sw128(aV + ka, 16, 1024), sdesc_sw128(aDO + qa, 16, 1024), id_s,
                      ks > 0 ? 1u : 0u);
          }
          umma_commit(&bars->s_full);
          // dV += P^T dO
          if (!mbar_wait(&bars->p_full, i & 1, wd)) break;
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < BQ / 16; ks++) {
            const uint64_t da = sdesc_sw128(aP + (ks >> 2) * C::PB_BLK + (ks & 3) * 32, 16, 1024);
            const uint64_t db = sdesc_sw128(aDO + s * C::QS_BYTES + ks * 2048, C::QB_BLK, 1024);
            umma_bf16(tmem + C::TM_DV, da, db, id_kv, (i > 0 || ks > 0) ? 1u : 0u);
          }
          umma_commit(&bars->p_free);
          // dK += dS^T Q
          if (!mbar_wait(&bars->ds_full, i & 1, wd)) break;
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < BQ / 16; ks++) {
            const uint64_t da = sdesc_sw128(aDS + (ks >> 2) * C::PB_BLK + (ks & 3) * 32, 16, 1024);
            const uint64_t db = sdesc_sw128(aQ + s * C::QS_BYTES + ks * 2048, C::QB_BLK, 1024);
            umma_bf16(tmem + C::TM_DK, da, db, id_kv, (i > 0 || ks > 0) ? 1u : 0u);
          }
          // dQ (d = 128: dQ^T = K^T dS^T; d = 64: dQ = dS K), fresh every step
          if (i >= 1 && !mbar_wait(&bars->dq_free, (i - 1) & 1, wd)) break;
          tc_fence_after();
#pragma unroll
          for (int ks = 0; ks < C::BN / 16; ks++) {
            uint64_t da, db;
            if constexpr (C::DQ_T) {
              da = sdesc_sw128(aK + ks * 2048, C::KV_BLK, 1024);
              db = sdesc_sw128(aDS + ks * 2048, C::PB_BLK, 1024);
            } else {
              da = sdesc_sw128(aDS + ks * 2048, C::PB_BLK, 1024);
              db = sdesc_sw128(aK + ks * 2048, C::KV_BLK, 1024);
            }
            umma_bf16(tmem + C::TM_DQ, da, db, id_dq, ks > 0 ? 1u : 0u);
          }
          umma_commit(&bars->dq_full);
          umma_commit(&bars->ds_free);
          umma_commit(&bars->q_empty[s]);
        }
      }
      umma_commit(&bars->mma_done);
      mbar_wait_drain(&bars->mma_done, 0, wd.limit_ns);
    }
  } else if (warp < 4) {
    // ---------------- P / dS warps: thread r <-> key row kv0 + r <-> TMEM lane r
    const int r = threadIdx.x;
    const int kv = kv0 + r;
    const int kvc = kv < p.L ? kv : p.L - 1;
    const int de = (int)(doc_end(p.offsets, p.n_offsets, seq0 + kvc, seq0 + p.L) - seq0);
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    const float sl2 = p.scale_log2;
    bool ok = true;
    for (int i = 0; i < nq && ok; i++) {
      const int s = i & 1;
      const int q0 = (m_lo + i) * BQ;
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full, i & 1, wd) && mbar_wait(&bars->q_full[s], (i >> 1) & 1, wd));
      if (!ok) break;
      tc_fence_after();
      const float* lse2 = sLSE + s * BQ;
      const float* del = sDEL + s * BQ;
      const bool need_mask = (q0 < kv) || (q0 + BQ > de);
#pragma unroll 1
      for (int c0 = 0; c0 < BQ; c0 += 32) {
        uint32_t sv[32], dp[32];
        tmem_ld32(tl + C::TM_S + c0, sv);
        tmem_ld32(tl + C::TM_DP + c0, dp);
        tmem_ld_wait(sv);
        tmem_ld_wait(dp);
        float pv[32], dsv[32];
#pragma unroll
        for (int e = 0; e < 32; e++) {
          const int q = q0 + c0 + e;
          float pe = exp2_approx(fmaf(__uint_as_float(sv[e]), sl2, -lse2[c0 + e]));
          if (need_mask && (q < kv || q >= de)) pe = 0.f;
          pv[e] = pe;
          dsv[e] = pe * (__uint_as_float(dp[e]) - del[c0 + e]);
        }
        // P^T row chunk -> sP (wait for the previous dV to release it)
        if (c0 == 0 && i >= 1) {
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->p_free, (i - 1) & 1, wd));
          if (!ok) break;
        }
#pragma unroll
        for (int cc = 0; cc < 4; cc++) {
          const int chunk = (c0 >> 3) + cc;  // 16-byte chunk of the 128-column... row of BQ bf16
          const uint32_t addr = smem_u32(sP) + (chunk >> 3) * C::PB_BLK + sw128_offset(r, chunk & 7);
          st_shared_v4(addr, pack_bf16x2(pv[8 * cc], pv[8 * cc + 1]), pack_bf16x2(pv[8 * cc + 2], pv[8 * cc + 3]),
                       pack_bf16x2(pv[8 * cc + 4], pv[8 * cc + 5]), pack_bf16x2(pv[8 * cc + 6], pv[8 * cc + 7]));
        }
        if (c0 == 0 && i >= 1) {
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->ds_free, (i - 1) & 1, wd));
          if (!ok) break;
        }
#pragma unroll
        for (int cc = 0; cc < 4; cc++) {
          const int chunk = (c0 >> 3) + cc;
          const uint32_t addr = smem_u32(sDS) + (chunk >> 3) * C::PB_BLK + sw128_offset(r, chunk & 7);
          st_shared_v4(addr, pack_bf16x2(dsv[8 * cc], dsv[8 * cc + 1]),
                       pack_bf16x2(dsv[8 * cc + 2], dsv[8 * cc + 3]), pack_bf16x2(dsv[8 * cc + 4], dsv[8 * cc + 5]),
                       pack_bf16x2(dsv[8 * cc + 6], dsv[8 * cc + 7]));
        }
      }
      if (!ok) break;
      // S^T / dP^T fully read; P^T and dS^T written.
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive_warp(&bars->sdp_free);
      mbar_arrive_warp(&bars->p_full);
      mbar_arrive_warp(&bars->ds_full);
    }
    // Epilogue: dV rows.
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, 0, wd));
    if (ok) {
      tc_fence_after();
      __nv_bfloat16* dst = p.dv + ((seq0 + kvc) * p.H + h) * D;
#pragma unroll 1
      for (int c = 0; c < D / 32; c++) {
        uint32_t v[32];
        tmem_ld32(tl + C::TM_DV + c * 32, v);
        tmem_ld_wait(v);
        if (kv < p.L) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + c * 32);
#pragma unroll
          for (int q = 0; q < 4; q++)
            d4[q] = make_uint4(pack_bf16x2(__uint_as_float(v[8 * q]), __uint_as_float(v[8 * q + 1])),
                               pack_bf16x2(__uint_as_float(v[8 * q + 2]), __uint_as_float(v[8 * q + 3])),
                               pack_bf16x2(__uint_as_float(v[8 * q + 4]), __uint_as_float(v[8 * q + 5])),
                               pack_bf16x2(__uint_as_float(v[8 * q + 6]), __uint_as_float(v[8 * q + 7])));
        }
      }
    }
  } else {
    // ---------------- dQ drain warps 4-7 (TMEM lane quarter = warp - 4), then dK rows
    const int t = threadIdx.x - 128;
    const uint32_t tl = tmem + ((uint32_t)((warp - 4) * 32) << 16);
    // Every drain warp runs the same sequence of named barriers even after an
    // abort (work is skipped, barriers are not).
    bool ok = true;
    for (int i = 0; i < nq; i++) {
      ok = __all_sync(0xffffffffu, ok && mbar_wait(&bars->dq_full, i & 1, wd));
      uint32_t v0[32], v1[32];
      if (ok) {
        tc_fence_after();
        tmem_ld32(tl + C::TM_DQ, v0);
        tmem_ld32(tl + C::TM_DQ + 32, v1);
        tmem_ld_wait(v0);
        tmem_ld_wait(v1);
        tc_fence_before();
        mbar_arrive_warp(&bars->dq_free);
      }
      if (t == 0) bulk_wait_read<0>();  // previous reduction has read the staging tile
      named_bar_sync(1, 128);
      if (ok) {
        if constexpr (C::DQ_T) {
          // thread t holds column d = t for query rows 0..63: staging is [BQ][D] row-major
#pragma unroll
          for (int e = 0; e < 32; e++) {
            sDQ[e * D + t] = __uint_as_float(v0[e]);
            sDQ[(32 + e) * D + t] = __uint_as_float(v1[e]);
          }
        } else {
          // thread t holds query row t, columns d = 0..63
          float4* row4 = reinterpret_cast<float4*>(sDQ + t * D);
#pragma unroll
          for (int e = 0; e < 8; e++) {
            row4[e] = make_float4(__uint_as_float(v0[4 * e]), __uint_as_float(v0[4 * e + 1]),
                                  __uint_as_float(v0[4 * e + 2]), __uint_as_float(v0[4 * e + 3]));
            row4[8 + e] = make_float4(__uint_as_float(v1[4 * e]), __uint_as_float(v1[4 * e + 1]),
                                      __uint_as_float(v1[4 * e + 2]), __uint_as_float(v1[4 * e + 3]));
          }
        }
        fence_proxy_async_smem();
      }
      named_bar_sync(1, 128);
      if (t == 0 && ok) {
        const int q0 = (m_lo + i) * BQ;
        bulk_reduce_add_f32(p.dq_acc + (vec0 + q0) * D, sDQ, C::DQS_BYTES);
        bulk_commit();
      }
    }
    if (t == 0) bulk_wait<0>();
    // Epilogue: dK rows (scaled).
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->mma_done, 0, wd));
    if (ok) {
      tc_fence_after();
      const int kv = kv0 + t;
      const int kvc = kv < p.L ? kv : p.L - 1;
      __nv_bfloat16* dst = p.dk + ((seq0 + kvc) * p.H + h) * D;
#pragma unroll 1
      for (int c = 0; c < D / 32; c++) {
        uint32_t v[32];
        tmem_ld32(tl + C::TM_DK + c * 32, v);
        tmem_ld_wait(v);
        if (kv < p.L) store_dk_row32(dst + c * 32, v, p.scale, p.rope_tab, kv, D, c * 8, 32);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

// Sequences of at most this many key tiles take the dQ-owned walk of the d = 80 / 128 main
// kernel: its CTAs own whole (sequence, head) pairs, keep their fp32 dQ rows in an L2-resident
// slot and write bf16 dq themselves, so the accumulator is neither zeroed (pre) nor converted
// (post). Measured against the shared accumulator in one process (H = 16, d = 128, 65536
// tokens): backward 0.742 -> 0.709 ms at L = 256, but 0.912 -> 0.943 at 512, 1.178 -> 1.423
// at 1024 and 1.642 -> 1.929 at 2048 (at 512 again with the dQ-owned walk's transposed dV
// epilogue: 0.926 -> 0.950). Per CTA the slot and the re-read window of its pair's
// Q / dO tiles grow with L (0.5 MB each at L = 1024, times 152 CTAs), so they fall out of L2,
// while the per-key-tile walk shares each Q / dO tile between the CTAs that work on one pair
// at the same time; and each pair's conversion holds the drain warps.
constexpr int kDqOwnedMaxTiles = 2;

template <int D>
static cudaError_t launch_bwd_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                const CUtensorMap& tdo, const BwdParams& p_in, int phases, cudaStream_t stream) {
  using C = BwdCfg<D>;
  BwdParams p = p_in;
  p.dq_owned = (D != 64 && p.nkt <= kDqOwnedMaxTiles) ? 1 : 0;
  static DeviceCache nsm_dev;
  int nsm = 0;
  // d = 64 has its own main kernel (its shared memory set here); the pre / post kernels use
  // none, and the d = 80 / 128 main kernels are set up by their launchers.
  cudaError_t e;
  if constexpr (D == 64)
    e = kernel_setup(nsm_dev, attn_bwd_main_kernel<D>, C::SMEM_BYTES, &nsm);
  else
    e = kernel_setup(nsm_dev, attn_bwd_pre_kernel<D>, 0, &nsm);
  if (e != cudaSuccess) return e;
  const long long work = (long long)p.B * p.L * p.H * (D / 8);
  const int ew_blocks = (int)std::min<long long>((work + 255) / 256, (long long)nsm * 8);
  if (phases & 1) {
    if (p.rope_tab && (e = launch_rope_table(p.L, D, p.rope, p.rope_tab, p.rope_tab_rows, stream)) != cudaSuccess)
      return e;
    attn_bwd_pre_kernel<D><<<ew_blocks, 256, 0, stream>>>(p);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  if (phases & 2) {
    if constexpr (D != 64) {
      if ((e = launch_attn_bwd_main_d128(D, tq, tk, tv, tdo, p, stream)) != cudaSuccess) return e;
    } else {
      dim3 grid(p.nkt, p.H, p.B);
      attn_bwd_main_kernel<D><<<grid, C::THREADS, C::SMEM_BYTES, stream>>>(tq, tk, tv, tdo, p);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  if ((phases & 4) && !p.dq_owned) {
    attn_bwd_post_kernel<D><<<ew_blocks, 256, 0, stream>>>(p);
    e = cudaGetLastError();
  }
  return e;
}

cudaError_t launch_attn_bwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const CUtensorMap& tdo, const BwdParams& p, int phases, cudaStream_t stream) {
  if (d == 64) return launch_bwd_d<64>(tq, tk, tv, tdo, p, phases, stream);
  if (d == 80) return launch_bwd_d<80>(tq, tk, tv, tdo, p, phases, stream);
  return launch_bwd_d<128>(tq, tk, tv, tdo, p, phases, stream);
}

}  // namespace ddattn
