// Causal / document-masked attention forward for sm_103a.
//
// One CTA computes one 128-row query tile of one (sequence, head):
//   O = softmax(scale * Q K^T + mask) V,  LSE = ln sum exp(scale * Q K^T + mask)
// over the live key tiles only (tile skipping from the causal diagonal and
// the first row's document start). Warp roles:
//   warps 0-3  softmax: thread r owns query row r = TMEM lane r. Reads the
//              S tile from TMEM, masks (diagonal / document-edge tiles only),
//              online max/sum in the log2 domain, writes P (bf16 pairs) back
//              over the first 64 columns of the same TMEM buffer, and
//              rescales O in TMEM when the running max grows by more than 2^8
//              (otherwise the stale max is kept; P <= 256 stays exact enough
//              in bf16/fp32).
//   warp 4     TMA producer for Q (once) and K tiles (3-stage ring); TMEM alloc.
//   warp 5     TMA producer for V tiles (3-stage ring).
//   warp 6     one thread issues tcgen05.mma: S[j%3] = Q K_j^T (TMEM, fp32),
//              then O += P_{j-1} V_{j-1} with P read from TMEM (the .ts form),
//              so the tensor core computes S_{j+1} while the softmax warps
//              work on S_j.
// TMEM: three S buffers at columns 0, 128, 256 (P over their first 64 columns),
// O at 384. With three, S_{j+2} goes to a buffer whose PV finished a tile ago,
// so the MMA thread never waits for the PV it has just issued (with two it
// did, leaving the tensor pipe idle for a PV's duration every tile).
// Head dims 64, 80, 128. Tiles are stored as 64-column swizzle blocks; for
// d = 80 the second block holds columns 64..79 and TMA zero fill beyond, and
// the contractions run at their true sizes (5 K-steps of 16 for QK^T, N = 80
// for PV).
#include "common.cuh"

namespace ddattn {

template <int D>
struct FwdCfg {
  static constexpr int BM = 128, BN = 128, STAGES = 3;
  static constexpr int DB = (D + 63) / 64;             // 64-column swizzle blocks per row (d = 80: the
                                                       // second block's columns 80..127 are TMA zero fill)
  static constexpr int DCH = (D + 31) / 32;            // 32-column TMEM chunks of O (the last may be partial)
  static constexpr int Q_BLK = BM * 128;               // bytes of one [128 rows][64] block
  static constexpr int KV_BLK = BN * 128;
  static constexpr int Q_BYTES = DB * Q_BLK;
  static constexpr int KV_BYTES = DB * KV_BLK;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_K = OFF_Q + Q_BYTES;
  static constexpr int OFF_V = OFF_K + STAGES * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + STAGES * KV_BYTES;
  static constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;
  static constexpr int PF = 4;                         // K / V tiles prefetched into L2 ahead of the ring
  static constexpr int NS = 3;                         // S buffers (P of tile j lives in buffer j % 3
                                                       // until PV_j has read it)
  static constexpr uint32_t TMEM_S = 0;                // S buffers at columns 0, 128, 256
  static constexpr uint32_t TMEM_O = 384;              // O: D columns
  static constexpr uint32_t TMEM_COLS = 512;
  static constexpr int THREADS = 224;
};

struct FwdBars {
  uint64_t q_full;
  uint64_t k_full[3], k_empty[3], v_full[3], v_empty[3];
  uint64_t s_full[3], p_full[3], pv_done[3];
  uint64_t mma_drain;
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(FwdBars) <= 256, "barrier block");

template <int D>
__global__ void __launch_bounds__(224, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV, const FwdParams p) {
  using C = FwdCfg<D>;
  constexpr int ST = C::STAGES;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  FwdBars* bars = reinterpret_cast<FwdBars*>(smem + C::OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  const int m = p.nqt - 1 - blockIdx.x;  // heaviest causal tiles first
  const int h = blockIdx.y, b = blockIdx.z;
  const long long seq0 = (long long)b * p.L;
  const int row0 = m * C::BM;
  // Live key tiles [n_lo, m]: keys before the first row's document start are
  // masked for every row of the tile (documents start in order).
  const int ds0 = (int)(doc_start(p.offsets, p.n_offsets, seq0 + row0, seq0) - seq0);
  const int n_lo = ds0 / C::BN;
  const int nt = m - n_lo + 1;
  Watchdog wd{&bars->abort_flag, p.status, p.timeout_ns};

  if (threadIdx.x == 0) {
    bars->abort_flag = 0;
    mbar_init(&bars->q_full, 1);
    for (int i = 0; i < ST; i++) {
      mbar_init(&bars->k_full[i], 1);
      mbar_init(&bars->k_empty[i], 1);
      mbar_init(&bars->v_full[i], 1);
      mbar_init(&bars->v_empty[i], 1);
    }
    for (int i = 0; i < C::NS; i++) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->p_full[i], 128);
      mbar_init(&bars->pv_done[i], 1);
    }
    mbar_init(&bars->mma_drain, 1);
    fence_mbar_init();
  }
  if (warp == 4) {
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

  if (warp == 4) {
    // ---------------- Q + K producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      mbar_arrive_expect_tx(&bars->q_full, C::Q_BYTES);
      for (int blk = 0; blk < C::DB; blk++) tma_load_4d(sQ + blk * C::Q_BLK, &tmQ, &bars->q_full, 64 * blk, h, row0, b);
      int issued = 0;
      for (int j = 0; j < nt; j++) {
        const int s = j % ST;
        if (j >= ST && !mbar_wait(&bars->k_empty[s], ((j / ST) - 1) & 1, wd)) break;
        mbar_arrive_expect_tx(&bars->k_full[s], C::KV_BYTES);
        const int kv0 = (n_lo + j) * C::BN;
        for (int blk = 0; blk < C::DB; blk++)
          tma_load_4d(sK + s * C::KV_BYTES + blk * C::KV_BLK, &tmK, &bars->k_full[s], 64 * blk, h, kv0, b);
        if (j + C::PF < nt)  // K tile j + PF into L2: the ring alone does not cover the load latency
          for (int blk = 0; blk < C::DB; blk++) tma_prefetch_4d(&tmK, 64 * blk, h, kv0 + C::PF * C::BN, b);
        issued = j + 1;
      }
      if (*wd.abort_flag) {  // let in-flight copies land before the CTA exits
        mbar_wait_drain(&bars->q_full, 0, wd.limit_ns);
        for (int j = issued - ST < 0 ? 0 : issued - ST; j < issued; j++)
          mbar_wait_drain(&bars->k_full[j % ST], (j / ST) & 1, wd.limit_ns);
      }
    }
  } else if (warp == 5) {
    // ---------------- V producer
    if (lane == 0) {
      prefetch_tmap(&tmV);
      int issued = 0;
      for (int j = 0; j < nt; j++) {
        const int s = j % ST;
        if (j >= ST && !mbar_wait(&bars->v_empty[s], ((j / ST) - 1) & 1, wd)) break;
        mbar_arrive_expect_tx(&bars->v_full[s], C::KV_BYTES);
        const int kv0 = (n_lo + j) * C::BN;
        for (int blk = 0; blk < C::DB; blk++)
          tma_load_4d(sV + s * C::KV_BYTES + blk * C::KV_BLK, &tmV, &bars->v_full[s], 64 * blk, h, kv0, b);
        if (j + C::PF < nt)
          for (int blk = 0; blk < C::DB; blk++) tma_prefetch_4d(&tmV, 64 * blk, h, kv0 + C::PF * C::BN, b);
        issued = j + 1;
      }
      if (*wd.abort_flag)
        for (int j = issued - ST < 0 ? 0 : issued - ST; j < issued; j++)
          mbar_wait_drain(&bars->v_full[j % ST], (j / ST) & 1, wd.limit_ns);
    }
  } else if (warp == 6) {
    // ---------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16(128, 128, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16(128, D, false, true);      // P (TMEM) x V (MN-major)
      // Descriptors are built once; a K-slice or ring stage is an added (byte offset >> 4)
      // on the 14-bit start-address field (smem offsets stay below 256 KB), so each
      // UMMA costs this thread one add instead of a descriptor rebuild.
      const uint64_t dQ0 = sdesc_sw128(smem_u32(sQ), 16, 1024);
      const uint64_t dK0 = sdesc_sw128(smem_u32(sK), 16, 1024);
      const uint64_t dV0 = sdesc_sw128(smem_u32(sV), C::KV_BLK, 1024);
      if (mbar_wait(&bars->q_full, 0, wd)) {
        for (int j = 0; j <= nt; j++) {
          if (j < nt) {
            const int ks = j % ST, sb = j % C::NS;
            if (!mbar_wait(&bars->k_full[ks], (j / ST) & 1, wd)) break;
            // S[sb] holds P_{j-2} until PV_{j-2} has read it.
            if (j >= C::NS && !mbar_wait(&bars->pv_done[sb], ((j / C::NS) - 1) & 1, wd)) break;
            tc_fence_after();
            const uint64_t dK = dK0 + ((uint32_t)(ks * C::KV_BYTES) >> 4);
            const uint32_t tS = tmem + C::TMEM_S + sb * 128;
#pragma unroll
            for (int kk = 0; kk < D / 16; kk++) {
              constexpr int q_blk = C::Q_BLK, kv_blk = C::KV_BLK;
              umma_bf16(tS, dQ0 + (uint32_t)(((kk >> 2) * q_blk + (kk & 3) * 32) >> 4),
                        dK + (uint32_t)(((kk >> 2) * kv_blk + (kk & 3) * 32) >> 4), idesc_s, kk > 0 ? 1u : 0u);
            }
            umma_commit(&bars->s_full[sb]);
            umma_commit(&bars->k_empty[ks]);
          }
          if (j >= 1) {
            const int i = j - 1, vs = i % ST, pb = i % C::NS;
            if (!mbar_wait(&bars->v_full[vs], (i / ST) & 1, wd)) break;
            if (!mbar_wait(&bars->p_full[pb], (i / C::NS) & 1, wd)) break;
            tc_fence_after();
            const uint64_t dV = dV0 + ((uint32_t)(vs * C::KV_BYTES) >> 4);
            const uint32_t tP = tmem + C::TMEM_S + pb * 128;
#pragma unroll
            for (int kk = 0; kk < C::BN / 16; kk++)
              umma_bf16_ts(tmem + C::TMEM_O, tP + kk * 8, dV + (uint32_t)((kk * 2048) >> 4), idesc_o,
                           (i > 0 || kk > 0) ? 1u : 0u);
            umma_commit(&bars->pv_done[pb]);
            umma_commit(&bars->v_empty[vs]);
          }
        }
      }
      umma_commit(&bars->mma_drain);
      mbar_wait_drain(&bars->mma_drain, 0, wd.limit_ns);
    }
  } else {
    // ---------------- softmax warps 0-3: thread r <-> query row r <-> TMEM lane r
    const int r = threadIdx.x;
    const int row = row0 + r;
    const int rowc = row < p.L ? row : p.L - 1;
    const int ds = (int)(doc_start(p.offsets, p.n_offsets, seq0 + rowc, seq0) - seq0);
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    const float sl2 = p.scale_log2;
    const uint64_t sl2x2 = f32x2(sl2, sl2);
    float m_run = -INFINITY, l_run = 0.f;
    bool ok = true;
    for (int j = 0; j < nt && ok; j++) {
      const int sb = j % C::NS;
      const int kv0 = (n_lo + j) * C::BN;
      const uint32_t sbuf = tl + C::TMEM_S + sb * 128;
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full[sb], (j / C::NS) & 1, wd));
      if (!ok) break;
      tc_fence_after();
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
      float mx = sc[0];
#pragma unroll
      for (int c = 1; c < 128; c++) mx = fmaxf(mx, sc[c]);
      const float m_tile = mx * sl2;
      float alpha = 1.f;
      bool rescale = false;
      if (m_tile > m_run + 8.f) {
        alpha = exp2_approx(m_run - m_tile);  // 0 when m_run = -inf
        rescale = (j > 0);
        m_run = m_tile;
      }
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
      const uint64_t negm = f32x2(-m_use, -m_use);
      uint64_t rs2 = f32x2(0.f, 0.f);
      uint32_t pk0[32], pk1[32];
#pragma unroll
      for (int c = 0; c < 64; c++) {
        const uint64_t x = fma_f32x2(f32x2(sc[2 * c], sc[2 * c + 1]), sl2x2, negm);
        const float p0 = exp2_approx(f32x2_lo(x));
        const float p1 = exp2_approx(f32x2_hi(x));
        rs2 = add_f32x2(rs2, f32x2(p0, p1));
        if (c < 32) pk0[c] = pack_bf16x2(p0, p1);
        else pk1[c - 32] = pack_bf16x2(p0, p1);
      }
      l_run = l_run * alpha + (f32x2_lo(rs2) + f32x2_hi(rs2));
      // P_j over the first 64 columns of its S buffer (all of S_j has been read).
      tmem_st32(sbuf + 0, pk0);
      tmem_st32(sbuf + 32, pk1);
      // O *= alpha, after PV_{j-1} landed and before PV_j is issued.
      if (__any_sync(0xffffffffu, rescale)) {
        ok = __all_sync(0xffffffffu, mbar_wait(&bars->pv_done[(j - 1) % C::NS], ((j - 1) / C::NS) & 1, wd));
        if (!ok) break;
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < C::DCH; c++) {  // columns past D of the last chunk are unused TMEM
          uint32_t ov[32];
          tmem_ld32(tl + C::TMEM_O + c * 32, ov);
          tmem_ld_wait(ov);
#pragma unroll
          for (int e = 0; e < 32; e++) ov[e] = __float_as_uint(__uint_as_float(ov[e]) * alpha);
          tmem_st32(tl + C::TMEM_O + c * 32, ov);
        }
      }
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&bars->p_full[sb]);
    }
    // Epilogue: O / l -> bf16, LSE = (m + log2 l) * ln2.
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&bars->pv_done[(nt - 1) % C::NS], ((nt - 1) / C::NS) & 1, wd));
    if (ok) {
      tc_fence_after();
      const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
      __nv_bfloat16* orow = p.o + (((long long)b * p.L + rowc) * p.H + h) * D;
#pragma unroll 1
      for (int c = 0; c < C::DCH; c++) {
        uint32_t ov[32];
        tmem_ld32(tl + C::TMEM_O + c * 32, ov);
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
      if (row < p.L)
        p.lse[((long long)b * p.H + h) * p.L + row] = l_run > 0.f ? (m_use + __log2f(l_run)) * kLn2 : -INFINITY;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    tc_fence_after();
    tmem_dealloc(tmem, C::TMEM_COLS);
  }
}

template <int D>
static cudaError_t launch_fwd_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                const FwdParams& p, cudaStream_t stream) {
  using C = FwdCfg<D>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  dim3 grid(p.nqt, p.H, p.B);
  attn_fwd_kernel<D><<<grid, C::THREADS, C::SMEM_BYTES, stream>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

cudaError_t launch_attn_fwd(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                            const FwdParams& p, cudaStream_t stream) {
  // Up to 16 query tiles per sequence (L <= 2048) the persistent kernel wins
  // (its loads and epilogues overlap across tiles: -3% at L = 2048 to -18% at
  // L = 256, H = 16, d = 128); for longer sequences one CTA per query tile
  // keeps the CTAs of a (sequence, head) in step and measured faster (-3% at
  // L = 4096, -8% at L = 8192).
  if (p.nqt <= 16) return launch_attn_fwd_persist(d, tq, tk, tv, p, stream);
  if (d == 64) return launch_fwd_d<64>(tq, tk, tv, p, stream);
  if (d == 80) return launch_fwd_d<80>(tq, tk, tv, p, stream);
  return launch_fwd_d<128>(tq, tk, tv, p, stream);
}

}  // namespace ddattn
