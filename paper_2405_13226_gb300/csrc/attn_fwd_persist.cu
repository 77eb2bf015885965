// Persistent causal / document-masked attention forward for sm_103a.
//
// Same arithmetic as attn_fwd_kernel (one 128-row query tile against its live
// 128-key tiles, online softmax in the log2 domain with lazy rescale, P kept
// in TMEM as the A operand of O += P V), but one CTA per SM walks a list of
// work items (query tile, head, sequence) so that nothing is exposed between
// items: the TMA producers load the next item's Q and K / V tiles while the
// current item computes, the MMA thread issues the next item's first S tiles
// while the softmax warps run the current item's epilogue, and every buffer is
// double-buffered across items:
//   smem  Q[2], K ring (3 stages), V ring (2 stages)
//   TMEM  S[2] at columns 0 / 128 (P over their first 64 columns),
//         O[2] at columns 256 / 384 (item parity)
// Items are numbered (sequence, head)-major with the heaviest query tile of a
// (sequence, head) first, and CTA c takes items c, c + G, c + 2G, ...: the
// items in flight at any time are neighbours, so they share K / V tiles in L2.
// G (the grid) is the SM count lowered until it is coprime with the number of
// query tiles, so that every CTA cycles through light and heavy tiles.
// Warp roles as in attn_fwd_kernel: warps 0-3 softmax + epilogue, warp 4 Q/K
// producer and TMEM owner, warp 5 V producer, warp 6 MMA issuer.
#include <algorithm>

#include "common.cuh"

namespace ddattn {

template <int D>
struct FwdPCfg {
  static constexpr int BM = 128, BN = 128;
  static constexpr int KST = 2, VST = 2;               // 3-stage K or V rings measured no faster here
  static constexpr int DB = (D + 63) / 64;
  static constexpr int DCH = (D + 31) / 32;
  static constexpr int BLK = 128 * 128;                // [128 rows][64] bf16, 128B swizzle
  static constexpr int TILE = DB * BLK;
  static constexpr int OFF_Q = 0;                      // 2 buffers
  static constexpr int OFF_K = OFF_Q + 2 * TILE;       // KST stages
  static constexpr int OFF_V = OFF_K + KST * TILE;     // VST stages
  static constexpr int OFF_BAR = OFF_V + VST * TILE;
  static constexpr int SMEM_BYTES = OFF_BAR + 256 + 1024;
  static constexpr uint32_t TMEM_S = 0, TMEM_O = 256;  // S[k] at 128 k, O[k] at 256 + 128 k
  static constexpr int THREADS = 224;
};

struct FwdPBars {
  uint64_t q_full[2], q_empty[2];
  uint64_t k_full[2], k_empty[2], v_full[2], v_empty[2];
  uint64_t s_full[2], p_full[2], pv_done[2];
  uint64_t o_full[2], o_empty[2];
  uint64_t mma_drain;
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(FwdPBars) <= 256, "barrier block");

struct FwdItem {
  int m, h, b, n_lo, nt;
  long long seq0;
};

// Item u: (sequence, head) group u / nqt, query tile nqt - 1 - u % nqt (heaviest
// first); live key tiles [n_lo, m] from the causal diagonal and the document
// start of the tile's first row.
__device__ __forceinline__ FwdItem fwd_item(const FwdParams& p, int u) {
  FwdItem it;
  const int g = u / p.nqt;
  it.m = p.nqt - 1 - (u - g * p.nqt);
  it.h = g % p.H;
  it.b = g / p.H;
  it.seq0 = (long long)it.b * p.L;
  const int ds0 = (int)(doc_start(p.offsets, p.n_offsets, it.seq0 + it.m * 128, it.seq0) - it.seq0);
  it.n_lo = ds0 / 128;
  it.nt = it.m - it.n_lo + 1;
  return it;
}

template <int D>
__global__ void __launch_bounds__(224, 1)
    attn_fwd_persist_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                            const __grid_constant__ CUtensorMap tmV, const FwdParams p) {
  using C = FwdPCfg<D>;
  constexpr int KST = C::KST, VST = C::VST;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  FwdPBars* bars = reinterpret_cast<FwdPBars*>(smem + C::OFF_BAR);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_items = p.nqt * p.H * p.B;
  const int G = gridDim.x;
  Watchdog wd{&bars->abort_flag, p.status, p.timeout_ns};

  if (threadIdx.x == 0) {
    bars->abort_flag = 0;
    for (int i = 0; i < 2; i++) {
      mbar_init(&bars->q_full[i], 1);
      mbar_init(&bars->q_empty[i], 1);
      mbar_init(&bars->v_full[i], 1);
      mbar_init(&bars->v_empty[i], 1);
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->p_full[i], 128);
      mbar_init(&bars->pv_done[i], 1);
      mbar_init(&bars->o_full[i], 1);
      mbar_init(&bars->o_empty[i], 128);
    }
    for (int i = 0; i < KST; i++) {
      mbar_init(&bars->k_full[i], 1);
      mbar_init(&bars->k_empty[i], 1);
    }
    mbar_init(&bars->mma_drain, 1);
    fence_mbar_init();
  }
  if (warp == 4) {
    tmem_alloc(&bars->tmem_base, 512);
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
      int kc = 0, qi = 0;  // K tiles / Q tiles issued by this CTA
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_items; u += G) {
        const FwdItem it = fwd_item(p, u);
        const int qb = qi & 1;
        if (qi >= 2 && !(ok = mbar_wait(&bars->q_empty[qb], ((qi >> 1) - 1) & 1, wd))) break;
        mbar_arrive_expect_tx(&bars->q_full[qb], C::TILE);
        for (int blk = 0; blk < C::DB; blk++)
          tma_load_4d(sQ + qb * C::TILE + blk * C::BLK, &tmQ, &bars->q_full[qb], 64 * blk, it.h, it.m * 128, it.b);
        qi++;
        for (int j = 0; j < it.nt; j++, kc++) {
          const int s = kc % KST;
          if (kc >= KST && !(ok = mbar_wait(&bars->k_empty[s], ((kc / KST) - 1) & 1, wd))) break;
          mbar_arrive_expect_tx(&bars->k_full[s], C::TILE);
          for (int blk = 0; blk < C::DB; blk++)
            tma_load_4d(sK + s * C::TILE + blk * C::BLK, &tmK, &bars->k_full[s], 64 * blk, it.h,
                        (it.n_lo + j) * 128, it.b);
        }
      }
      if (!ok) {  // let in-flight copies land before the CTA exits
        for (int i = qi >= 2 ? qi - 2 : 0; i < qi; i++) mbar_wait_drain(&bars->q_full[i & 1], (i >> 1) & 1, wd.limit_ns);
        for (int i = kc >= KST ? kc - KST : 0; i < kc; i++)
          mbar_wait_drain(&bars->k_full[i % KST], (i / KST) & 1, wd.limit_ns);
      }
    }
  } else if (warp == 5) {
    // ---------------- V producer
    if (lane == 0) {
      prefetch_tmap(&tmV);
      int vc = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < n_items; u += G) {
        const FwdItem it = fwd_item(p, u);
        for (int j = 0; j < it.nt; j++, vc++) {
          const int s = vc % VST;
          if (vc >= VST && !(ok = mbar_wait(&bars->v_empty[s], ((vc / VST) - 1) & 1, wd))) break;
          mbar_arrive_expect_tx(&bars->v_full[s], C::TILE);
          for (int blk = 0; blk < C::DB; blk++)
            tma_load_4d(sV + s * C::TILE + blk * C::BLK, &tmV, &bars->v_full[s], 64 * blk, it.h,
                        (it.n_lo + j) * 128, it.b);
        }
      }
      if (!ok)
        for (int i = vc >= VST ? vc - VST : 0; i < vc; i++)
          mbar_wait_drain(&bars->v_full[i % VST], (i / VST) & 1, wd.limit_ns);
    }
  } else if (warp == 6) {
    // ---------------- MMA issuer: S(g + 1) is issued before PV(g), across items too.
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16(128, 128, false, false);  // Q, K both K-major
      constexpr uint32_t idesc_o = idesc_bf16(128, D, false, true);      // P (TMEM) x V (MN-major)
      const uint32_t aQ = smem_u32(sQ), aK = smem_u32(sK), aV = smem_u32(sV);
      // S cursor: item su (ordinal si), tile sj; PV cursor: item pu (ordinal pi), tile pj.
      int su = blockIdx.x, si = 0, sj = 0, pu = blockIdx.x, pi = 0, pj = 0;
      FwdItem sit = su < n_items ? fwd_item(p, su) : FwdItem{}, pit = sit;
      int sc = 0, pc = 0;  // S tiles / PV tiles issued (global within the CTA)
      bool ok = true;
      while (ok && (su < n_items || pc < sc)) {
        // At an item boundary with a PV still pending, start the next item's S
        // only if its Q and K are already in smem; otherwise issue the PV first,
        // so the current item's epilogue never waits on the next item's loads.
        bool do_s = su < n_items;

        if (do_s) {
          const int ks = sc % KST, sb = sc & 1, qb = si & 1;
          if (sj == 0 && !(ok = mbar_wait(&bars->q_full[qb], (si >> 1) & 1, wd))) break;
          if (!(ok = mbar_wait(&bars->k_full[ks], (sc / KST) & 1, wd))) break;
          // S[sb] holds P of tile sc - 2 until its PV has read it.
          if (sc >= 2 && !(ok = mbar_wait(&bars->pv_done[sb], ((sc >> 1) - 1) & 1, wd))) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < D / 16; kk++) {
            const uint64_t da = sdesc_sw128(aQ + qb * C::TILE + (kk >> 2) * C::BLK + (kk & 3) * 32, 16, 1024);
            const uint64_t db = sdesc_sw128(aK + ks * C::TILE + (kk >> 2) * C::BLK + (kk & 3) * 32, 16, 1024);
            umma_bf16(tmem + C::TMEM_S + sb * 128, da, db, idesc_s, kk > 0 ? 1u : 0u);
          }
          umma_commit(&bars->s_full[sb]);
          umma_commit(&bars->k_empty[ks]);
          sc++;
          if (++sj == sit.nt) {  // the item's last S: its Q buffer is free
            umma_commit(&bars->q_empty[qb]);
            sj = 0;
            si++;
            su += G;
            if (su < n_items) sit = fwd_item(p, su);
          }
        }
        if (pc < sc - 1 || (su >= n_items && pc < sc)) {
          const int vs = pc % VST, pb = pc & 1, ob = pi & 1;
          if (!(ok = mbar_wait(&bars->v_full[vs], (pc / VST) & 1, wd))) break;
          if (!(ok = mbar_wait(&bars->p_full[pb], (pc >> 1) & 1, wd))) break;
          // O[ob] was last used by item pi - 2: its epilogue must have read it.
          if (pj == 0 && pi >= 2 && !(ok = mbar_wait(&bars->o_empty[ob], ((pi >> 1) - 1) & 1, wd))) break;
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < C::BN / 16; kk++) {
            const uint64_t db = sdesc_sw128(aV + vs * C::TILE + kk * 2048, C::BLK, 1024);
            umma_bf16_ts(tmem + C::TMEM_O + ob * 128, tmem + C::TMEM_S + pb * 128 + kk * 8, db, idesc_o,
                         (pj > 0 || kk > 0) ? 1u : 0u);
          }
          umma_commit(&bars->pv_done[pb]);
          umma_commit(&bars->v_empty[vs]);
          pc++;
          if (++pj == pit.nt) {
            umma_commit(&bars->o_full[ob]);
            pj = 0;
            pi++;
            pu += G;
            if (pu < n_items) pit = fwd_item(p, pu);
          }
        }
      }
      umma_commit(&bars->mma_drain);
      mbar_wait_drain(&bars->mma_drain, 0, wd.limit_ns);
    }
  } else {
    // ---------------- softmax warps 0-3: thread r <-> query row r <-> TMEM lane r
    const int r = threadIdx.x;
    const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
    const float sl2 = p.scale_log2;
    const uint64_t sl2x2 = f32x2(sl2, sl2);
    int sc = 0, ii = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < n_items; u += G, ii++) {
      const FwdItem it = fwd_item(p, u);
      const int row = it.m * 128 + r;
      const int rowc = row < p.L ? row : p.L - 1;
      const int ds = (int)(doc_start(p.offsets, p.n_offsets, it.seq0 + rowc, it.seq0) - it.seq0);
      const int ob = ii & 1;
      const uint32_t obuf = tl + C::TMEM_O + ob * 128;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < it.nt; j++, sc++) {
        const int sb = sc & 1;
        const int kv0 = (it.n_lo + j) * 128;
        const uint32_t sbuf = tl + C::TMEM_S + sb * 128;
        ok = __all_sync(0xffffffffu, mbar_wait(&bars->s_full[sb], (sc >> 1) & 1, wd));
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
        float scv[128];
#pragma unroll
        for (int c = 0; c < 32; c++) {
          scv[c] = __uint_as_float(v0[c]);
          scv[32 + c] = __uint_as_float(v1[c]);
          scv[64 + c] = __uint_as_float(v2[c]);
          scv[96 + c] = __uint_as_float(v3[c]);
        }
        if (kv0 + 127 > row || kv0 < ds) {
#pragma unroll
          for (int c = 0; c < 128; c++) {
            const int kv = kv0 + c;
            if (kv > row || kv < ds) scv[c] = -INFINITY;
          }
        }
        float mx = scv[0];
#pragma unroll
        for (int c = 1; c < 128; c++) mx = fmaxf(mx, scv[c]);
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
          const uint64_t x = fma_f32x2(f32x2(scv[2 * c], scv[2 * c + 1]), sl2x2, negm);
          const float p0 = exp2_approx(f32x2_lo(x));
          const float p1 = exp2_approx(f32x2_hi(x));
          rs2 = add_f32x2(rs2, f32x2(p0, p1));
          if (c < 32) pk0[c] = pack_bf16x2(p0, p1);
          else pk1[c - 32] = pack_bf16x2(p0, p1);
        }
        l_run = l_run * alpha + (f32x2_lo(rs2) + f32x2_hi(rs2));
        tmem_st32(sbuf + 0, pk0);
        tmem_st32(sbuf + 32, pk1);
        // O *= alpha, after the previous tile's PV landed and before this tile's PV.
        if (__any_sync(0xffffffffu, rescale)) {
          ok = __all_sync(0xffffffffu, mbar_wait(&bars->pv_done[(sc - 1) & 1], ((sc - 1) >> 1) & 1, wd));
          if (!ok) break;
          tc_fence_after();
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
        mbar_arrive(&bars->p_full[sb]);
      }
      if (!ok) break;
      // Epilogue: O / l -> bf16, LSE = (m + log2 l) * ln2; then O[ob] is free.
      ok = __all_sync(0xffffffffu, mbar_wait(&bars->o_full[ob], (ii >> 1) & 1, wd));
      if (!ok) break;
      tc_fence_after();
      const float inv_l = l_run > 0.f ? 1.f / l_run : 0.f;
      const float m_use = (m_run == -INFINITY) ? 0.f : m_run;
      __nv_bfloat16* orow = p.o + ((it.seq0 + rowc) * p.H + it.h) * D;
#pragma unroll 1
      for (int c = 0; c < C::DCH; c++) {
        uint32_t ov[32];
        tmem_ld32(obuf + c * 32, ov);
        tmem_ld_wait(ov);
        if (row < p.L) {
          uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
          const int nv = (D - c * 32 >= 32) ? 4 : (D - c * 32) / 8;
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
      tc_fence_before();
      mbar_arrive(&bars->o_empty[ob]);
      if (row < p.L)
        p.lse[((long long)it.b * p.H + it.h) * p.L + row] =
            l_run > 0.f ? (m_use + __log2f(l_run)) * kLn2 : -INFINITY;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 4) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

static int gcd_int(int a, int b) {
  while (b) {
    const int t = a % b;
    a = b;
    b = t;
  }
  return a;
}

template <int D>
static cudaError_t launch_fwd_persist_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                        const FwdParams& p, int n_sm, cudaStream_t stream) {
  using C = FwdPCfg<D>;
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(attn_fwd_persist_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const long long n_items = (long long)p.nqt * p.H * p.B;
  int g = (int)std::min<long long>(n_items, n_sm);
  while (g > 1 && gcd_int(g, p.nqt) != 1) g--;
  attn_fwd_persist_kernel<D><<<g, C::THREADS, C::SMEM_BYTES, stream>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

cudaError_t launch_attn_fwd_persist(int d, const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv,
                                    const FwdParams& p, cudaStream_t stream) {
  static int n_sm = 0;
  if (!n_sm) {
    int dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n_sm, cudaDevAttrMultiProcessorCount, dev);
    if (n_sm < 1) n_sm = 152;
  }
  if (d == 64) return launch_fwd_persist_d<64>(tq, tk, tv, p, n_sm, stream);
  if (d == 80) return launch_fwd_persist_d<80>(tq, tk, tv, p, n_sm, stream);
  return launch_fwd_persist_d<128>(tq, tk, tv, p, n_sm, stream);
}

}  // namespace ddattn
