// Rotary position embedding of q and k (consecutive component pairs rotated by
// m * f_b^(-2j/d), m = position inside the sequence), and the (cos, sin) table
// the backward uses to rotate dq and dk back (layout of rope_tab_index).
//
// rope_qk_kernel is bound by HBM: it reads q and k once and writes q_rot and
// k_rot once (4 * B*L*H*d*2 bytes). A CTA takes kRows consecutive token rows:
// their (cos, sin) values (kRows x d/2) are computed once into shared memory
// and serve every head of both tensors; the rows of one tensor are one
// contiguous span, walked with 16-byte vectors in memory order.
#include <algorithm>

#include "common.cuh"

namespace ddattn {

namespace {
constexpr int kRows = 8;       // token rows per CTA
constexpr int kThreads = 256;
constexpr int kBatch = 4;      // 16-byte vectors in flight per thread
}  // namespace

__global__ void __launch_bounds__(kThreads) rope_qk_kernel(const __grid_constant__ RopeParams p) {
  __shared__ float2 cs[kRows][64];
  const int half = p.d / 2;
  const long long r0 = (long long)blockIdx.x * kRows;
  const int nrows = (int)(p.rows - r0 < kRows ? p.rows - r0 : kRows);
  for (int t = threadIdx.x; t < nrows * half; t += kThreads) {
    const int rr = t / half, j = t - rr * half;
    const int m = (int)((r0 + rr) % p.L);
    cs[rr][j] = rope_cos_sin(m, p.f.hi[j], p.f.lo[j]);
  }
  __syncthreads();
  const int vpr = p.H * p.d / 8;        // 16-byte vectors per token row
  const int per_tensor = nrows * vpr;
  const int total = (p.q ? 2 : 1) * per_tensor;  // q == nullptr: k only
  const long long base = r0 * p.H * p.d;
  for (int t0 = threadIdx.x; t0 < total; t0 += kThreads * kBatch) {
    uint4 x[kBatch];
#pragma unroll
    for (int u = 0; u < kBatch; u++) {
      const int t = t0 + u * kThreads;
      if (t < total) {
        const bool is_k = !p.q || t >= per_tensor;
        const int idx = (p.q && is_k) ? t - per_tensor : t;
        const uint4* src = reinterpret_cast<const uint4*>((is_k ? p.k : p.q) + base) + idx;
        x[u] = __ldcs(src);   // read once: streaming
      }
    }
#pragma unroll
    for (int u = 0; u < kBatch; u++) {
      const int t = t0 + u * kThreads;
      if (t < total) {
        const bool is_k = !p.q || t >= per_tensor;
        const int idx = (p.q && is_k) ? t - per_tensor : t;
        const int rr = idx / vpr;
        const int col = ((idx - rr * vpr) * 8) % p.d;   // head-local column of the first element
        const float2* c = &cs[rr][col >> 1];
        uint32_t w[4] = {x[u].x, x[u].y, x[u].z, x[u].w};
#pragma unroll
        for (int e = 0; e < 4; e++) {
          const float2 v = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w[e]));
          const float2 r = c[e];
          w[e] = rope_rotate_bf16x2(v.x, v.y, r.x, r.y);
        }
        uint4* dst = reinterpret_cast<uint4*>((is_k ? p.k_rot : p.q_rot) + base) + idx;
        __stcs(dst, make_uint4(w[0], w[1], w[2], w[3]));
      }
    }
  }
}

// One thread per (position m, pair-pair jj): two (cos, sin) values into the
// float4 of rope_tab_index(m, d, jj) (unless tab is null) and into the row-major copy.
__global__ void __launch_bounds__(256) rope_table_kernel(int L, int d, const __grid_constant__ RopeFreq f,
                                                         float4* tab, float2* tab_rows) {
  const int quarter = d / 4;
  const long long n = (long long)L * quarter;
  for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += (long long)gridDim.x * blockDim.x) {
    const int m = (int)(t / quarter), jj = (int)(t % quarter);
    const float2 a = rope_cos_sin(m, f.hi[2 * jj], f.lo[2 * jj]);
    const float2 b = rope_cos_sin(m, f.hi[2 * jj + 1], f.lo[2 * jj + 1]);
    if (tab) tab[rope_tab_index(m, d, jj)] = make_float4(a.x, a.y, b.x, b.y);
    reinterpret_cast<float4*>(tab_rows)[t] = make_float4(a.x, a.y, b.x, b.y);  // = [m][2jj], [m][2jj+1]
  }
}

cudaError_t launch_rope_qk(const RopeParams& p, cudaStream_t stream) {
  const long long blocks = (p.rows + kRows - 1) / kRows;
  if (blocks > 0x7fffffffLL) return cudaErrorInvalidValue;
  rope_qk_kernel<<<(unsigned)blocks, kThreads, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_rope_table(int L, int d, const RopeFreq& f, float4* tab, float2* tab_rows, cudaStream_t stream) {
  const long long n = (long long)L * (d / 4);
  const int blocks = (int)std::min<long long>((n + 255) / 256, 4096);
  rope_table_kernel<<<blocks, 256, 0, stream>>>(L, d, f, tab, tab_rows);
  return cudaGetLastError();
}

}  // namespace ddattn
