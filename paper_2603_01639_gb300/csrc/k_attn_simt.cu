// Tree attention on CUDA cores (LTD section 3.2, "Draft Tree Verification";
// tree mask as in SpecInfer).  Serves fp32 inputs and head dims the tensor-core
// kernel does not take.
//
// Grid (row tiles, KV heads, batch); a CTA owns 16 query rows of one KV head
// (row r = slot * G + g, query head = kv * G + g), so every K/V tile staged in
// shared memory is reused by all G heads of the group.  Keys stream in tiles
// of 32: lane j scores key j against one row (q pre-scaled), the row's online
// softmax (max, sum) lives in the warp, and each lane accumulates D/32 output
// dims.  Keys 0..ctx-1 are always visible; key ctx+j is visible to slot i iff
// bit j of mask row i is set; keys from ctx+N on are never read.
#include "ltd_common.cuh"
#include "ltd_internal.h"

namespace ltd {

namespace {

constexpr int kRowsPerWarp = 4;
constexpr int kWarps = 4;
constexpr int kRows = kRowsPerWarp * kWarps;  // 16 rows per CTA
constexpr int kKeys = 32;

template <typename T, int D>
__global__ void __launch_bounds__(kWarps * kWarp) attn_simt_kernel(const AttnParams p) {
  constexpr int DU = D / kWarp;
  __shared__ float Qs[kRows][D];
  __shared__ float Ks[kKeys][D + 1];
  __shared__ float Vs[kKeys][D];
  grid_wait();
  trigger_dependents();

  const int tile = blockIdx.x, kvh = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int G = p.hq / p.hkv;
  const int ctx = p.ctx[b];
  const int N = p.n_verify[b];
  if (N < 1 || N > p.n_max || ctx < 0 || ctx > p.max_ctx || ctx + N > p.s_cap) {
    if (tid == 0 && tile == 0 && kvh == 0)
      flag_error(p.err, (N < 1 || N > p.n_max) ? LTD_DEVERR_NVERIFY : LTD_DEVERR_CTX);
    return;
  }
  const int M = N * G;
  const int row0 = tile * kRows;
  if (row0 >= M) return;
  const int W32 = (p.n_max + 31) / 32;

  const T* q = reinterpret_cast<const T*>(p.q);
  const T* kc = reinterpret_cast<const T*>(p.k) +
                (static_cast<int64_t>(b) * p.hkv + kvh) * p.s_cap * D;
  const T* vc = reinterpret_cast<const T*>(p.v) +
                (static_cast<int64_t>(b) * p.hkv + kvh) * p.s_cap * D;

  // stage this CTA's query rows, pre-scaled
  for (int idx = tid; idx < kRows * D; idx += kWarps * kWarp) {
    const int r = idx / D, t = idx % D;
    const int R = row0 + r;
    float val = 0.f;
    if (R < M) {
      const int slot = R / G, g = R % G;
      val = to_f<T>(q[((static_cast<int64_t>(b) * p.n_max + slot) * p.hq + kvh * G + g) * D + t]) *
            p.scale;
    }
    Qs[r][t] = val;
  }

  float mrow[kRowsPerWarp], lrow[kRowsPerWarp], o[kRowsPerWarp][DU];
#pragma unroll
  for (int rr = 0; rr < kRowsPerWarp; ++rr) {
    mrow[rr] = -CUDART_INF_F;
    lrow[rr] = 0.f;
#pragma unroll
    for (int u = 0; u < DU; ++u) o[rr][u] = 0.f;
  }

  const int n_keys = ctx + N;
  for (int kb = 0; kb < n_keys; kb += kKeys) {
    __syncthreads();
    for (int idx = tid; idx < kKeys * D; idx += kWarps * kWarp) {
      const int j = idx / D, t = idx % D;
      const int key = kb + j;
      float kv = 0.f, vv = 0.f;
      if (key < n_keys) {
        kv = to_f<T>(kc[static_cast<int64_t>(key) * D + t]);
        vv = to_f<T>(vc[static_cast<int64_t>(key) * D + t]);
      }
      Ks[j][t] = kv;
      Vs[j][t] = vv;
    }
    __syncthreads();
    const int key = kb + lane;
#pragma unroll
    for (int rr = 0; rr < kRowsPerWarp; ++rr) {
      const int r = warp * kRowsPerWarp + rr;
      const int R = row0 + r;
      if (R >= M) continue;  // warp-uniform
      const int slot = R / G;
      bool vis = key < ctx;
      if (!vis && key < n_keys) {
        const int js = key - ctx;
        const uint32_t w =
            p.mask[(static_cast<int64_t>(b) * p.n_max + slot) * W32 + (js >> 5)];
        vis = (w >> (js & 31)) & 1u;
      }
      float sc = 0.f;
#pragma unroll 8
      for (int t = 0; t < D; ++t) sc = fmaf(Qs[r][t], Ks[lane][t], sc);
      sc = vis ? sc : -CUDART_INF_F;
      const float tmax = warp_max_f(sc);
      const float mnew = fmaxf(mrow[rr], tmax);
      if (mnew == -CUDART_INF_F) continue;  // nothing visible yet
      const float alpha = __expf(mrow[rr] - mnew);
      const float pj = vis ? __expf(sc - mnew) : 0.f;
      lrow[rr] = lrow[rr] * alpha + warp_sum_f(pj);
      mrow[rr] = mnew;
#pragma unroll
      for (int u = 0; u < DU; ++u) o[rr][u] *= alpha;
#pragma unroll 4
      for (int j = 0; j < kKeys; ++j) {
        const float pb = __shfl_sync(0xFFFFFFFFu, pj, j);
#pragma unroll
        for (int u = 0; u < DU; ++u) o[rr][u] = fmaf(pb, Vs[j][lane + kWarp * u], o[rr][u]);
      }
    }
  }

  T* out = reinterpret_cast<T*>(p.out);
#pragma unroll
  for (int rr = 0; rr < kRowsPerWarp; ++rr) {
    const int R = row0 + warp * kRowsPerWarp + rr;
    if (R >= M) continue;
    const int slot = R / G, g = R % G;
    const float inv = lrow[rr] > 0.f ? 1.f / lrow[rr] : 0.f;
    T* dst = out + ((static_cast<int64_t>(b) * p.n_max + slot) * p.hq + kvh * G + g) * D;
#pragma unroll
    for (int u = 0; u < DU; ++u) {
      const float val = o[rr][u] * inv;
      if constexpr (sizeof(T) == 2) dst[lane + kWarp * u] = __float2bfloat16_rn(val);
      else dst[lane + kWarp * u] = val;
    }
  }
}

template <typename T>
cudaError_t launch_t(const AttnParams& p, cudaStream_t s) {
  const int G = p.hq / p.hkv;
  const int tiles = (p.n_max * G + kRows - 1) / kRows;
  const dim3 grid(tiles, p.hkv, p.batch);
  const dim3 block(kWarps * kWarp);
  switch (p.d) {
    case 32: return launch(attn_simt_kernel<T, 32>, grid, block, 0, s, nullptr, 0, p);
    case 64: return launch(attn_simt_kernel<T, 64>, grid, block, 0, s, nullptr, 0, p);
    case 96: return launch(attn_simt_kernel<T, 96>, grid, block, 0, s, nullptr, 0, p);
    default: return launch(attn_simt_kernel<T, 128>, grid, block, 0, s, nullptr, 0, p);
  }
}

}  // namespace

size_t attn_simt_workspace(const AttnParams&) { return 0; }

cudaError_t launch_attn_simt(const AttnParams& p, ltd_dtype dtype, cudaStream_t s) {
  return dtype == LTD_BF16 ? launch_t<__nv_bfloat16>(p, s) : launch_t<float>(p, s);
}

}  // namespace ltd
