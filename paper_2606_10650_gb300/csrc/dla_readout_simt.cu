// dla_readout_simt.cu -- K2 on CUDA cores (fp32 FFMA): the read-out
// o_t = sum_i lambda_{t,i} S_i q_t of Eq. (capacity_bounded_output) for one
// 64-token interval of one stream per CTA.
//
// The cache seen by token t is the cache at the interval start (snapshot from
// K1: m0 pool entries, logical order) regrouped by the merges decided inside
// the interval, plus the interval's own tokens.  Because merges only add
// states, o_t splits into
//   sum_{x < m0} lambda_{t, L_t(x)} S_x q_t                  (snapshot part)
// + sum_{s <= t in interval} lambda_{t, L_t(e(s))} (q_t . k_s) v_s  (token part)
// where L_t(x) is the logical slot at time t of the cache entry that holds
// snapshot entry x (or token s's entry e(s)).  L_t is rebuilt here from the
// boundary flags and merge indices K1 wrote: a merge at index j lowers every
// logical slot above j by one; a boundary appends a new slot.
//
// This kernel keeps fp32 arithmetic end to end (fp32 snapshots), which the
// fp32-input path needs for its 1e-4 tolerance.
#include "dla_common.cuh"

namespace dla {

namespace {

constexpr int NT = 256;
constexpr int L = kReadoutSimtInterval;  // 64 tokens per CTA
constexpr int MAXE = kMaxC + L;          // snapshot entries + entries opened in the interval

template <int D>
struct RoSmem {
  static constexpr int KP = D + 4;
  float Q[L * KP];
  float K[L * KP];
  float V[L * KP];
  float S[D * KP];          // snapshot entry, fp32 [d_v][d_k] (padded rows)
  float P[L * (L + 1)];     // lambda-weighted q.k of the token part
  float wpre[L * kMaxC];    // lambda_{t, L_t(x)} of the snapshot entries
  unsigned char tab[L * MAXE];  // L_t(x)
  int logi[MAXE];
  int ent[L];
  int ids[kMaxC];
};

template <int D, typename Tin>
__device__ __forceinline__ void load_rows(float* dst, const Tin* src, int row_stride, int valid) {
  constexpr int KP = D + 4;
  constexpr int V4 = D / 4;
  for (int e = threadIdx.x; e < L * V4; e += NT) {
    int r = e / V4, c = (e % V4) * 4;
    float4 val = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < valid) val = load4(src + (long long)r * row_stride + c);
    store4(dst + r * KP + c, val);
  }
}

}  // namespace

template <int D, typename Tin, typename Tpool, typename Tout>
__global__ void __launch_bounds__(NT, 1) readout_simt_kernel(ReadoutArgs a) {
  constexpr int KP = D + 4;
  constexpr int TJ = D / 16;
  extern __shared__ __align__(16) unsigned char smem_raw[];
  RoSmem<D>& sm = *reinterpret_cast<RoSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, row_t_end(a.seq_lens, b, a.t_begin, a.t_end) - c0);
  if (Lc <= 0) return;  // the interval lies past this row's length: padding, o not written
  const int row_stride = a.H * D;
  const long long tok0 = (row_tok0(a.row_start, b, a.T) + c0) * a.H + h;  // row index of token c0
  const int m0 = a.snap_m0[(long long)bh * a.snap_stride + a.snap_base + s];
  const uint8_t* bnd = a.boundary + (long long)bh * a.T + c0;
  const int32_t* mlog = a.merge_log + (long long)bh * a.T + c0;

  load_rows<D, Tin>(sm.Q, reinterpret_cast<const Tin*>(a.q) + tok0 * D, row_stride, Lc);
  load_rows<D, Tin>(sm.K, reinterpret_cast<const Tin*>(a.k) + tok0 * D, row_stride, Lc);
  load_rows<D, Tin>(sm.V, reinterpret_cast<const Tin*>(a.v) + tok0 * D, row_stride, Lc);
  for (int i = tid; i < m0; i += NT) sm.ids[i] = a.snap_ids[((long long)bh * a.snap_stride + a.snap_base + s) * C + i];

  // ---- logical slot of every entry at every token (warp 0)
  if (warp == 0) {
    for (int x = lane; x < MAXE; x += 32) sm.logi[x] = (x < m0) ? x : -1;
    __syncwarp();
    int nent = m0, cnt = m0, open = m0 - 1;
    for (int t = 0; t < Lc; ++t) {
      if (bnd[t]) {
        const int j = mlog[t];
        if (j >= 0) {
          for (int x = lane; x < nent; x += 32)
            if (sm.logi[x] > j) sm.logi[x] -= 1;
          cnt -= 1;
        }
        __syncwarp();
        if (lane == 0) sm.logi[nent] = cnt;
        open = nent;
        nent += 1;
        cnt += 1;
        __syncwarp();
      }
      if (lane == 0) sm.ent[t] = open;
      for (int x = lane; x < nent; x += 32) sm.tab[t * MAXE + x] = (unsigned char)sm.logi[x];
      __syncwarp();
    }
  }
  __syncthreads();
  // ---- lambda weights
  for (int e = tid; e < L * kMaxC; e += NT) {
    int t = e / kMaxC, x = e % kMaxC;
    float w = 0.f;
    if (t < Lc && x < m0) {
      int li = sm.tab[t * MAXE + x];
      w = a.lam ? a.lam[(tok0 + (long long)t * a.H) * C + li] : 1.f;
    }
    sm.wpre[e] = w;
  }
  {  // token part: P[t][s] = lambda_{t, L_t(e(s))} (q_t . k_s), s <= t
    const int tt = tid / 16, ss = tid % 16;
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    for (int e = 0; e < D; e += 4) {
      float4 qv[4], kv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        qv[i] = load4(sm.Q + (tt * 4 + i) * KP + e);
        kv[i] = load4(sm.K + (ss * 4 + i) * KP + e);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j)
          acc[i][j] += qv[i].x * kv[j].x + qv[i].y * kv[j].y + qv[i].z * kv[j].z + qv[i].w * kv[j].w;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        int t = tt * 4 + i, u = ss * 4 + j;
        float w = 0.f;
        if (u <= t && t < Lc) {
          int li = sm.tab[t * MAXE + sm.ent[u]];
          w = a.lam ? a.lam[(tok0 + (long long)t * a.H) * C + li] : 1.f;
        }
        sm.P[t * (L + 1) + u] = acc[i][j] * w;
      }
  }
  __syncthreads();
  // ---- O = P V + sum_x wpre[:, x] * (Q S_x^T)
  const int tb = tid % 16, jb = tid / 16;  // tokens tb*4..+3, rows jb*TJ..+TJ-1
  float o[4][TJ];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int r = 0; r < TJ; ++r) o[i][r] = 0.f;
  for (int u = 0; u < L; ++u) {
    float pv[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) pv[i] = sm.P[(tb * 4 + i) * (L + 1) + u];
#pragma unroll
    for (int r4 = 0; r4 < TJ; r4 += 4) {
      float4 v4 = load4(sm.V + u * KP + jb * TJ + r4);
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        o[i][r4] += pv[i] * v4.x;
        o[i][r4 + 1] += pv[i] * v4.y;
        o[i][r4 + 2] += pv[i] * v4.z;
        o[i][r4 + 3] += pv[i] * v4.w;
      }
    }
  }
  const Tpool* pool = reinterpret_cast<const Tpool*>(a.pool) + (long long)bh * a.pool_cap * D * D;
  for (int x = 0; x < m0; ++x) {
    __syncthreads();
    const Tpool* src = pool + (long long)sm.ids[x] * D * D;
    for (int e = tid * 4; e < D * D; e += NT * 4) {
      int r = e / D, cc = e % D;
      store4(sm.S + r * KP + cc, load4(src + e));
    }
    __syncthreads();
    float y[4][TJ];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int r = 0; r < TJ; ++r) y[i][r] = 0.f;
    for (int kk = 0; kk < D; kk += 4) {
      float4 qv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) qv[i] = load4(sm.Q + (tb * 4 + i) * KP + kk);
#pragma unroll
      for (int r = 0; r < TJ; ++r) {
        float4 s4 = load4(sm.S + (jb * TJ + r) * KP + kk);
#pragma unroll
        for (int i = 0; i < 4; ++i) y[i][r] += qv[i].x * s4.x + qv[i].y * s4.y + qv[i].z * s4.z + qv[i].w * s4.w;
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      float w = sm.wpre[(tb * 4 + i) * kMaxC + x];
#pragma unroll
      for (int r = 0; r < TJ; ++r) o[i][r] += w * y[i][r];
    }
  }
  // ---- write o
  Tout* out = reinterpret_cast<Tout*>(a.o);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int t = tb * 4 + i;
    if (t < Lc) {
      Tout* row = out + (tok0 + (long long)t * a.H) * D + jb * TJ;
#pragma unroll
      for (int r4 = 0; r4 < TJ; r4 += 4) store4(row + r4, make_float4(o[i][r4], o[i][r4 + 1], o[i][r4 + 2], o[i][r4 + 3]));
    }
  }
}

template <int D, typename Tin, typename Tpool, typename Tout>
static cudaError_t launch_ro_t(const ReadoutArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(RoSmem<D>);
  auto kern = readout_simt_kernel<D, Tin, Tpool, Tout>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.nsnap, a.B * a.H);
  kern<<<grid, NT, smem, st>>>(a);
  return cudaGetLastError();
}

template <int D, typename Tin, typename Tpool>
static cudaError_t launch_ro_o(const ReadoutArgs& a, cudaStream_t st) {
  return a.out_bf16 ? launch_ro_t<D, Tin, Tpool, __nv_bfloat16>(a, st) : launch_ro_t<D, Tin, Tpool, float>(a, st);
}

// fp32 pool entries (the scans of the configurations this read-out serves write them)
template <int D>
static cudaError_t launch_ro_d(const ReadoutArgs& a, bool in_bf16, cudaStream_t st) {
  return in_bf16 ? launch_ro_o<D, __nv_bfloat16, float>(a, st) : launch_ro_o<D, float, float>(a, st);
}

cudaError_t launch_readout_simt(const ReadoutArgs& a, int d, bool in_bf16, cudaStream_t st) {
  return d == 128 ? launch_ro_d<128>(a, in_bf16, st) : launch_ro_d<64>(a, in_bf16, st);
}

}  // namespace dla
