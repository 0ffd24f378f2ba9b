// dla_readout_intra.cu -- K2a: the intra-interval part of the read-out
// (Eq. capacity_bounded_output restricted to the tokens of the interval):
//   o_intra[t] = sum_{s <= t in interval} lambda_{t, L_t(e(s))} (q_t . k_s) v_s
// for one 128-token interval of one stream per CTA (bf16 inputs), written in
// fp32 to a scratch buffer [B*H][round tokens][d] that the snapshot part of
// the read-out (K2b) starts from.
// Warp-level tensor cores (mma.sync), causal tiles skipped:
//   P  = Q K^T           (warp w: token rows 16w.., key columns s <= 16w+15)
//   Pt = P o W           (W: the lambda of the logical slot of s's entry at t)
//   O  = Pt V            (V read transposed by ldmatrix.trans)
// L_t is rebuilt from the interval's boundary flags and merge indices as in
// the other read-out kernels: one table row per boundary event.
#include "dla_common.cuh"
#include "dla_mma.cuh"

namespace dla {

namespace {

constexpr int NT = 256;
constexpr int L = kReadoutTcInterval;  // 128 tokens per CTA
constexpr int MAXE = kMaxC + L;

template <int D>
struct IntraSmem {
  static constexpr int RP = D + 8;  // bf16 rows padded for conflict-free ldmatrix
  static constexpr int PP = L + 8;
  __nv_bfloat16 q[L * RP];
  __nv_bfloat16 k[L * RP];
  __nv_bfloat16 v[L * RP];
  __nv_bfloat16 pt[L * PP];
  unsigned char tab[(L + 1) * MAXE];
  int logi[MAXE];
  int ent[L];
  int evt[L];
  int mlog[L];
  uint8_t bnd[L];
};

}  // namespace

template <int D>
__global__ void __launch_bounds__(NT, 1) readout_intra_kernel(ReadoutArgs a) {
  constexpr int RP = D + 8;
  constexpr int PP = L + 8;
  constexpr int NJ = D / 8;  // n8 tiles over the value dimension
  extern __shared__ __align__(16) unsigned char smem_raw[];
  IntraSmem<D>& sm = *reinterpret_cast<IntraSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tg = lane & 3, q = lane >> 3, r8 = lane & 7;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, a.t_end - c0);
  const int m0 = a.snap_m0[(long long)bh * a.snap_stride + a.snap_base + s];
  const long long rowbase = ((long long)b * a.T + c0) * a.H + h;
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q);
  const __nv_bfloat16* kg = reinterpret_cast<const __nv_bfloat16*>(a.k);
  const __nv_bfloat16* vg = reinterpret_cast<const __nv_bfloat16*>(a.v);

  // ---- stage q, k, v rows and the interval's trace
  {
    constexpr int V16 = D / 8;
    for (int e = tid; e < L * V16; e += NT) {
      const int r = e / V16, cc = (e % V16) * 8;
      uint4 qv = make_uint4(0, 0, 0, 0), kv = qv, vv = qv;
      if (r < Lc) {
        const long long off = (rowbase + (long long)r * a.H) * D + cc;
        qv = *reinterpret_cast<const uint4*>(qg + off);
        kv = *reinterpret_cast<const uint4*>(kg + off);
        vv = *reinterpret_cast<const uint4*>(vg + off);
      }
      *reinterpret_cast<uint4*>(sm.q + r * RP + cc) = qv;
      *reinterpret_cast<uint4*>(sm.k + r * RP + cc) = kv;
      *reinterpret_cast<uint4*>(sm.v + r * RP + cc) = vv;
    }
    if (tid < L) {
      const bool in = tid < Lc;
      sm.bnd[tid] = in ? a.boundary[(long long)bh * a.T + c0 + tid] : (uint8_t)0;
      sm.mlog[tid] = in ? a.merge_log[(long long)bh * a.T + c0 + tid] : -1;
    }
  }
  __syncthreads();
  // ---- slot table, one row per boundary event (warp 0); events per token (warps 0-3)
  if (warp == 0) {
    for (int x = lane; x < MAXE; x += 32) {
      sm.logi[x] = (x < m0) ? x : -1;
      if (x < m0) sm.tab[x] = (unsigned char)x;
    }
    __syncwarp();
    unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
    for (int w4 = 0; w4 < 4; ++w4) {
      const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
      if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
      else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
    }
    int nent = m0, cnt = m0, ev = 0;
    while (lo64 | hi64) {
      const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
      if (lo64) lo64 &= lo64 - 1;
      else hi64 &= hi64 - 1;
      const int j = sm.mlog[tt];
      if (j >= 0) {
        for (int x = lane; x < nent; x += 32)
          if (sm.logi[x] > j) sm.logi[x] -= 1;
        cnt -= 1;
      }
      __syncwarp();
      if (lane == 0) sm.logi[nent] = cnt;
      nent += 1;
      cnt += 1;
      ev += 1;
      __syncwarp();
      for (int x = lane; x < nent; x += 32) sm.tab[ev * MAXE + x] = (unsigned char)sm.logi[x];
      __syncwarp();
    }
  }
  if (warp < 4) {
    const int tt = tid;
    int e = 0;
#pragma unroll
    for (int w4 = 0; w4 < 4; ++w4) {
      const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
      if (32 * w4 + 31 <= tt) e += __popc(m);
      else if (32 * w4 <= tt) e += __popc(m & (0xffffffffu >> (31 - (tt - 32 * w4))));
    }
    sm.evt[tt] = e;
    sm.ent[tt] = (e == 0) ? m0 - 1 : m0 + e - 1;
  }
  __syncthreads();

  // ---- P = Q K^T for this warp's 16 token rows, key tiles s <= 16 warp + 15
  const int t_lo = 16 * warp;
  float p[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) p[n][e] = 0.f;
#pragma unroll 2
  for (int kk = 0; kk < D; kk += 16) {
    uint32_t af[4];
    ldsm4(af, sm.q + (t_lo + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < 8; ++np) {
      if (np <= warp) {
        uint32_t bf[4];
        ldsm4(bf, sm.k + (16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
        mma16816(p[2 * np], af, bf[0], bf[1]);
        mma16816(p[2 * np + 1], af, bf[2], bf[3]);
      }
    }
  }
  // ---- Pt = P o W (bf16), causal and lambda-weighted
  {
    const int ta = t_lo + g, tb = ta + 8;
    const float* lam_a = (a.lam && ta < Lc) ? a.lam + (rowbase + (long long)ta * a.H) * C : nullptr;
    const float* lam_b = (a.lam && tb < Lc) ? a.lam + (rowbase + (long long)tb * a.H) * C : nullptr;
    const int ea = sm.evt[ta], eb = sm.evt[tb];
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      if (n <= 2 * warp + 1) {
        const int s0 = 8 * n + 2 * tg;
        float w[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int t = (e < 2) ? ta : tb;
          const int ss = s0 + (e & 1);
          float wt = 0.f;
          if (ss <= t && t < Lc) {
            const int li = sm.tab[((e < 2) ? ea : eb) * MAXE + sm.ent[ss]];
            const float* lr = (e < 2) ? lam_a : lam_b;
            wt = lr ? lr[li] : 1.f;
          }
          w[e] = p[n][e] * wt;
        }
        *reinterpret_cast<__nv_bfloat162*>(sm.pt + ta * PP + s0) = __floats2bfloat162_rn(w[0], w[1]);
        *reinterpret_cast<__nv_bfloat162*>(sm.pt + tb * PP + s0) = __floats2bfloat162_rn(w[2], w[3]);
      }
    }
  }
  __syncwarp();
  // ---- O = Pt V over key steps s <= 16 warp + 15
  float o[NJ][4];
#pragma unroll
  for (int n = 0; n < NJ; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[n][e] = 0.f;
  for (int ks = 0; ks <= warp; ++ks) {
    uint32_t af[4];
    ldsm4(af, sm.pt + (t_lo + (q & 1) * 8 + r8) * PP + 16 * ks + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < NJ / 2; ++np) {
      uint32_t bf[4];
      ldsm4t(bf, sm.v + (16 * ks + (q & 1) * 8 + r8) * RP + 16 * np + (q >> 1) * 8);
      mma16816(o[2 * np], af, bf[0], bf[1]);
      mma16816(o[2 * np + 1], af, bf[2], bf[3]);
    }
  }
  // ---- o_intra rows (fp32)
  {
    const int ta = t_lo + g, tb = ta + 8;
    float* orow = a.ointra + ((long long)bh * a.ointra_T + (c0 - a.t_begin)) * D;
#pragma unroll
    for (int n = 0; n < NJ; ++n) {
      const int j = 8 * n + 2 * tg;
      if (ta < Lc) *reinterpret_cast<float2*>(orow + (long long)ta * D + j) = make_float2(o[n][0], o[n][1]);
      if (tb < Lc) *reinterpret_cast<float2*>(orow + (long long)tb * D + j) = make_float2(o[n][2], o[n][3]);
    }
  }
}

cudaError_t launch_readout_intra(const ReadoutArgs& a, cudaStream_t st) {
  const size_t smem = sizeof(IntraSmem<128>);
  auto kern = readout_intra_kernel<128>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.nsnap, a.B * a.H);
  kern<<<grid, NT, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace dla
