// dla_readout_intra.cu -- K2a: the intra-interval part of the read-out
// (Eq. capacity_bounded_output restricted to the tokens of the interval):
//   o_intra[t] = sum_{s <= t in interval} lambda_{t, L_t(e(s))} (q_t . k_s) v_s
// for one 128-token interval of one stream per CTA (bf16 inputs), written in
// fp32 to a scratch buffer that the snapshot part of the read-out (K2b) starts
// from.  Warp-level tensor cores (mma.sync), causal tiles skipped:
//   P  = Q K^T           (warp w: token rows 16w.., key columns s <= 16w+15)
//   Pt = P o W           (W: the lambda of the logical slot of s's entry at t)
//   O  = Pt V            (V read transposed by ldmatrix.trans)
// The entry holding token s is the one opened by the last boundary event at or
// before s (event 0: the snapshot's open state), so W only needs the slot of
// "the entry opened at event i" after event e: one table row per event.
// Shared memory (88 KB, two CTAs per SM): Q, then Pt, in one buffer; K, then V,
// in another (V streams in while Pt is formed).
//
// Scratch layout, per interval a 128 x 128 fp32 block in column-quad order:
// element (t, j) at ((j / 4) * 128 + t) * 4 + j % 4, so that the consumer (one
// token row per thread, 64 columns) reads 512 contiguous bytes per warp load.
#include "dla_common.cuh"
#include "dla_mma.cuh"

namespace dla {

namespace {

constexpr int NT = 256;
constexpr int L = kReadoutTcInterval;  // 128 tokens per CTA
constexpr int TW = L + 1;              // table row: events 0 .. L

template <int D>
struct IntraSmem {
  static constexpr int RP = D + 8;  // bf16 rows padded for conflict-free ldmatrix
  __nv_bfloat16 qp[L * RP];         // Q, then Pt (row stride RP >= L + 8)
  __nv_bfloat16 kv[L * RP];         // K, then V
  unsigned char tab[TW * TW];       // tab[e][i]: slot of the entry opened at event i, after event e
  unsigned char evt[L];             // events at or before token t
  int logi[TW];
  int mlog[L];
  uint8_t bnd[L];
};

template <int D>
__device__ __forceinline__ void stage_rows(__nv_bfloat16* dst, const __nv_bfloat16* src, long long row_stride,
                                           int valid) {
  constexpr int RP = D + 8;
  constexpr int V16 = D / 8;
  for (int e = threadIdx.x; e < L * V16; e += NT) {
    const int r = e / V16, cc = (e % V16) * 8;
    const int nbytes = (r < valid) ? 16 : 0;  // rows past the sequence end are zero-filled
    const __nv_bfloat16* s = (r < valid) ? src + r * row_stride + cc : src;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(su32(dst + r * RP + cc)), "l"(s),
                 "r"(nbytes)
                 : "memory");
  }
}

}  // namespace

template <int D>
__global__ void __launch_bounds__(NT, 2) readout_intra_kernel(ReadoutArgs a) {
  constexpr int RP = D + 8;
  constexpr int NJ = D / 8;  // n8 tiles over the value dimension
  static_assert(RP >= L + 8, "Pt reuses the Q rows");
  extern __shared__ __align__(16) unsigned char smem_raw[];
  IntraSmem<D>& sm = *reinterpret_cast<IntraSmem<D>*>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, tg = lane & 3, q = lane >> 3, r8 = lane & 7;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, a.t_end - c0);
  // with a scan running concurrently: the interval must be complete; its list
  // and trace are then read past L1 (__ldcg)
  wait_progress(a.progress, a.progress_ctas, bh, a.snap_base + s + 1, a.status);
  __syncthreads();
  const int m0 = __ldcg(a.snap_m0 + (long long)bh * a.snap_stride + a.snap_base + s);
  const long long rowbase = ((long long)b * a.T + c0) * a.H + h;
  const long long row_stride = (long long)a.H * D;
  const __nv_bfloat16* qg = reinterpret_cast<const __nv_bfloat16*>(a.q) + rowbase * D;
  const __nv_bfloat16* kg = reinterpret_cast<const __nv_bfloat16*>(a.k) + rowbase * D;
  const __nv_bfloat16* vg = reinterpret_cast<const __nv_bfloat16*>(a.v) + rowbase * D;

  // ---- Q and K rows, the interval's trace
  stage_rows<D>(sm.qp, qg, row_stride, Lc);
  stage_rows<D>(sm.kv, kg, row_stride, Lc);
  asm volatile("cp.async.commit_group;" ::: "memory");
  if (tid < L) {
    const bool in = tid < Lc;
    sm.bnd[tid] = in ? __ldcg(a.boundary + (long long)bh * a.T + c0 + tid) : (uint8_t)0;
    sm.mlog[tid] = in ? __ldcg(a.merge_log + (long long)bh * a.T + c0 + tid) : -1;
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
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
    ldsm4(af, sm.qp + (t_lo + (q & 1) * 8 + r8) * RP + kk + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < 8; ++np) {
      if (np <= warp) {
        uint32_t bf[4];
        ldsm4(bf, sm.kv + (16 * np + (q >> 1) * 8 + r8) * RP + kk + (q & 1) * 8);
        mma16816(p[2 * np], af, bf[0], bf[1]);
        mma16816(p[2 * np + 1], af, bf[2], bf[3]);
      }
    }
  }
  // ---- slot table (warp 0, which has the least P work) and events per token (warps 0-3)
  if (warp == 0) {
    // lane x owns the entries opened at events x, x + 32, ...; a merge at index
    // j moves every slot above j down by one, so no lane reads another's entries
    if (lane == 0) {
      sm.logi[0] = m0 - 1;  // the snapshot's open entry (unused when m0 = 0)
      sm.tab[0] = (unsigned char)(m0 - 1);
    }
    unsigned long long lo64 = 0, hi64 = 0;
#pragma unroll
    for (int w4 = 0; w4 < 4; ++w4) {
      const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
      if (w4 < 2) lo64 |= (unsigned long long)m << (32 * w4);
      else hi64 |= (unsigned long long)m << (32 * (w4 - 2));
    }
    int cnt = m0, ev = 0;
    while (lo64 | hi64) {
      const int tt = lo64 ? (__ffsll((long long)lo64) - 1) : (64 + __ffsll((long long)hi64) - 1);
      if (lo64) lo64 &= lo64 - 1; else hi64 &= hi64 - 1;
      const int j = sm.mlog[tt];
      if (j >= 0) cnt -= 1;
      ev += 1;
      if ((ev & 31) == lane) sm.logi[ev] = cnt;
      cnt += 1;
      for (int i = lane; i <= ev; i += 32) {
        int li = sm.logi[i];
        if (j >= 0 && i < ev && li > j) sm.logi[i] = --li;
        sm.tab[ev * TW + i] = (unsigned char)li;
      }
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
    sm.evt[tt] = (unsigned char)e;
  }
  __syncthreads();  // table ready, every warp done with K
  // ---- V into the K buffer while Pt is formed
  stage_rows<D>(sm.kv, vg, row_stride, Lc);
  asm volatile("cp.async.commit_group;" ::: "memory");
  // ---- Pt = P o W (bf16), causal and lambda-weighted, over this warp's Q rows
  {
    const int ta = t_lo + g, tb = ta + 8;
    const float* lam_a = (a.lam && ta < Lc) ? a.lam + (rowbase + (long long)ta * a.H) * C : nullptr;
    const float* lam_b = (a.lam && tb < Lc) ? a.lam + (rowbase + (long long)tb * a.H) * C : nullptr;
    const unsigned char* tab_a = sm.tab + sm.evt[ta] * TW;
    const unsigned char* tab_b = sm.tab + sm.evt[tb] * TW;
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
            const int li = ((e < 2) ? tab_a : tab_b)[sm.evt[ss]];
            const float* lr = (e < 2) ? lam_a : lam_b;
            wt = lr ? lr[li] : 1.f;
          }
          w[e] = p[n][e] * wt;
        }
        *reinterpret_cast<__nv_bfloat162*>(sm.qp + ta * RP + s0) = __floats2bfloat162_rn(w[0], w[1]);
        *reinterpret_cast<__nv_bfloat162*>(sm.qp + tb * RP + s0) = __floats2bfloat162_rn(w[2], w[3]);
      }
    }
  }
  asm volatile("cp.async.wait_group 0;" ::: "memory");
  __syncthreads();
  // ---- O = Pt V over key steps s <= 16 warp + 15
  float o[NJ][4];
#pragma unroll
  for (int n = 0; n < NJ; ++n)
#pragma unroll
    for (int e = 0; e < 4; ++e) o[n][e] = 0.f;
  for (int ks = 0; ks <= warp; ++ks) {
    uint32_t af[4];
    ldsm4(af, sm.qp + (t_lo + (q & 1) * 8 + r8) * RP + 16 * ks + (q >> 1) * 8);
#pragma unroll
    for (int np = 0; np < NJ / 2; ++np) {
      uint32_t bf[4];
      ldsm4t(bf, sm.kv + (16 * ks + (q & 1) * 8 + r8) * RP + 16 * np + (q >> 1) * 8);
      mma16816(o[2 * np], af, bf[0], bf[1]);
      mma16816(o[2 * np + 1], af, bf[2], bf[3]);
    }
  }
  // ---- o_intra block of this interval (fp32, column-quad order)
  {
    const int ta = t_lo + g, tb = ta + 8;
    float* blk = a.ointra + ((long long)bh * a.ointra_T + (c0 - a.t_begin)) * D;
#pragma unroll
    for (int n = 0; n < NJ; ++n) {
      const int j = 8 * n + 2 * tg;
      float* col = blk + (long long)(j >> 2) * L * 4 + (j & 3);
      if (ta < Lc) *reinterpret_cast<float2*>(col + ta * 4) = make_float2(o[n][0], o[n][1]);
      if (tb < Lc) *reinterpret_cast<float2*>(col + tb * 4) = make_float2(o[n][2], o[n][3]);
    }
  }
}

cudaError_t preload_readout_intra() {
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, readout_intra_kernel<128>);
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
