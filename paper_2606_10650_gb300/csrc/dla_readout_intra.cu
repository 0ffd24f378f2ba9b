// dla_readout_intra.cu -- K2a on the 5th-generation tensor cores (tcgen05 +
// TMEM + TMA): the intra-interval part of the read-out
// (Eq. capacity_bounded_output restricted to the tokens of the interval):
//   o_intra[t] = sum_{s <= t in interval} lambda_{t, L_t(e(s))} (q_t . k_s) v_s
// for one 128-token interval of one stream per CTA (bf16 inputs, d = 128),
// written in fp32 to a scratch buffer that the snapshot part of the read-out
// (K2b) starts from.  Two MMAs of M = N = K = 128 (bf16 in, fp32 in TMEM):
//   P  = Q K^T                                        TMEM columns [0, 128)
//   Pt = P o W  (bf16, W_ts = lambda_{t, L_t(e(s))} for s <= t, else 0)
//   O  = Pt V   (V^T as the K-major B operand)        TMEM columns [128, 256)
// The entry holding token s is the one opened by the last boundary event at or
// before s (event 0: the snapshot's open state), so W only needs the slot of
// "the entry opened at event i" after event e: one table row per event.
// Q and K arrive by TMA; once P is done their tiles are overwritten with Pt and
// V^T by the epilogue warps.  83 KB of shared memory and 256 TMEM columns: two
// CTAs per SM.
// Roles: warp 0 issues the TMA loads, warp 1 the MMAs (one thread), warps 2-5
// are the epilogue (one token row per thread: warp w reads TMEM lane quadrant
// w % 4).
//
// Scratch layout, per interval a 128 x 128 fp32 block in column-quad order:
// element (t, j) at ((j / 4) * 128 + t) * 4 + j % 4, so that a warp's 32 rows
// of one column quad are 512 contiguous bytes.
#include "dla_common.cuh"
#include "dla_sm100.cuh"
#include "dla_tmap.h"

namespace dla {

namespace {

using namespace sm100;

constexpr int L = kReadoutTcInterval;  // 128 tokens per CTA
constexpr int D = 128;
constexpr int NT = 192;                // 6 warps
constexpr int NEPI = 4;                // epilogue warps
constexpr int TW = L + 1;              // table row: events 0 .. L
constexpr uint32_t kTile = L * 128;    // one K-major 128B-swizzled tile: 128 rows x 64 bf16
constexpr uint32_t kTmemCols = 256;    // P [0, 128), O [128, 256)

struct IntraSmem {
  uint8_t A[2][kTile];         // Q (two k-halves), then Pt (two s-halves)   32 KB
  uint8_t Bm[2][kTile];        // K (two k-halves), then V^T (two s-halves)  32 KB
  unsigned char tab[TW * TW];  // tab[e][i]: slot of the entry opened at event i, after event e
  unsigned char evt[L];        // events at or before token t
  int logi[TW];
  int mlog[L];
  uint8_t bnd[L];
  uint64_t bar_qk, bar_p, bar_pt, bar_o, bar_done;
  uint32_t tmem_base;
  int abort_flag;
};

}  // namespace

__global__ void __launch_bounds__(NT, 2)
    readout_intra_kernel(ReadoutArgs a, const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                         int32_t* status) {
  extern __shared__ uint8_t smem_raw[];
  IntraSmem& sm = *reinterpret_cast<IntraSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int s = blockIdx.x, bh = blockIdx.y;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const int c0 = a.t_begin + s * L;
  const int Lc = min(L, a.t_end - c0);
  volatile int* abort = &sm.abort_flag;
  // with a scan running concurrently: the interval must be complete; its list
  // and trace are then read past L1 (__ldcg)
  wait_progress(a.progress, a.progress_ctas, bh, a.snap_base + s + 1, status);

  if (tid == 0) {
    mbar_init(&sm.bar_qk, 1);
    mbar_init(&sm.bar_p, 1);
    mbar_init(&sm.bar_pt, NEPI);
    mbar_init(&sm.bar_o, 1);
    mbar_init(&sm.bar_done, 1);
    sm.abort_flag = 0;
    fence_mbar_init();
  }
  if (warp == 1) tmem_alloc(&sm.tmem_base, kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const int m0 = __ldcg(a.snap_m0 + (long long)bh * a.snap_stride + a.snap_base + s);
  const long long rowbase = ((long long)b * a.T + c0) * a.H + h;  // row index of token c0

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      mbar_expect_tx(&sm.bar_qk, 4 * kTile);
      tma_load_4d(sm.A[0], &tmQ, &sm.bar_qk, 0, h, c0, b);
      tma_load_4d(sm.A[1], &tmQ, &sm.bar_qk, 64, h, c0, b);
      tma_load_4d(sm.Bm[0], &tmK, &sm.bar_qk, 0, h, c0, b);
      tma_load_4d(sm.Bm[1], &tmK, &sm.bar_qk, 64, h, c0, b);
      if (!mbar_wait(&sm.bar_qk, 0, abort, status)) mbar_wait_drain(&sm.bar_qk, 0);  // copies land before exit
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(L, L);
      bool ok = mbar_wait(&sm.bar_qk, 0, abort, status);
      if (ok) {  // P = Q K^T
        tc_fence_after();
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (uint32_t)(kk & 3) * 32;
          mma_bf16(tmem, desc_kmajor_sw128(smem_u32(sm.A[kk >> 2]) + off),
                   desc_kmajor_sw128(smem_u32(sm.Bm[kk >> 2]) + off), idesc, kk > 0);
        }
        mma_commit(&sm.bar_p);
        ok = mbar_wait(&sm.bar_pt, 0, abort, status);
      }
      if (ok) {  // O = Pt V: A = Pt [t][s], B = V^T [j][s]
        tc_fence_after();
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t off = (uint32_t)(kk & 3) * 32;
          mma_bf16(tmem + 128, desc_kmajor_sw128(smem_u32(sm.A[kk >> 2]) + off),
                   desc_kmajor_sw128(smem_u32(sm.Bm[kk >> 2]) + off), idesc, kk > 0);
        }
        mma_commit(&sm.bar_o);
      }
      mma_commit(&sm.bar_done);  // every MMA issued above has completed once this fires
      mbar_wait_drain(&sm.bar_done, 0);
    }
  } else {
    // ------------------------------------------------------------ epilogue warps
    const int etid = tid - 64;          // 0..127: staging index
    const int quad = warp & 3;          // TMEM lane quadrant of this warp
    const int t = quad * 32 + lane;     // token row of this thread
    const uint32_t lane_addr = tmem + ((uint32_t)(quad * 32) << 16);
    {  // the interval's trace
      const bool in = etid < Lc;
      sm.bnd[etid] = in ? __ldcg(a.boundary + (long long)bh * a.T + c0 + etid) : (uint8_t)0;
      sm.mlog[etid] = in ? __ldcg(a.merge_log + (long long)bh * a.T + c0 + etid) : -1;
    }
    // row etid of V, loaded now and written transposed once P no longer needs K's tile
    uint4 vraw[D / 8];
    {
      const __nv_bfloat16* vrow = reinterpret_cast<const __nv_bfloat16*>(a.v) + (rowbase + (long long)etid * a.H) * D;
#pragma unroll
      for (int i = 0; i < D / 8; ++i)
        vraw[i] = (etid < Lc) ? *reinterpret_cast<const uint4*>(vrow + 8 * i) : make_uint4(0, 0, 0, 0);
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    if (warp == 2) {
      // slot table: lane x owns the entries opened at events x, x + 32, ...;
      // a merge at index j moves every slot above j down by one
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
    {  // events at or before each token (one token per thread: etid)
      int e = 0;
#pragma unroll
      for (int w4 = 0; w4 < 4; ++w4) {
        const unsigned m = __ballot_sync(0xffffffffu, sm.bnd[32 * w4 + lane] != 0);
        if (32 * w4 + 31 <= etid) e += __popc(m);
        else if (32 * w4 <= etid) e += __popc(m & (0xffffffffu >> (31 - (etid - 32 * w4))));
      }
      sm.evt[etid] = (unsigned char)e;
    }
    asm volatile("bar.sync 1, 128;" ::: "memory");
    const float* lam_t = (a.lam && t < Lc) ? a.lam + (rowbase + (long long)t * a.H) * C : nullptr;
    const unsigned char* tab_t = sm.tab + sm.evt[t] * TW;
    // tcgen05.ld below is warp-wide: the warp takes one decision
    bool ok = __all_sync(0xffffffffu, mbar_wait(&sm.bar_p, 0, abort, status));
    if (ok) {
      tc_fence_after();
      // V^T into K's tile: element (j, s = etid) of the K-major operand [j][s]
#pragma unroll
      for (int i = 0; i < D / 8; ++i) {
        const __nv_bfloat16* vv = reinterpret_cast<const __nv_bfloat16*>(&vraw[i]);
        uint8_t* tile = sm.Bm[etid >> 6];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          *reinterpret_cast<__nv_bfloat16*>(tile + sw128_offset(8 * i + u, etid & 63)) = vv[u];
      }
      // Pt into Q's tile: row t, columns s (weights of the causal, lambda-weighted term).
      // The weight of column s depends on s only through evt[s], which changes at
      // the interval's boundaries: it is looked up again only when evt[s] changes.
      int last_e = -1;
      float last_w = 0.f;
#pragma unroll
      for (int c = 0; c < L; c += 32) {
        float p[32];
        tmem_ld32(lane_addr + c, p);
        uint8_t* tile = sm.A[c >> 6];
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          uint32_t packed[4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            float w2[2];
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int ss = c + 8 * c8 + 2 * i + u;
              float wt = 0.f;
              if (ss <= t && t < Lc) {
                const int e = sm.evt[ss];
                if (e != last_e) {
                  last_e = e;
                  last_w = lam_t ? __ldg(lam_t + tab_t[e]) : 1.f;
                }
                wt = last_w;
              }
              w2[u] = p[8 * c8 + 2 * i + u] * wt;
            }
            const __nv_bfloat162 pr = __floats2bfloat162_rn(w2[0], w2[1]);
            packed[i] = *reinterpret_cast<const uint32_t*>(&pr);
          }
          const int chunk = ((c & 63) >> 3) + c8;  // 16-byte chunk of the row
          *reinterpret_cast<uint4*>(tile + t * 128 + (((chunk ^ (t & 7)) & 7) << 4)) =
              make_uint4(packed[0], packed[1], packed[2], packed[3]);
        }
      }
    }
    fence_proxy_async();  // the generic-proxy writes above feed the tensor core
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.bar_pt);
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(&sm.bar_o, 0, abort, status));
    if (ok) {  // o_intra row t (fp32, column-quad order)
      tc_fence_after();
      float* blk = a.ointra + ((long long)bh * a.ointra_T + (c0 - a.t_begin)) * D;
#pragma unroll
      for (int c = 0; c < D; c += 32) {
        float o[32];
        tmem_ld32(lane_addr + 128 + c, o);  // tcgen05.ld is warp-wide: every lane loads, rows past Lc store nothing
        if (t < Lc)
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4)
            *reinterpret_cast<float4*>(blk + ((long long)((c >> 2) + j4) * L + t) * 4) =
                make_float4(o[4 * j4], o[4 * j4 + 1], o[4 * j4 + 2], o[4 * j4 + 3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
}

cudaError_t preload_readout_intra() {
  cudaFuncAttributes fa;
  return cudaFuncGetAttributes(&fa, readout_intra_kernel);
}

cudaError_t launch_readout_intra(const ReadoutArgs& a, cudaStream_t st) {
  CUtensorMap mq, mk;
  if (!tmap_tokens(&mq, a.q, a.B, a.T, a.H) || !tmap_tokens(&mk, a.k, a.B, a.T, a.H)) return cudaErrorInvalidValue;
  const size_t smem = sizeof(IntraSmem) + 1024;
  cudaError_t e = cudaFuncSetAttribute(readout_intra_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  dim3 grid(a.nsnap, a.B * a.H);
  readout_intra_kernel<<<grid, NT, smem, st>>>(a, mq, mk, a.status);
  return cudaGetLastError();
}

}  // namespace dla
