// dla_scan.cu -- K1: the sequential part of the DLA forward pass.
//
// One CTA owns one (batch, head) stream and walks its tokens in chunks of
// kScanL = 64.  Per chunk it
//   1. stages k, v rows in shared memory (fp32),
//   2. forms the three scalars the score needs for every token -- a_t = |s_t|^2,
//      beta_t = <s_t, S_cur> and gam_t = |S_cur|^2 -- from the Gram entries
//      G[t][s] = (k_t.k_s)(v_t.v_s) and x_t = v_t^T S_open k_t, so no token
//      state s_t = v_t k_t^T is ever materialised (Sec. 3.1 score, Algorithm 1);
//   3. finds the boundaries b_t = 1[I_t >= tau] by "score all, take the first
//      firing token, restart the segment there" passes (one per boundary);
//   4. replays the chunk's decisions in order in one warp: per-token counts and
//      summed scores, Algorithm 2's adjacent-pair argmin and merge bookkeeping
//      when a boundary meets a full cache, appends (Sec. 3.2);
//   5. applies the state updates: closed segments are written to their
//      physical cache slot, merges add slot to slot, the open state stays in
//      shared memory (S = sum v k^T, row-major [d_v][d_k], fp32);
//   6. every `snap_chunks` chunks, writes a read-out snapshot: every cache
//      entry whose state changed is copied (fp32 or bf16) into this stream's
//      pool and the chunk's list of pool ids is recorded for K2.
// The live cache (fp32 states in physical slots + logical metadata) persists in
// global memory between rounds, so a round can start from any cache.
#include "dla_common.cuh"
#include "dla_kernels.h"

namespace dla {

namespace {

constexpr int NT = 256;  // threads per CTA

enum : int { OP_CLOSE = 0, OP_MERGE = 1 };

template <int D>
struct ScanSmem {
  static constexpr int L = kScanL;
  static constexpr int KP = D + 4;  // padded row (floats) of the k / v tiles
  float S[D * D];                   // open state [d_v][d_k]
  __nv_bfloat16 raw[2][2][L * D];   // bf16 k / v of the next chunk, in flight (bf16 inputs only)
  float K[L * KP];
  float V[L * KP];
  float G[L * (L + 1)];             // G[t][s] = (k_t.k_s)(v_t.v_s), s < t
  float x[L];                       // x_t = v_t^T S_open k_t
  float a[L];                       // a_t = |k_t|^2 |v_t|^2
  float red[16 * L];                // partial sums
  float wsum[4];
  float Itok[L];                    // score of every token in the chunk
  float gpart[NT / 32];             // per-warp partial sums of |S_open|^2
  double ibar[kMaxC];               // logical metadata of the cache (summed scores)
  float gam_open;
  int n[kMaxC];
  int slot[kMaxC];
  int pid[kMaxC];                   // pool id of the entry's latest snapshot
  int dirty[kMaxC];
  int bnd[L];                       // boundary flag per chunk token
  int mlog[L];                      // merge index per chunk token (-1)
  int ops[3 * L + 4][4];            // state operations of the chunk, in order
  int snap_src[kMaxC][2];           // snapshot jobs: (pool id, source)
  int first_fire[2];
  int nops, nsnapjobs;
  int m, cur, js, seg_pre, pool_next;
};

template <int D, typename Tin>
__device__ __forceinline__ void load_rows(float* dst, const Tin* src, int row_stride, int rows,
                                          int valid) {
  constexpr int KP = D + 4;
  constexpr int V4 = D / 4;  // float4 per row
  for (int e = threadIdx.x; e < rows * V4; e += NT) {
    int r = e / V4, c = (e % V4) * 4;
    float4 val = make_float4(0.f, 0.f, 0.f, 0.f);
    if (r < valid) val = load4(src + (long long)r * row_stride + c);
    store4(dst + r * KP + c, val);
  }
}

// Starts asynchronous 16-byte copies of `rows` k and v rows (bf16) into the
// staging buffers; rows >= valid are zero-filled.
template <int D>
__device__ __forceinline__ void prefetch_kv(__nv_bfloat16* dk, __nv_bfloat16* dv, const __nv_bfloat16* ks,
                                            const __nv_bfloat16* vs, int row_stride, int valid) {
  constexpr int V16 = D / 8;  // 16-byte pieces per row
  for (int e = threadIdx.x; e < kScanL * V16; e += NT) {
    const int r = e / V16, c = (e % V16) * 8;
    const int nbytes = (r < valid) ? 16 : 0;
    const __nv_bfloat16* sk = (r < valid) ? ks + (long long)r * row_stride + c : ks;
    const __nv_bfloat16* sv = (r < valid) ? vs + (long long)r * row_stride + c : vs;
    const uint32_t ak = static_cast<uint32_t>(__cvta_generic_to_shared(dk + r * D + c));
    const uint32_t av = static_cast<uint32_t>(__cvta_generic_to_shared(dv + r * D + c));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(ak), "l"(sk), "r"(nbytes) : "memory");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(av), "l"(sv), "r"(nbytes) : "memory");
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// Copies a D x D fp32 state into an fp32 pool entry.
template <int D>
__device__ __forceinline__ void copy_state(float* dst, const float* src) {
  for (int e = threadIdx.x * 4; e < D * D; e += NT * 4) store4(dst + e, load4(src + e));
}

}  // namespace

template <int D, typename Tin, typename Tpool>
__global__ void __launch_bounds__(NT, 1) scan_kernel(ScanArgs a) {
  constexpr int L = kScanL;
  constexpr int KP = D + 4;
  constexpr int TJ = D / 16;  // open-state tile per thread: TJ x TJ
  extern __shared__ __align__(16) unsigned char smem_raw[];
  ScanSmem<D>& sm = *reinterpret_cast<ScanSmem<D>*>(smem_raw);

  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int bh = blockIdx.x;
  const int b = bh / a.H, h = bh % a.H;
  const int C = a.C;
  const float Df = (float)(D * D);
  const long long tok0 = row_tok0(a.row_start, b, a.T);  // token row of the row's first token
  const Tin* kbase = reinterpret_cast<const Tin*>(a.k) + (tok0 * a.H + h) * D;
  const Tin* vbase = reinterpret_cast<const Tin*>(a.v) + (tok0 * a.H + h) * D;
  const int row_stride = a.H * D;
  float* states = a.states + (long long)bh * C * D * D;
  constexpr long long kEntry = (long long)D * D;  // elements per pool entry
  Tpool* pool = a.pool ? reinterpret_cast<Tpool*>(a.pool) + (long long)bh * a.pool_cap * kEntry : nullptr;
  uint8_t* bnd_out = a.boundary + (long long)bh * a.T;
  int32_t* mlog_out = a.merge_log + (long long)bh * a.T;

  // thread tile of the open state: rows j0.., cols k0..
  const int jb = tid / 16, kb = tid % 16;
  const int j0 = jb * TJ, k0 = kb * TJ;

  // ---------------------------------------------------------------- round start
  if (tid == 0) {
    int m0 = a.m[bh];
    if (m0 < 0 || m0 > C) {  // corrupted cache: flag it and start empty
      atomicExch(a.status, 6);
      m0 = 0;
    }
    sm.m = m0;
    sm.pool_next = 0;
  }
  __syncthreads();
  for (int i = tid; i < C; i += NT) {
    int sl = a.slot[(long long)bh * C + i];
    if (sl < 0 || sl >= C) {
      atomicExch(a.status, 6);
      sl = i;
    }
    sm.slot[i] = sl;
    sm.n[i] = a.n[(long long)bh * C + i];
    sm.ibar[i] = a.ibar[(long long)bh * C + i];
    sm.pid[i] = -1;
    sm.dirty[i] = 0;
  }
  __syncthreads();
  const int m_start = sm.m;
  if (m_start > 0) {
    const float* src = states + (long long)sm.slot[m_start - 1] * D * D;
    for (int e = tid * 4; e < D * D; e += NT * 4) store4(sm.S + e, load4(src + e));
  } else {
    for (int e = tid * 4; e < D * D; e += NT * 4) store4(sm.S + e, make_float4(0.f, 0.f, 0.f, 0.f));
  }
  if (pool) {
    const long long lst = (long long)bh * a.snap_stride + a.snap_base;  // list row of this round's first interval
    if (a.carry_in) {  // the pool continues: the previous round wrote this interval's list
      if (tid == 0) sm.pool_next = a.pstate[bh];
      for (int i = tid; i < m_start; i += NT) sm.pid[i] = a.pstate[a.B * a.H + (long long)bh * C + i];
    } else {  // snapshot 0: every live entry as it stands at the start of the round
      for (int i = 0; i < m_start; ++i) {
        if (i >= a.pool_cap) break;
        copy_state<D>(pool + (long long)i * kEntry, states + (long long)sm.slot[i] * D * D);
      }
      if (tid < m_start) sm.pid[tid] = tid;
      if (tid == 0) {
        sm.pool_next = m_start;
        a.snap_m0[lst] = m_start;
      }
      for (int i = tid; i < m_start; i += NT) a.snap_ids[lst * C + i] = i;
    }
  }
  __syncthreads();

  const int t_end = row_t_end(a.seq_lens, b, a.t_begin, a.t_end);  // this row's end of the round
  const int ntok = t_end - a.t_begin;
  const int nchunks = (ntok + L - 1) / L;
  if (sizeof(Tin) == 2 && ntok > 0) {  // a row that ended before this round has no chunk to load
    prefetch_kv<D>(sm.raw[0][0], sm.raw[0][1], reinterpret_cast<const __nv_bfloat16*>(kbase) +
                                                   (long long)a.t_begin * row_stride,
                   reinterpret_cast<const __nv_bfloat16*>(vbase) + (long long)a.t_begin * row_stride, row_stride,
                   min(L, ntok));
  }
  for (int c = 0; c < nchunks; ++c) {
    const int t0 = a.t_begin + c * L;
    const int Lc = min(L, t_end - t0);
    // ------------------------------------------------ 1. stage k, v
    if constexpr (sizeof(Tin) == 2) {
      // bf16: this chunk was prefetched during the previous one; start the next
      if (c + 1 < nchunks) {
        const int t1 = t0 + L;
        prefetch_kv<D>(sm.raw[(c + 1) & 1][0], sm.raw[(c + 1) & 1][1],
                       reinterpret_cast<const __nv_bfloat16*>(kbase) + (long long)t1 * row_stride,
                       reinterpret_cast<const __nv_bfloat16*>(vbase) + (long long)t1 * row_stride, row_stride,
                       min(L, t_end - t1));
        asm volatile("cp.async.wait_group 1;" ::: "memory");
      } else {
        asm volatile("cp.async.wait_group 0;" ::: "memory");
      }
      __syncthreads();
      load_rows<D, __nv_bfloat16>(sm.K, sm.raw[c & 1][0], D, L, L);
      load_rows<D, __nv_bfloat16>(sm.V, sm.raw[c & 1][1], D, L, L);
    } else {
      load_rows<D, Tin>(sm.K, kbase + (long long)t0 * row_stride, row_stride, L, Lc);
      load_rows<D, Tin>(sm.V, vbase + (long long)t0 * row_stride, row_stride, L, Lc);
    }
    if (tid < L) {
      sm.bnd[tid] = 0;
      sm.mlog[tid] = -1;
      sm.Itok[tid] = 0.f;
    }
    __syncthreads();
    const int m_chunk = sm.m;
    // ------------------------------------------------ 2. x_t and |S_open|^2
    if (m_chunk > 0) {
      // gam_open = |S_open|^2: per-thread partial sums, then a tree (fp32)
      float g = 0.f;
      for (int e = tid * 4; e < D * D; e += NT * 4) {
        float4 s4 = load4(sm.S + e);
        g += s4.x * s4.x + s4.y * s4.y + s4.z * s4.z + s4.w * s4.w;
      }
      g = warp_sum(g);
      if (lane == 0) sm.gpart[warp] = g;
      // x_t: thread = (tokens tb + 16 i, rows rb*TJ..); rows 16 apart keep the
      // float4 loads of 16 threads on 8 distinct bank groups
      const int tb = tid % 16, rb = tid / 16;
      float y[4][TJ];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int r = 0; r < TJ; ++r) y[i][r] = 0.f;
      for (int kk = 0; kk < D; kk += 4) {
        float4 kv[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) kv[i] = load4(sm.K + (tb + 16 * i) * KP + kk);
#pragma unroll
        for (int r = 0; r < TJ; ++r) {
          float4 s4 = load4(sm.S + (rb * TJ + r) * D + kk);
#pragma unroll
          for (int i = 0; i < 4; ++i)
            y[i][r] += s4.x * kv[i].x + s4.y * kv[i].y + s4.z * kv[i].z + s4.w * kv[i].w;
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        float part = 0.f;
#pragma unroll
        for (int r = 0; r < TJ; ++r) part += sm.V[(tb + 16 * i) * KP + rb * TJ + r] * y[i][r];
        sm.red[rb * L + tb + 16 * i] = part;
      }
      __syncthreads();
      if (tid < L) {
        float xs = 0.f;
#pragma unroll
        for (int r = 0; r < 16; ++r) xs += sm.red[r * L + tid];
        sm.x[tid] = xs;
      }
      if (tid == 0) {
        float gs = 0.f;
        for (int w = 0; w < NT / 32; ++w) gs += sm.gpart[w];
        sm.gam_open = gs;
      }
    } else {
      if (tid < L) sm.x[tid] = 0.f;
      if (tid == 0) sm.gam_open = 0.f;
    }
    // ------------------------------------------------ 3. Gram G[t][s] and a_t
    {
      const int tt = tid / 16, ss = tid % 16;  // tokens tt + 16 i, ss + 16 j
      float kk4[4][4], vv4[4][4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) kk4[i][j] = vv4[i][j] = 0.f;
      for (int e = 0; e < D; e += 4) {
        float4 kt[4], ks[4], vt[4], vs[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          kt[i] = load4(sm.K + (tt + 16 * i) * KP + e);
          ks[i] = load4(sm.K + (ss + 16 * i) * KP + e);
          vt[i] = load4(sm.V + (tt + 16 * i) * KP + e);
          vs[i] = load4(sm.V + (ss + 16 * i) * KP + e);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i)
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            kk4[i][j] += kt[i].x * ks[j].x + kt[i].y * ks[j].y + kt[i].z * ks[j].z + kt[i].w * ks[j].w;
            vv4[i][j] += vt[i].x * vs[j].x + vt[i].y * vs[j].y + vt[i].z * vs[j].z + vt[i].w * vs[j].w;
          }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          int t = tt + 16 * i, s = ss + 16 * j;
          float gv = kk4[i][j] * vv4[i][j];
          sm.G[t * (L + 1) + s] = (s < t) ? gv : 0.f;
          if (s == t) sm.a[t] = gv;
        }
    }
    if (tid == 0) {
      sm.cur = 0;
      sm.js = 0;
      sm.seg_pre = (m_chunk > 0) ? 1 : 0;
      if (m_chunk == 0) {  // the very first token of an empty cache opens state 0
        sm.bnd[0] = 1;
        sm.Itok[0] = 0.f;
        sm.cur = 1;
      }
    }
    __syncthreads();
    // ------------------------------------------------ 4. boundary passes
    while (true) {
      const int cur = sm.cur;
      if (cur >= Lc) break;
      const int js = sm.js;
      const int pre = sm.seg_pre;
      if (tid < L) {
        const int t = tid;
        float beta = 0.f, w = 0.f;
        if (t >= js && t < Lc) {
          float bs = pre ? sm.x[t] : 0.f;
          for (int s = js; s < t; ++s) bs += sm.G[t * (L + 1) + s];
          beta = bs;
          w = 2.f * beta + sm.a[t];
        }
        // exclusive scan of w over the 64 tokens (two warps)
        float inc = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          float up = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += up;
        }
        if (lane == 31) sm.wsum[warp] = inc;
        asm volatile("bar.sync 1, 64;");
        float excl = inc - w + (warp == 1 ? sm.wsum[0] : 0.f);
        bool fire = false;
        if (t >= cur && t < Lc) {
          const float gam = (pre ? sm.gam_open : 0.f) + excl;
          const float I = info_score(sm.a[t], beta, gam, Df, a.sp);
          sm.Itok[t] = I;
          fire = ((double)I >= a.sp.tau);
        }
        unsigned bal = __ballot_sync(0xffffffffu, fire);
        if (lane == 0) sm.first_fire[warp] = bal ? (warp * 32 + __ffs(bal) - 1) : L;
      }
      __syncthreads();
      if (tid == 0) {
        int ts = min(sm.first_fire[0], sm.first_fire[1]);
        if (ts >= Lc) {
          sm.cur = Lc;
        } else {
          sm.bnd[ts] = 1;
          sm.js = ts;
          sm.seg_pre = 0;
          sm.cur = ts + 1;
        }
      }
      __syncthreads();
    }
    // ------------------------------------------------ 5. replay decisions (warp 0)
    if (warp == 0) {
      int m = sm.m;
      int seg_u0 = 0;
      int nops = 0;
      int run0 = 0;  // first token of the current run of non-boundary tokens
      for (int t = 0; t <= Lc; ++t) {
        if (t < Lc && !sm.bnd[t]) continue;
        if (t > run0) {  // tokens [run0, t) joined the open state: count and summed score
          float part = 0.f;
          for (int u = run0 + lane; u < t; u += 32) part += sm.Itok[u];
          part = warp_sum(part);
          if (lane == 0) {
            sm.n[m - 1] += t - run0;
            sm.ibar[m - 1] += (double)part;
            sm.dirty[m - 1] = 1;
          }
          __syncwarp();
        }
        run0 = t + 1;
        if (t == Lc) break;
        if (m > 0 && lane == 0) {
          sm.ops[nops][0] = OP_CLOSE;
          sm.ops[nops][1] = sm.slot[m - 1];
          sm.ops[nops][2] = seg_u0;
          sm.ops[nops][3] = t;
        }
        if (m > 0) ++nops;
        int j = -1, phys_new = m;
        __syncwarp();
        if (m == C) {
          j = pair_argmin_warp(sm.n, sm.ibar, m);
          const int dst = sm.slot[j], src = sm.slot[j + 1];
          __syncwarp();
          if (lane == 0) {
            sm.ops[nops][0] = OP_MERGE;
            sm.ops[nops][1] = dst;
            sm.ops[nops][2] = src;
            sm.ops[nops][3] = 0;
            sm.n[j] += sm.n[j + 1];
            sm.ibar[j] += sm.ibar[j + 1];
            sm.dirty[j] = 1;
            sm.pid[j] = -1;
          }
          ++nops;
          __syncwarp();
          // shift logical entries j+2..m-1 down by one
          for (int base = j + 1; base < m - 1; base += 32) {
            int i = base + lane;
            int nv = 0, sv = 0, pv = 0, dv = 0;
            double iv = 0.0;
            if (i < m - 1) {
              nv = sm.n[i + 1]; sv = sm.slot[i + 1]; pv = sm.pid[i + 1]; dv = sm.dirty[i + 1];
              iv = sm.ibar[i + 1];
            }
            __syncwarp();
            if (i < m - 1) {
              sm.n[i] = nv; sm.slot[i] = sv; sm.pid[i] = pv; sm.dirty[i] = dv; sm.ibar[i] = iv;
            }
            __syncwarp();
          }
          phys_new = src;
          m -= 1;
        }
        if (lane == 0) {
          sm.slot[m] = phys_new;
          sm.n[m] = 1;
          sm.ibar[m] = (double)sm.Itok[t];
          sm.pid[m] = -1;
          sm.dirty[m] = 1;
          sm.mlog[t] = j;
        }
        __syncwarp();
        m += 1;
        seg_u0 = t;
      }
      if (lane == 0) {
        sm.m = m;
        sm.nops = nops;
        sm.js = seg_u0;  // in-chunk start of the open segment at chunk end
      }
    }
    __syncthreads();
    // ------------------------------------------------ 6. state updates
    {
      float acc[TJ][TJ];
#pragma unroll
      for (int r = 0; r < TJ; ++r) {
#pragma unroll
        for (int q4 = 0; q4 < TJ; q4 += 4) {
          float4 s4 = load4(sm.S + (j0 + r) * D + k0 + q4);
          acc[r][q4] = s4.x; acc[r][q4 + 1] = s4.y; acc[r][q4 + 2] = s4.z; acc[r][q4 + 3] = s4.w;
        }
      }
      const int nops = sm.nops;
      int u_done = 0;  // tokens [0, u_done) of the chunk are already in some state
      for (int op = 0; op < nops; ++op) {
        const int kind = sm.ops[op][0];
        if (kind == OP_CLOSE) {
          const int phys = sm.ops[op][1], u0 = sm.ops[op][2], u1 = sm.ops[op][3];
          for (int u = u0; u < u1; ++u) {
#pragma unroll
            for (int r = 0; r < TJ; ++r) {
              float vj = sm.V[u * KP + j0 + r];
#pragma unroll
              for (int q4 = 0; q4 < TJ; q4 += 4) {
                float4 k4 = load4(sm.K + u * KP + k0 + q4);
                acc[r][q4] += vj * k4.x; acc[r][q4 + 1] += vj * k4.y;
                acc[r][q4 + 2] += vj * k4.z; acc[r][q4 + 3] += vj * k4.w;
              }
            }
          }
          float* dst = states + (long long)phys * D * D;
#pragma unroll
          for (int r = 0; r < TJ; ++r)
#pragma unroll
            for (int q4 = 0; q4 < TJ; q4 += 4) {
              store4(dst + (j0 + r) * D + k0 + q4,
                     make_float4(acc[r][q4], acc[r][q4 + 1], acc[r][q4 + 2], acc[r][q4 + 3]));
              acc[r][q4] = acc[r][q4 + 1] = acc[r][q4 + 2] = acc[r][q4 + 3] = 0.f;
            }
          u_done = u1;
        } else {
          const float* src = states + (long long)sm.ops[op][2] * D * D;
          float* dst = states + (long long)sm.ops[op][1] * D * D;
          for (int e = tid * 4; e < D * D; e += NT * 4) {
            float4 x = load4(dst + e), y = load4(src + e);
            store4(dst + e, make_float4(x.x + y.x, x.y + y.y, x.z + y.z, x.w + y.w));
          }
        }
        __syncthreads();
      }
      (void)u_done;
      // tail of the chunk joins the open state
      const int u0 = sm.js;
      for (int u = u0; u < Lc; ++u) {
#pragma unroll
        for (int r = 0; r < TJ; ++r) {
          float vj = sm.V[u * KP + j0 + r];
#pragma unroll
          for (int q4 = 0; q4 < TJ; q4 += 4) {
            float4 k4 = load4(sm.K + u * KP + k0 + q4);
            acc[r][q4] += vj * k4.x; acc[r][q4 + 1] += vj * k4.y;
            acc[r][q4 + 2] += vj * k4.z; acc[r][q4 + 3] += vj * k4.w;
          }
        }
      }
#pragma unroll
      for (int r = 0; r < TJ; ++r)
#pragma unroll
        for (int q4 = 0; q4 < TJ; q4 += 4)
          store4(sm.S + (j0 + r) * D + k0 + q4,
                 make_float4(acc[r][q4], acc[r][q4 + 1], acc[r][q4 + 2], acc[r][q4 + 3]));
    }
    // per-token trace
    if (tid < Lc) {
      bnd_out[t0 + tid] = (uint8_t)sm.bnd[tid];
      mlog_out[t0 + tid] = sm.mlog[tid];
    }
    __syncthreads();
    // ------------------------------------------------ 7. read-out snapshot
    const bool interval_end = ((c + 1) % a.snap_chunks) == 0;
    const int snap_idx = (c + 1) / a.snap_chunks;
    const long long lrow = (long long)bh * a.snap_stride + a.snap_base + snap_idx;
    if (pool && interval_end && (snap_idx < a.nsnap || a.snap_at_end)) {
      if (tid == 0) {
        int nj = 0;
        const int m = sm.m;
        for (int i = 0; i < m; ++i) {
          if (sm.dirty[i] || sm.pid[i] < 0) {
            int p = sm.pool_next++;
            if (p >= a.pool_cap) {  // cannot happen with a correctly sized workspace
              atomicExch(a.status, 6);
              p = a.pool_cap - 1;
            }
            sm.pid[i] = p;
            sm.dirty[i] = 0;
            sm.snap_src[nj][0] = p;
            sm.snap_src[nj][1] = (i == m - 1) ? -1 : sm.slot[i];
            ++nj;
          }
        }
        sm.nsnapjobs = nj;
        a.snap_m0[lrow] = m;
      }
      __syncthreads();
      const int m = sm.m;
      for (int i = tid; i < m; i += NT)
        a.snap_ids[lrow * C + i] = sm.pid[i];
      for (int jj = 0; jj < sm.nsnapjobs; ++jj) {
        const int p = sm.snap_src[jj][0], srcslot = sm.snap_src[jj][1];
        const float* src = srcslot < 0 ? sm.S : states + (long long)srcslot * D * D;
        copy_state<D>(pool + (long long)p * kEntry, src);
      }
      __syncthreads();
    }
  }
  // ---------------------------------------------------------------- round end
  fill_padding_trace(bnd_out, mlog_out, t_end, a.t_end, tid, NT);
  {
    const int m = sm.m;
    if (m > 0) {
      float* dst = states + (long long)sm.slot[m - 1] * D * D;
      for (int e = tid * 4; e < D * D; e += NT * 4) store4(dst + e, load4(sm.S + e));
    }
    for (int i = tid; i < C; i += NT) {
      a.slot[(long long)bh * C + i] = sm.slot[i];
      a.n[(long long)bh * C + i] = (i < m) ? sm.n[i] : 0;
      a.ibar[(long long)bh * C + i] = (i < m) ? sm.ibar[i] : 0.0;
    }
    if (tid == 0) a.m[bh] = m;
    if (pool && a.pstate) {  // counters for a following round that continues this pool
      if (tid == 0) a.pstate[bh] = sm.pool_next;
      for (int i = tid; i < m; i += NT) a.pstate[a.B * a.H + (long long)bh * C + i] = sm.pid[i];
    }
  }
}

template <int D, typename Tin, typename Tpool>
static cudaError_t launch_scan_t(const ScanArgs& a, cudaStream_t s) {
  const size_t smem = sizeof(ScanSmem<D>);
  auto kern = scan_kernel<D, Tin, Tpool>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<a.B * a.H, NT, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_scan(const ScanArgs& a, int d, cudaStream_t s) {
  return d == 128 ? launch_scan_t<128, float, float>(a, s) : launch_scan_t<64, float, float>(a, s);
}

size_t scan_smem_bytes(int d) { return d == 128 ? sizeof(ScanSmem<128>) : sizeof(ScanSmem<64>); }

}  // namespace dla
