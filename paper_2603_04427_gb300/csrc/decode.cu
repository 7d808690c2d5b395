// Decode attention over a thin-key / full-value cache: a persistent, evenly
// partitioned stream over the whole cache, with the per-group products on the
// tensor cores.
//
// Paper: Section 2.1, Eq. 4 with a single query row per head; decode is the
// bandwidth-bound case of Section 4.2 (every step streams the whole cache).
//
// Work units are 64-token chunks of one (sequence b, kv head g) pair in the
// order b, g, chunk; sequence b has n_b = ceil(L_b / 64) chunks per kv head, so
// the units form a flat range [0, T).  CTA c of the N persistent CTAs owns
// units [c*T/N, (c+1)*T/N): every CTA streams the same number of chunks to
// within one, whatever the length mix.  The split is computed on the device
// from seq_lens (prefix sums of n_b in shared memory).
//
//   warp 4 (producer): walks the CTA's units and loads each chunk into an
//     NSTAGE-deep shared-memory ring: the 64 K rows and V rows as TMA tiles
//     with 32/64/128-byte swizzle (conflict-free ldmatrix), the key scales
//     and the pair's G query rows with 1-D bulk copies.  For paged caches its
//     32 lanes look up the page ids of the next 32 units in parallel.
//   warps 0-3 (consumers): warp w owns tokens 16w..16w+15 of every chunk.  With
//     the G query heads of the kv head as the n=8 dimension of mma.m16n8k16:
//       S^T (16 tokens x 8 heads) = K (16 x r) Q^T          (k = r)
//       O^T (d_v x 8 heads)      += V^T (d_v x 16) P^T       (k = 16 tokens)
//     bf16 operands, fp32 accumulation.  P moves from the S^T accumulator
//     layout to the B-operand layout with movmatrix.  int8 and int4 keys
//     (Section 6's composition with key quantisation; int4 two codes per byte)
//     are widened to bf16 in registers (exactly), with the query's r index
//     permuted to match the code order ldmatrix delivers; the per-token scale
//     multiplies the fp32 score.  Scores are kept in log2 units; online
//     softmax per head.
//   warp 5 (merger): a segment is the run of one pair's chunks inside the
//     CTA's range.  At a segment end each consumer warp deposits (m, l, O) in a
//     double-buffered shared-memory record and carries on streaming; the merger
//     warp combines the four records.  A pair inside the range is written out
//     directly; a pair that straddles CTA boundaries (at most two per CTA) is
//     written as a partial to the workspace, and the last CTA to arrive on the
//     pair's counter (acquire/release atomic) merges the partials, loading
//     them in parallel batches.  No CTA ever waits for another.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "common.cuh"
#include "kernels.h"
#include "kv_row.cuh"
#include "widen.cuh"

namespace tk {
namespace {

constexpr int kChunk = 64;                  // tokens per unit / pipeline stage
constexpr int kCW = 4;                      // consumer warps (16 tokens each)
constexpr int kThreads = (kCW + 2) * 32;    // + one producer warp + one merger warp
constexpr int kMaxBatch = 1024;             // prefix arrays live in shared memory
constexpr int kCtaSmemTarget = 110 * 1024;  // aim for two CTAs per SM

// KF: key format, 0 bf16, 1 int8, 2 int4 (two codes per byte, R >= 32).
template <int R, int DV, int G, int KF>
struct Cfg {
  static constexpr bool KQ = KF != 0;                  // quantised keys with fp32 scales
  static constexpr int RB = KF == 0 ? 2 * R : (KF == 1 ? R : R / 2);  // bytes per key row
  static constexpr int KSW = RB >= 128 ? 128 : RB;     // K tile swizzle span (16 = none)
  static constexpr int KBOX_N = RB / KSW;              // K boxes per chunk
  static constexpr int KBOX = kChunk * KSW;            // bytes per K box
  static constexpr int VBOX_N = DV / 64;               // V boxes (64 bf16 = 128 bytes wide)
  static constexpr int VBOX = kChunk * 128;
  static constexpr int KB = KBOX_N * KBOX, VB = VBOX_N * VBOX;
  static constexpr int SB = KQ ? kChunk * 4 : 0;
  static constexpr int QB = (G * R * 2 + 15) / 16 * 16;
  static constexpr int OFF_V = (KB + 1023) / 1024 * 1024;
  static constexpr int OFF_S = OFF_V + VB;
  static constexpr int OFF_QS = OFF_S + SB;
  static constexpr int STAGE = (OFF_QS + QB + 1023) / 1024 * 1024;
  static constexpr int KSTEPS = R / 16;
  static constexpr int REC = (G * DV + 2 * G + 3) / 4 * 4;  // floats per merge record
  static constexpr int TAIL = 2 * kCW * REC * 4 + 512 + 1024;
  static constexpr int PRE = (kMaxBatch + 1) * 8 + kMaxBatch * 4;
  static constexpr int NSTAGE_2 = (kCtaSmemTarget - TAIL - PRE) / STAGE;
  static constexpr int NSTAGE_1 = (220 * 1024 - TAIL - PRE) / STAGE;
  // two CTAs per SM when at least three stages fit in half the SM
  static constexpr int CTAS_PER_SM = NSTAGE_2 >= 3 ? 2 : 1;
  static constexpr int NSTAGE_RAW = CTAS_PER_SM == 2 ? NSTAGE_2 : NSTAGE_1;
  static constexpr int NSTAGE = NSTAGE_RAW > 8 ? 8 : NSTAGE_RAW;
  static_assert(NSTAGE >= 2, "shared memory budget too small for two stages");
  static constexpr int RING = NSTAGE * STAGE;
  static constexpr int OFF_MERGE = RING;                         // [2][kCW][REC] f32
  static constexpr int OFF_BAR = OFF_MERGE + 2 * kCW * REC * 4;  // mbarriers
  static constexpr int OFF_PRE = OFF_BAR + 512;                  // [B+1] i64, [B] i32
  static_assert(OFF_PRE + PRE + 1024 <= 227 * 1024, "shared memory");
};

// ---------------------------------------------------------------- small PTX helpers
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                        uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x2(uint32_t addr, uint32_t& a, uint32_t& b) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];"
               : "=r"(a), "=r"(b)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& a, uint32_t& b, uint32_t& c,
                                          uint32_t& d) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(a), "=r"(b), "=r"(c), "=r"(d)
               : "r"(addr));
}
__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
  uint32_t y;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
__device__ __forceinline__ void mma16816(float* d, uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// Byte offset of (row, byte) inside a TMA box whose rows are SPAN bytes wide
// and swizzled over SPAN bytes (16 = no swizzle).  Box bases are 1 KB aligned.
template <int SPAN>
__device__ __forceinline__ uint32_t swz(uint32_t row, uint32_t byte) {
  uint32_t a = row * SPAN + byte;
  if constexpr (SPAN == 128) a ^= ((a >> 7) & 7u) << 4;
  if constexpr (SPAN == 64) a ^= ((a >> 7) & 3u) << 4;
  if constexpr (SPAN == 32) a ^= ((a >> 7) & 1u) << 4;
  return a;
}

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_addr(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(policy)
      : "memory");
}

// Position of a unit in the (b, g, chunk) order, walked forward one unit at a time.
struct Walker {
  int b, g, chunk, nb, Lb;
  long long cp;  // first unit of the current pair
  __device__ void seek(long long u, const long long* pre, const int* lens, int B, int Hkv) {
    int lo = 0, hi = B;  // last b with pre[b] <= u
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (pre[mid] <= u) lo = mid; else hi = mid;
    }
    b = lo;
    while (pre[b + 1] <= u) ++b;  // empty sequences have pre[b] == pre[b+1]
    nb = static_cast<int>((pre[b + 1] - pre[b]) / Hkv);
    const long long off = u - pre[b];
    g = static_cast<int>(off / nb);
    chunk = static_cast<int>(off % nb);
    Lb = lens[b];
    cp = pre[b] + static_cast<long long>(g) * nb;
  }
  // Advance to the next unit; only called when one exists.
  __device__ void next(const long long* pre, const int* lens, int Hkv) {
    if (++chunk < nb) return;
    chunk = 0;
    cp += nb;
    if (++g < Hkv) return;
    g = 0;
    do { ++b; } while (pre[b + 1] == pre[b]);
    nb = static_cast<int>((pre[b + 1] - pre[b]) / Hkv);
    Lb = lens[b];
    cp = pre[b];
  }
};

// CTAs that share T units: about four units each, so that short contexts are
// not split across CTAs (every split adds a merge); but one unit each when
// four-unit shares would leave three quarters of the grid idle, so that small
// batches spread over the GPU.  Measured: a GPT-2-sized step (60 units) 277 ->
// 215 us per layer of 32 steps with one unit per CTA; one unit per CTA slowed
// B = 16 at context 256 (512 units) from 7.8 to 11.8 us; shares in between
// (3.4 units) were slower than both at B = 4, context 512 (11.1 us against
// 9.1 and 8.8 us), cutting most pairs at two places.
__device__ __forceinline__ int split_ctas(long long T, int grid) {
  const long long four = (T + 3) / 4;
  const long long want = four < grid / 4 ? T : four;
  return static_cast<int>(min(static_cast<long long>(grid), max(want, 1LL)));
}

// CTA owning unit u when CTA c owns [floor(c T / N), floor((c+1) T / N)).
__device__ __forceinline__ int cta_of(long long u, long long T, int N) {
  return static_cast<int>(((u + 1) * N - 1) / T);
}

// Vectorised copies of a lane's E consecutive floats.
template <int E>
__device__ __forceinline__ void ld_cg_vec(const float* src, float* dst) {
  if constexpr (E % 4 == 0) {
#pragma unroll
    for (int i = 0; i < E; i += 4) {
      const float4 x = __ldcg(reinterpret_cast<const float4*>(src + i));
      dst[i] = x.x; dst[i + 1] = x.y; dst[i + 2] = x.z; dst[i + 3] = x.w;
    }
  } else {
#pragma unroll
    for (int i = 0; i < E; i += 2) {
      const float2 x = __ldcg(reinterpret_cast<const float2*>(src + i));
      dst[i] = x.x; dst[i + 1] = x.y;
    }
  }
}

__device__ __forceinline__ void write_out(const DecodeParams& p, long long o, float v) {
  if (p.out_f32) reinterpret_cast<float*>(p.out)[o] = v;
  else reinterpret_cast<__nv_bfloat16*>(p.out)[o] = __float2bfloat16_rn(v);
}

// The merger warp: for every segment of the CTA's range, combine the consumer
// warps' records; write the output of pairs inside the range, or the partial of
// pairs that straddle CTAs and, on the last arrival, merge all their partials.
// Lane l owns E = G*DV/32 consecutive elements of the [G][DV] output, all in
// head (l*E)/DV.
template <int R, int DV, int G, int KF>
__device__ void merge_segments(const DecodeParams& p, const float* merge, uint64_t* deposit,
                               uint64_t* mfree, const long long* pre, const int* lens,
                               long long T, int N, int c, long long u_begin, long long u_end,
                               int lane) {
  using C = Cfg<R, DV, G, KF>;
  constexpr bool KI8 = KF != 0;  // quantised keys (int8 or int4)
  constexpr int E = G * DV / 32;
  constexpr int CB = E >= 32 ? 2 : (E >= 16 ? 4 : 8);  // segments loaded per batch
  const int e0 = lane * E, hh = e0 / DV;
  if (u_begin == u_end) return;
  Walker wk;
  wk.seek(u_begin, pre, lens, p.B, p.Hkv);
  long long u = u_begin;
  for (int seg = 0; u < u_end; ++seg) {
    const int buf = seg & 1;
    if (!mbar_wait(&deposit[buf], (seg >> 1) & 1, p.err)) return;
    const float* recs = merge + buf * kCW * C::REC;
    float f[kCW], M = -INFINITY, L = 0.f;
#pragma unroll
    for (int w = 0; w < kCW; ++w) M = fmaxf(M, recs[w * C::REC + G * DV + hh]);
#pragma unroll
    for (int w = 0; w < kCW; ++w) {
      f[w] = fast_exp2(recs[w * C::REC + G * DV + hh] - M);  // 0 for a warp without tokens
      L += recs[w * C::REC + G * DV + G + hh] * f[w];
    }
    float acc[E];
#pragma unroll
    for (int i = 0; i < E; ++i) {
      float a = 0.f;
#pragma unroll
      for (int w = 0; w < kCW; ++w) a += recs[w * C::REC + e0 + i] * f[w];
      acc[i] = a;
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&mfree[buf]);  // records read: the consumers may reuse them

    const int pair = wk.b * p.Hkv + wk.g;
    const long long cp = wk.cp;
    const long long seg_end = min(u_end, cp + wk.nb);
    const int c_first = cta_of(cp, T, N), c_last = cta_of(cp + wk.nb - 1, T, N);
    const long long obase = (static_cast<long long>(wk.b) * p.Hq + wk.g * G) * DV;
    if (c_first == c_last) {
      const float inv = 1.f / L;
#pragma unroll
      for (int i = 0; i < E; ++i) write_out(p, obase + e0 + i, acc[i] * inv);
    } else {
      float* mine = p.part + (static_cast<long long>(c) * 2 + (cp <= u_begin ? 0 : 1)) * C::REC;
#pragma unroll
      for (int i = 0; i < E; ++i) mine[e0 + i] = acc[i];
      if (e0 % DV == 0) {
        mine[G * DV + hh] = M;
        mine[G * DV + G + hh] = L;
      }
      __syncwarp();
      int last = 0;
      if (lane == 0) {
        int old;
        asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;"
                     : "=r"(old)
                     : "l"(p.counters + pair)
                     : "memory");
        last = old == c_last - c_first;
      }
      last = __shfl_sync(0xffffffffu, last, 0);
      __syncwarp();
      if (last) {
        // merge the partials of CTAs c_first..c_last: each batch of CB partials
        // is one round of loads (m, l and o together), folded in with an online
        // rescale; every partial holds at least one token, so its m is finite
        auto slot = [&](int cc) {
          const long long sc = T * cc / N;
          return p.part + (static_cast<long long>(cc) * 2 + (cp <= sc ? 0 : 1)) * C::REC;
        };
        float Mt = -INFINITY, Lt = 0.f;
        float out[E];
#pragma unroll
        for (int i = 0; i < E; ++i) out[i] = 0.f;
        for (int b0 = c_first; b0 <= c_last; b0 += CB) {
          float oo[CB][E], mm[CB], ll[CB];
#pragma unroll
          for (int k = 0; k < CB; ++k) {
            mm[k] = -INFINITY;
            ll[k] = 0.f;
            if (b0 + k <= c_last) {
              const float* sl = slot(b0 + k);
              mm[k] = __ldcg(sl + G * DV + hh);
              ll[k] = __ldcg(sl + G * DV + G + hh);
              ld_cg_vec<E>(sl + e0, oo[k]);
            } else {
#pragma unroll
              for (int i = 0; i < E; ++i) oo[k][i] = 0.f;
            }
          }
          float Mn = Mt;
#pragma unroll
          for (int k = 0; k < CB; ++k) Mn = fmaxf(Mn, mm[k]);
          const float a = Mt == -INFINITY ? 0.f : fast_exp2(Mt - Mn);
          Lt *= a;
#pragma unroll
          for (int i = 0; i < E; ++i) out[i] *= a;
#pragma unroll
          for (int k = 0; k < CB; ++k) {
            const float wk2 = (b0 + k <= c_last) ? fast_exp2(mm[k] - Mn) : 0.f;
            Lt += ll[k] * wk2;
#pragma unroll
            for (int i = 0; i < E; ++i) out[i] += oo[k][i] * wk2;
          }
          Mt = Mn;
        }
        const float inv = 1.f / Lt;
#pragma unroll
        for (int i = 0; i < E; ++i) write_out(p, obase + e0 + i, out[i] * inv);
        if (lane == 0) p.counters[pair] = 0;  // ready for the next launch
      }
    }
    u = seg_end;
    if (u < u_end) wk.seek(u, pre, lens, p.B, p.Hkv);
  }
}

struct DecodeMaps {
  CUtensorMap k, v;
};
// L2 prefetch of a CTA's first chunks, issued by its producer warp before the
// dependent-launch wait: while the previous kernel on the stream finishes,
// the CTA's first TMA reads after the wait then come from L2.  The context
// lengths and page table read here may be stale (the previous kernel may
// still write them); they are clamped so that every prefetched address lies
// inside the cache, and a wrong guess only wastes the prefetch (L2 is
// coherent, so nothing stale is ever read).  Batches of up to 32 sequences.
// Twice the ring depth measured best on the Mistral GQA shape (28.5 us
// against 29.2 us for one ring, 29.2 us for four).
template <int RB, int DV>
__device__ void prefetch_first_chunks(const DecodeParams& p, int lane, int limit, int nunits) {
  const int B = p.B, Hkv = p.Hkv;
  int L = 0;
  if (lane < B) {
    L = p.seq_lens[lane];
    if (p.fuse_append && L >= 0) ++L;
    L = min(max(L, 0), limit);
  }
  const long long x = static_cast<long long>((L + kChunk - 1) / kChunk) * Hkv;  // units of sequence `lane`
  long long inc = x;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const long long y = __shfl_up_sync(0xffffffffu, inc, off);
    if (lane >= off) inc += y;
  }
  const long long T = __shfl_sync(0xffffffffu, inc, 31);
  const long long pre = inc - x;
  const int N = split_ctas(T, gridDim.x);
  const int c = blockIdx.x;
  if (T == 0 || c >= N) return;  // warp-uniform
  const long long u_begin = T * c / N, u_end = T * (c + 1) / N;
  const long long u = u_begin + lane;
  int b = 0;
  for (int bb = 0; bb < B; ++bb) {
    const long long pb = __shfl_sync(0xffffffffu, pre, bb), xb = __shfl_sync(0xffffffffu, x, bb);
    if (pb <= u && u < pb + xb) b = bb;
  }
  const int Lb = __shfl_sync(0xffffffffu, L, b);
  const long long pb = __shfl_sync(0xffffffffu, pre, b);
  const int nb = (Lb + kChunk - 1) / kChunk;
  if (lane >= nunits || u >= u_end || nb == 0) return;
  const long long off = u - pb;
  const int g = static_cast<int>(off / nb), t0 = static_cast<int>(off % nb) * kChunk;
  long long row;
  int rows;
  if (p.page_size == 0) {
    row = (static_cast<long long>(b) * Hkv + g) * p.capacity + t0;
    rows = min(kChunk, p.capacity - t0);
  } else {
    const int pidx = t0 >> p.page_shift;
    if (pidx >= p.max_pages) return;
    const int page = p.page_table[static_cast<long long>(b) * p.max_pages + pidx];
    if (page < 0 || page >= p.num_pages) return;
    const int in_page = t0 & (p.page_size - 1);
    row = (static_cast<long long>(page) * Hkv + g) * p.page_size + in_page;
    rows = min(kChunk, p.page_size - in_page);
  }
  if (rows <= 0) return;
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const unsigned char*>(p.k) + row * RB),
               "r"(static_cast<uint32_t>(rows * RB))
               : "memory");
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(static_cast<const unsigned char*>(p.v) + row * DV * 2),
               "r"(static_cast<uint32_t>(rows * DV * 2))
               : "memory");
}


// The grid is persistent (CTAS_PER_SM CTAs on every SM at once): the bound
// keeps the register count low enough for that many CTAs to be resident.
template <int R, int DV, int G, int KF>
__global__ void __launch_bounds__(kThreads, Cfg<R, DV, G, KF>::CTAS_PER_SM)
decode_kernel(const __grid_constant__ DecodeMaps maps, const DecodeParams p) {
  using C = Cfg<R, DV, G, KF>;
  constexpr bool KI8 = KF != 0;  // quantised keys (int8 or int4)
  extern __shared__ __align__(1024) unsigned char smem_raw[];
  unsigned char* smem = reinterpret_cast<unsigned char*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  float* merge = reinterpret_cast<float*>(smem + C::OFF_MERGE);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + C::NSTAGE;
  uint64_t* deposit = empty + C::NSTAGE;                            // [2] records ready
  uint64_t* mfree = deposit + 2;                                    // [2] records free
  long long* pre = reinterpret_cast<long long*>(smem + C::OFF_PRE);  // [B+1] (in units)
  int* lens = reinterpret_cast<int*>(pre + (p.B + 1));               // [B]

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int c = blockIdx.x;
  const int B = p.B, Hkv = p.Hkv;

  if (tid == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kCW);
    }
    for (int b2 = 0; b2 < 2; ++b2) {
      mbar_init(&deposit[b2], kCW);
      mbar_init(&mfree[b2], 1);
    }
    fence_barrier_init();
  }
  // ---- clamped context lengths and prefix sums of units
  int limit = p.max_seq_len;
  if (p.page_size == 0) limit = min(limit, p.capacity);
  else limit = min(limit, p.max_pages * p.page_size);
  // before the wait only reads that may be stale and L2 prefetches are issued
  if (warp == kCW && B <= 32) prefetch_first_chunks<C::RB, DV>(p, lane, limit, 2 * C::NSTAGE);
  pdl_wait();
  pdl_trigger();

  for (int b = tid; b < B; b += kThreads) {
    int L = p.seq_lens[b];
    if (p.fuse_append && L >= 0) ++L;  // the appended token is part of the context
    if (L < 0 || L > limit) {
      record_error(p.err, TK_DEVERR_INDEX);
      L = L < 0 ? 0 : limit;
    }
    lens[b] = L;
  }
  __syncthreads();
  if (warp == 0) {
    long long run = 0;
    for (int base = 0; base < B; base += 32) {
      const int b = base + lane;
      const long long x = b < B ? static_cast<long long>((lens[b] + kChunk - 1) / kChunk) * Hkv : 0;
      long long inc = x;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const long long y = __shfl_up_sync(0xffffffffu, inc, off);
        if (lane >= off) inc += y;
      }
      if (b < B) pre[b] = run + inc - x;
      run += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (lane == 0) pre[B] = run;
  }
  __syncthreads();
  const long long T = pre[B];
  // Partition over N = split_ctas(T, grid) CTAs: every owning CTA gets at
  // least one unit and the CTAs sharing a pair are consecutive; the rest own
  // nothing.
  const int N = split_ctas(T, gridDim.x);
  const long long u_begin = c < N ? T * c / N : T, u_end = c < N ? T * (c + 1) / N : T;

  if (warp == kCW) {
    // ------------------------------------------------------------------ producer
    const uint64_t pol = l2_policy_evict_first();
    const unsigned char* sbase = reinterpret_cast<const unsigned char*>(p.k_scale);
    const unsigned char* qbase = static_cast<const unsigned char*>(p.q);
    const int ps = p.page_size;
    const int rows_per_box = (ps == 0 || ps >= kChunk) ? kChunk : ps;
    if (lane == 0) {
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.k)) : "memory");
      asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&maps.v)) : "memory");
    }
    bool ok = true;
    for (long long w0 = u_begin; ok && w0 < u_end; w0 += 32) {
      // lane j prepares unit w0 + j: first cache row of the chunk, valid tokens, query offset
      long long row = 0, app = -1;
      int n = 0, qoff = 0, g = 0, b = 0, t0 = 0;
      const long long u = w0 + lane;
      if (u < u_end) {
        Walker wk;
        wk.seek(u, pre, lens, B, Hkv);
        b = wk.b; g = wk.g;
        t0 = wk.chunk * kChunk;
        n = min(kChunk, wk.Lb - t0);
        qoff = (b * p.Hq + g * G) * R;
        // Append fused into the decode: the chunk holding a pair's last token gets
        // the step's new token written at position seq_lens[b] (exactly as the
        // append kernel does) just before its TMA loads are issued; no other CTA
        // reads that chunk.  A clamped length (the token does not fit) gets no write.
        if (p.fuse_append && wk.chunk + 1 == wk.nb && p.seq_lens[b] == wk.Lb - 1) {
          const int pos = wk.Lb - 1;
          if (ps == 0) {
            app = (static_cast<long long>(b) * Hkv + g) * p.capacity + pos;
          } else {
            const int page = p.page_table[static_cast<long long>(b) * p.max_pages + (pos >> p.page_shift)];
            if (page >= 0 && page < p.num_pages)
              app = (static_cast<long long>(page) * Hkv + g) * ps + (pos & (ps - 1));
            else
              record_error(p.err, TK_DEVERR_INDEX);
          }
        }
        if (ps == 0) {
          row = (static_cast<long long>(b) * Hkv + g) * p.capacity + t0;
        } else {
          int page = p.page_table[static_cast<long long>(b) * p.max_pages + (t0 >> p.page_shift)];
          if (page < 0 || page >= p.num_pages) {
            record_error(p.err, TK_DEVERR_INDEX);
            page = 0;
          }
          row = (static_cast<long long>(page) * Hkv + g) * ps + (t0 & (ps - 1));
        }
      }
      const int cnt = static_cast<int>(min(32LL, u_end - w0));
      for (int j = 0; j < cnt; ++j) {
        const long long rj = __shfl_sync(0xffffffffu, row, j);
        const int nj = __shfl_sync(0xffffffffu, n, j);
        const int qj = __shfl_sync(0xffffffffu, qoff, j);
        const int bj = __shfl_sync(0xffffffffu, b, j);
        const int gj = __shfl_sync(0xffffffffu, g, j);
        const int tj = __shfl_sync(0xffffffffu, t0, j);
        const long long aj = __shfl_sync(0xffffffffu, app, j);
        if (aj >= 0) {
          // the new row, then a proxy fence: the TMA reads below see it
          const long long src = static_cast<long long>(bj) * Hkv + gj;
          write_kv_row<R, DV, KF>(const_cast<void*>(p.k), const_cast<void*>(p.v),
                                   const_cast<float*>(p.k_scale), static_cast<size_t>(aj),
                                   static_cast<const unsigned char*>(p.k_new) + src * 2 * R,
                                   static_cast<const unsigned char*>(p.v_new) + src * 2 * DV, lane);
          asm volatile("fence.proxy.async.global;" ::: "memory");
          __syncwarp();
          asm volatile("fence.proxy.async.global;" ::: "memory");
        }
        if (lane == 0) {
          const long long i = w0 + j - u_begin;
          const int st = static_cast<int>(i % C::NSTAGE);
          if (i >= C::NSTAGE && !mbar_wait(&empty[st], ((i / C::NSTAGE) - 1) & 1, p.err)) ok = false;
          if (ok) {
            unsigned char* sk = smem + st * C::STAGE;
            const uint32_t sbytes = KI8 ? ((nj + 3) & ~3) * 4 : 0;
            mbar_arrive_expect_tx(&full[st], C::KB + C::VB + sbytes + C::QB);
            // rows_per_box = 64 except for pages of 16 or 32 tokens
            for (int t = 0; t < kChunk; t += rows_per_box) {
              long long r2 = rj + t;
              if (t > 0 && ps != 0) {
                const int pidx = (tj + t) >> p.page_shift;
                // pages past the context are never read back: any valid page will do
                int page = pidx < p.max_pages ? p.page_table[static_cast<long long>(bj) * p.max_pages + pidx] : 0;
                if (page < 0 || page >= p.num_pages) page = 0;
                r2 = (static_cast<long long>(page) * Hkv + gj) * ps;
              }
#pragma unroll
              for (int kb = 0; kb < C::KBOX_N; ++kb)
                tma_load_2d(sk + kb * C::KBOX + t * C::KSW, &maps.k, kb * (C::KSW / (KI8 ? 1 : 2)),
                            static_cast<int>(r2), &full[st], pol);
#pragma unroll
              for (int vb = 0; vb < C::VBOX_N; ++vb)
                tma_load_2d(sk + C::OFF_V + vb * C::VBOX + t * 128, &maps.v, vb * 64,
                            static_cast<int>(r2), &full[st], pol);
              if (KI8) {
                const int m = min(rows_per_box, nj - t);
                if (m > 0)
                  bulk_g2s_hint(sk + C::OFF_S + t * 4, sbase + r2 * 4, ((m + 3) & ~3) * 4, &full[st], pol);
              }
            }
            bulk_g2s(sk + C::OFF_QS, qbase + static_cast<long long>(qj) * 2, C::QB, &full[st]);
          }
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
      }
    }
    return;
  }

  if (warp == kCW + 1) {
    // ------------------------------------------------------------------ merger
    // Empty contexts: zero rows (CTA b % grid writes sequence b).
    for (int b = c; b < B; b += gridDim.x) {
      if (lens[b] != 0) continue;
      for (int e = lane; e < p.Hq * DV; e += 32) {
        const long long o = static_cast<long long>(b) * p.Hq * DV + e;
        if (p.out_f32) reinterpret_cast<float*>(p.out)[o] = 0.f;
        else reinterpret_cast<__nv_bfloat16*>(p.out)[o] = __float2bfloat16_rn(0.f);
      }
    }
    merge_segments<R, DV, G, KF>(p, merge, deposit, mfree, pre, lens, T, N, c, u_begin, u_end, lane);
    return;
  }

  // -------------------------------------------------------------------- consumers
  if (u_begin == u_end) return;

  const int gq = lane >> 2, tq = lane & 3;  // mma fragment row group / column pair
  const int h0 = 2 * tq, h1 = 2 * tq + 1;    // the two heads (columns) this lane holds
  const float sl2 = p.scale_log2;
  uint32_t qf[C::KSTEPS][2];                 // Q^T as B fragments (bf16 pairs)
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[DV / 16][4];
  int seg = 0;
  bool dead = false;
  Walker wk;
  wk.seek(u_begin, pre, lens, B, Hkv);

  for (long long u = u_begin; u < u_end; ++u) {
    const long long i = u - u_begin;
    const int st = static_cast<int>(i % C::NSTAGE);
    if (!dead && !mbar_wait(&full[st], (i / C::NSTAGE) & 1, p.err)) dead = true;
    const unsigned char* sk = smem + st * C::STAGE;
    const uint32_t k_s = smem_addr(sk), v_s = smem_addr(sk + C::OFF_V);
    const float* ss = reinterpret_cast<const float*>(sk + C::OFF_S);
    const __nv_bfloat16* sq = reinterpret_cast<const __nv_bfloat16*>(sk + C::OFF_QS);
    const bool seg_first = (u == u_begin) || wk.chunk == 0;
    const bool seg_last = (u + 1 == u_end) || wk.chunk + 1 == wk.nb;
    if (seg_first) {
      // B fragments of Q^T: b0b1 = q[head gq][k 2tq, 2tq+1], b2b3 = q[gq][k 2tq+8, +9] of each
      // 16-wide k step.  For quantised keys the k order follows the codes ldmatrix
      // delivers: int8, mma k (2t, 2t+1, 8+2t, 9+2t) <-> r (4t .. 4t+3) within the step;
      // int4, steps 2c and 2c+1 take r 32c + 8t + {0..3} and 32c + 8t + {4..7}.
#pragma unroll
      for (int ks = 0; ks < C::KSTEPS; ++ks) {
        const int base = ks * 16;
        int k0, k2;
        if constexpr (KF == 2) {
          k0 = (ks >> 1) * 32 + (ks & 1) * 4 + 8 * tq;
          k2 = k0 + 2;
        } else if constexpr (KF == 1) {
          k0 = base + 4 * tq;
          k2 = k0 + 2;
        } else {
          k0 = base + 2 * tq;
          k2 = base + 2 * tq + 8;
        }
        float x0 = 0.f, x1 = 0.f, x2 = 0.f, x3 = 0.f;
        if (gq < G && !dead) {
          x0 = __bfloat162float(sq[gq * R + k0]);
          x1 = __bfloat162float(sq[gq * R + k0 + 1]);
          x2 = __bfloat162float(sq[gq * R + k2]);
          x3 = __bfloat162float(sq[gq * R + k2 + 1]);
        }
        qf[ks][0] = pack_bf16(x0, x1);  // exact: the values are bf16
        qf[ks][1] = pack_bf16(x2, x3);
      }
      m0 = m1 = -INFINITY;
      l0 = l1 = 0.f;
#pragma unroll
      for (int mt = 0; mt < DV / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    }
    const int nvalid = dead ? 0 : min(16, wk.Lb - wk.chunk * kChunk - warp * 16);
    if (nvalid > 0 && nvalid < 16) {
      // Ragged chunk: the rows past the context take part in V^T P^T with p = 0,
      // so clear them (unused cache slots may hold non-finite bytes).  A row of a
      // swizzled box is its 128 contiguous bytes, whatever the swizzle.
      unsigned char* vz = const_cast<unsigned char*>(sk) + C::OFF_V;
      const int nrow = 16 - nvalid;
      for (int e = lane; e < nrow * C::VBOX_N * 8; e += 32) {
        const int rrow = warp * 16 + nvalid + e / (C::VBOX_N * 8);
        const int rest = e % (C::VBOX_N * 8);
        *reinterpret_cast<uint4*>(vz + (rest / 8) * C::VBOX + rrow * 128 + (rest % 8) * 16) =
            make_uint4(0u, 0u, 0u, 0u);
      }
      // order these generic-proxy writes before the next TMA write of this stage
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
    }
    if (nvalid > 0) {
      // ---- S^T (16 tokens x 8 heads) = K Q^T
      float s[4] = {0.f, 0.f, 0.f, 0.f};
      const int mi = lane >> 3, rr = lane & 7;
      const uint32_t krow = warp * 16 + (mi & 1) * 8 + rr;
      if constexpr (!KI8) {
        // bf16 keys: one ldmatrix.x4 per 16-wide k step
#pragma unroll
        for (int ks = 0; ks < C::KSTEPS; ++ks) {
          const int kc = ks * 2 + (mi >> 1);  // 16-byte chunk of the key row
          const uint32_t addr = k_s + (kc / (C::KSW / 16)) * C::KBOX +
                                swz<C::KSW>(krow, (kc % (C::KSW / 16)) * 16);
          uint32_t a0, a1, a2, a3;
          ldsm_x4(addr, a0, a1, a2, a3);
          mma16816(s, a0, a1, a2, a3, qf[ks][0], qf[ks][1]);
        }
      } else if constexpr (KF == 2) {
        // int4 keys: a 16-byte chunk of a row holds 32 codes, two k steps; ldmatrix
        // hands lane (g, t) codes 8t..8t+7 of row g: 8t..8t+3 feed the first step,
        // 8t+4..8t+7 the second (the query's r order above matches)
        if constexpr (C::KSTEPS == 2) {
          uint32_t w0, w1;
          ldsm_x2(k_s + swz<C::KSW>(krow, 0), w0, w1);
          uint32_t x01, x23, x45, x67, y01, y23, y45, y67;
          i4x8_to_bf16(w0, x01, x23, x45, x67);
          i4x8_to_bf16(w1, y01, y23, y45, y67);
          mma16816(s, x01, y01, x23, y23, qf[0][0], qf[0][1]);
          mma16816(s, x45, y45, x67, y67, qf[1][0], qf[1][1]);
        } else {
#pragma unroll
          for (int kp = 0; kp < C::KSTEPS / 4; ++kp) {
            const int kc = kp * 2 + (mi >> 1);
            const uint32_t addr = k_s + (kc / (C::KSW / 16)) * C::KBOX +
                                  swz<C::KSW>(krow, (kc % (C::KSW / 16)) * 16);
            uint32_t w0, w1, w2, w3;  // (rows 0-7, chunk 2kp), (8-15, 2kp), (0-7, 2kp+1), (8-15, 2kp+1)
            ldsm_x4(addr, w0, w1, w2, w3);
            uint32_t x01, x23, x45, x67, y01, y23, y45, y67;
            i4x8_to_bf16(w0, x01, x23, x45, x67);
            i4x8_to_bf16(w1, y01, y23, y45, y67);
            mma16816(s, x01, y01, x23, y23, qf[4 * kp][0], qf[4 * kp][1]);
            mma16816(s, x45, y45, x67, y67, qf[4 * kp + 1][0], qf[4 * kp + 1][1]);
            i4x8_to_bf16(w2, x01, x23, x45, x67);
            i4x8_to_bf16(w3, y01, y23, y45, y67);
            mma16816(s, x01, y01, x23, y23, qf[4 * kp + 2][0], qf[4 * kp + 2][1]);
            mma16816(s, x45, y45, x67, y67, qf[4 * kp + 3][0], qf[4 * kp + 3][1]);
          }
        }
      } else {
        // int8 keys: a 16-byte chunk of a row holds one k step; ldmatrix hands lane
        // (g, t) bytes 4t..4t+3 of row g, widened here to bf16 pairs
        if constexpr (C::KSTEPS == 1) {
          uint32_t w0, w1;
          ldsm_x2(k_s + swz<C::KSW>(krow, 0), w0, w1);
          uint32_t a0, a1, a2, a3;
          i8x4_to_bf16(w0, a0, a2);
          i8x4_to_bf16(w1, a1, a3);
          mma16816(s, a0, a1, a2, a3, qf[0][0], qf[0][1]);
        } else {
#pragma unroll
          for (int kp = 0; kp < C::KSTEPS / 2; ++kp) {
            const int kc = kp * 2 + (mi >> 1);
            const uint32_t addr = k_s + (kc / (C::KSW / 16)) * C::KBOX +
                                  swz<C::KSW>(krow, (kc % (C::KSW / 16)) * 16);
            uint32_t w0, w1, w2, w3;  // (rows 0-7, step 2kp), (8-15, 2kp), (0-7, 2kp+1), (8-15, 2kp+1)
            ldsm_x4(addr, w0, w1, w2, w3);
            uint32_t a0, a1, a2, a3;
            i8x4_to_bf16(w0, a0, a2);
            i8x4_to_bf16(w1, a1, a3);
            mma16816(s, a0, a1, a2, a3, qf[2 * kp][0], qf[2 * kp][1]);
            i8x4_to_bf16(w2, a0, a2);
            i8x4_to_bf16(w3, a1, a3);
            mma16816(s, a0, a1, a2, a3, qf[2 * kp + 1][0], qf[2 * kp + 1][1]);
          }
        }
      }
      // s[0]: (token gq, head h0), s[1]: (gq, h1), s[2]: (gq+8, h0), s[3]: (gq+8, h1)
      const int ta = warp * 16 + gq, tb = ta + 8;
      float ka = sl2, kb = sl2;
      if (KI8) {
        ka *= ss[ta];
        kb *= ss[tb];
      }
      s[0] *= ka; s[1] *= ka; s[2] *= kb; s[3] *= kb;
      if (gq >= nvalid) s[0] = s[1] = -INFINITY;
      if (gq + 8 >= nvalid) s[2] = s[3] = -INFINITY;
      // ---- online softmax per head (the 8 lanes with the same tq hold one head pair)
      float c0 = fmaxf(s[0], s[2]), c1 = fmaxf(s[1], s[3]);
#pragma unroll
      for (int off = 4; off <= 16; off <<= 1) {
        c0 = fmaxf(c0, __shfl_xor_sync(0xffffffffu, c0, off));
        c1 = fmaxf(c1, __shfl_xor_sync(0xffffffffu, c1, off));
      }
      const float n0 = fmaxf(m0, c0), n1 = fmaxf(m1, c1);
      const float al0 = fast_exp2(m0 - n0), al1 = fast_exp2(m1 - n1);  // 0 on a segment's first chunk
      m0 = n0;
      m1 = n1;
      const float p0 = fast_exp2(s[0] - n0), p1 = fast_exp2(s[1] - n1);
      const float p2 = fast_exp2(s[2] - n0), p3 = fast_exp2(s[3] - n1);
      l0 = l0 * al0 + (p0 + p2);
      l1 = l1 * al1 + (p1 + p3);
      // P^T as the B operand: transpose the two 8x8 bf16 blocks of the S^T accumulator
      const uint32_t pb0 = movm_t(pack_bf16(p0, p1));
      const uint32_t pb1 = movm_t(pack_bf16(p2, p3));
      // ---- O^T = alpha O^T + V^T P^T
      const uint32_t vrow = warp * 16 + (mi >> 1) * 8 + rr;
#pragma unroll
      for (int mt = 0; mt < DV / 16; ++mt) {
        o[mt][0] *= al0; o[mt][1] *= al1; o[mt][2] *= al0; o[mt][3] *= al1;
        const int dc = mt * 2 + (mi & 1);   // 16-byte chunk of the value row (8 values)
        const uint32_t addr = v_s + (dc / 8) * C::VBOX + swz<128>(vrow, (dc % 8) * 16);
        uint32_t a0, a1, a2, a3;
        ldsm_x4_t(addr, a0, a1, a2, a3);
        mma16816(o[mt], a0, a1, a2, a3, pb0, pb1);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[st]);

    if (seg_last) {
      // ---------------------------------------------------------------- segment end
      // deposit this warp's state for the merger warp and keep streaming
      const int buf = seg & 1;
      if (seg >= 2 && !dead && !mbar_wait(&mfree[buf], ((seg >> 1) - 1) & 1, p.err)) dead = true;
      float* rec = merge + (buf * kCW + warp) * C::REC;  // [G][DV] O, [G] m, [G] l
      float lt0 = l0, lt1 = l1;
#pragma unroll
      for (int off = 4; off <= 16; off <<= 1) {
        lt0 += __shfl_xor_sync(0xffffffffu, lt0, off);
        lt1 += __shfl_xor_sync(0xffffffffu, lt1, off);
      }
      if (h0 < G) {
#pragma unroll
        for (int mt = 0; mt < DV / 16; ++mt) {
          rec[h0 * DV + mt * 16 + gq] = o[mt][0];
          rec[h0 * DV + mt * 16 + gq + 8] = o[mt][2];
        }
        if (gq == 0) {
          rec[G * DV + h0] = m0;
          rec[G * DV + G + h0] = lt0;
        }
      }
      if (h1 < G) {
#pragma unroll
        for (int mt = 0; mt < DV / 16; ++mt) {
          rec[h1 * DV + mt * 16 + gq] = o[mt][1];
          rec[h1 * DV + mt * 16 + gq + 8] = o[mt][3];
        }
        if (gq == 0) {
          rec[G * DV + h1] = m1;
          rec[G * DV + G + h1] = lt1;
        }
      }
      __threadfence_block();
      __syncwarp();
      if (lane == 0) mbar_arrive(&deposit[buf]);
      ++seg;
    }
    if (u + 1 < u_end) wk.next(pre, lens, Hkv);
  }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D map over `rows` rows of `width` elements, box (box_w elements x box_rows rows).
bool make_map_2d(CUtensorMap* m, const void* base, bool int8, long long width, long long rows,
                 int box_w, int box_rows, int swizzle_bytes) {
  auto enc = encode_fn();
  if (!enc) return false;
  const int es = int8 ? 1 : 2;
  cuuint64_t dims[2] = {static_cast<cuuint64_t>(width), static_cast<cuuint64_t>(rows)};
  cuuint64_t strides[1] = {static_cast<cuuint64_t>(width) * es};
  cuuint32_t box[2] = {static_cast<cuuint32_t>(box_w), static_cast<cuuint32_t>(box_rows)};
  cuuint32_t estr[2] = {1, 1};
  CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                          : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                          : swizzle_bytes == 32 ? CU_TENSOR_MAP_SWIZZLE_32B
                                                : CU_TENSOR_MAP_SWIZZLE_NONE;
  return enc(m, int8 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
             const_cast<void*>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
             CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int R, int DV, int G, int KF>
cudaError_t launch_t(const DecodeParams& p, cudaStream_t stream) {
  using C = Cfg<R, DV, G, KF>;
  constexpr bool KI8 = KF != 0;  // quantised keys (int8 or int4)
  // cache rows: contiguous [B*Hkv*cap], paged [P*Hkv*page_size]
  const long long rows = p.page_size == 0
                             ? static_cast<long long>(p.B) * p.Hkv * p.capacity
                             : static_cast<long long>(p.num_pages) * p.Hkv * p.page_size;
  if (rows >= (1LL << 31)) return cudaErrorInvalidValue;  // TMA row coordinates are 32-bit
  const int box_rows = (p.page_size == 0 || p.page_size >= kChunk) ? kChunk : p.page_size;
  DecodeMaps maps;
  if (!make_map_2d(&maps.k, p.k, KI8, KF == 2 ? R / 2 : R, rows, C::KSW / (KI8 ? 1 : 2), box_rows,
                   C::KSW) ||
      !make_map_2d(&maps.v, p.v, false, DV, rows, 64, box_rows, 128))
    return cudaErrorInvalidValue;
  auto kern = decode_kernel<R, DV, G, KF>;
  const int smem = C::OFF_PRE + (p.B + 1) * 8 + p.B * 4 + 1024;  // + alignment slack
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(kern, dim3(p.n_cta), dim3(kThreads), smem, stream, maps, p);
}

// Calls f.template run<R, DV, G, KF>() for the compiled shape; sets *uns otherwise.
template <typename F>
auto dispatch(int R, int DV, int G, int kf, F&& f, int* uns) {
  using Ret = decltype(f.template run<16, 64, 1, 0>());
#define TK_G(R_, DV_, K_)                                      \
  switch (G) {                                                 \
    case 1: return f.template run<R_, DV_, 1, K_>();           \
    case 2: return f.template run<R_, DV_, 2, K_>();           \
    case 4: return f.template run<R_, DV_, 4, K_>();           \
    case 8: return f.template run<R_, DV_, 8, K_>();           \
  }
#define TK_DV(R_, K_)        \
  if (DV == 64) {            \
    TK_G(R_, 64, K_)         \
  } else if (DV == 128) {    \
    TK_G(R_, 128, K_)        \
  }
#define TK_R(K_)                     \
  switch (R) {                       \
    case 32: { TK_DV(32, K_) } break;  \
    case 64: { TK_DV(64, K_) } break;  \
    case 128: { TK_DV(128, K_) } break; \
  }
  if (kf == 0) {
    if (R == 16) { TK_DV(16, 0) }
    TK_R(0)
  } else if (kf == 1) {
    if (R == 16) { TK_DV(16, 1) }
    TK_R(1)
  } else if (kf == 2) {
    TK_R(2)  // int4 keys need r >= 32
  }
#undef TK_R
#undef TK_DV
#undef TK_G
  *uns = 1;
  return Ret{};
}

struct CtasPerSm {
  template <int R, int DV, int G, int K>
  int run() { return Cfg<R, DV, G, K>::CTAS_PER_SM; }
};

struct Launch {
  const DecodeParams* p;
  cudaStream_t s;
  template <int R, int DV, int G, int K>
  cudaError_t run() { return launch_t<R, DV, G, K>(*p, s); }
};

}  // namespace

int decode_max_batch() { return kMaxBatch; }

DecodePlan plan_decode(int B, int Hq, int Hkv, int R, int DV, int k_fmt, int num_sms) {
  DecodePlan pl{};
  int uns = 0;
  const int per_sm = dispatch(R, DV, Hq / Hkv, k_fmt, CtasPerSm{}, &uns);
  pl.n_cta = num_sms * (uns ? 1 : per_sm);
  const int G = Hq / Hkv;
  const size_t rec = (static_cast<size_t>(G) * DV + 2 * G + 3) / 4 * 4;
  auto align = [](size_t x) { return (x + 255) / 256 * 256; };
  pl.off_counters = 0;
  pl.off_part = align(static_cast<size_t>(B) * Hkv * 4);
  pl.bytes = pl.off_part + align(static_cast<size_t>(pl.n_cta) * 2 * rec * 4);
  return pl;
}

cudaError_t launch_decode(const DecodeParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  if (p.B > kMaxBatch) {
    *unsupported = 1;
    return cudaSuccess;
  }
  return dispatch(p.R, p.DV, p.G, p.k_fmt, Launch{&p, stream}, unsupported);
}

}  // namespace tk
