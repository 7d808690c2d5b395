// Split-KV decode attention over a thin-key / full-value cache.
//
// Paper: Section 2.1, Eq. 4 with a single query row per head; decode is the
// bandwidth-bound case of Section 4.2 (every step streams the whole cache).
//
// One CTA handles one (sequence b, kv head g, token split s).  It streams the
// split's r-wide key rows and d_v-wide value rows from HBM once and serves all
// G = h_q / h_kv query heads of the group from that single read.
//
//   warp 4 (producer, one lane): 1-D bulk async copies (cp.async.bulk) of
//     64-token chunks into an NSTAGE-deep shared-memory ring, completion
//     tracked by "full" mbarriers; it refills a stage once the four consumer
//     warps have released it on its "empty" mbarrier.
//   warps 0-3 (consumers): warp w owns tokens 16w..16w+15 of every chunk and
//     keeps its own online-softmax state (running max m, sum l, output acc)
//     for the G heads; lane = (token, half of the heads) for the scores,
//     lane = (d_v / 32 columns, all heads) for the weighted sum.  No block
//     barrier inside the loop.
//   After the loop the four warp states are merged in shared memory.  With a
//   single split the CTA writes the normalised output; otherwise it writes
//   its (m, l, o) partial and bumps an arrival counter, and the last CTA of
//   the (b, g) group merges all splits (no CTA ever waits for another).
//
// Scores are kept in log2 units (q pre-multiplied by scale * log2 e) so the
// softmax uses exp2.  All accumulation is fp32.
#include "common.cuh"
#include "kernels.h"

namespace tk {
namespace {

constexpr int kChunk = 64;         // tokens per pipeline stage
constexpr int kConsumerWarps = 4;
constexpr int kTokPerWarp = kChunk / kConsumerWarps;  // 16
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kMaxSplit = 256;

__device__ __forceinline__ void consumer_sync() {
  asm volatile("bar.sync 1, 128;" ::: "memory");
}

template <int R, int DV, int G, bool KI8>
struct Cfg {
  static constexpr int KROW = KI8 ? R : 2 * R;  // bytes per cached key row
  static constexpr int VROW = 2 * DV;
  static constexpr int KB = kChunk * KROW;
  static constexpr int VB = kChunk * VROW;
  static constexpr int SB = KI8 ? kChunk * 4 : 0;
  static constexpr int STAGE = KB + VB + SB;
  static constexpr int NSTAGE_RAW = 98304 / STAGE;
  static constexpr int NSTAGE = NSTAGE_RAW < 2 ? 2 : (NSTAGE_RAW > 8 ? 8 : NSTAGE_RAW);
  static constexpr int RING = NSTAGE * STAGE;
  static constexpr int QPAD = R + 4;  // padded fp32 row of the scaled query
  static constexpr int HPL = G >= 2 ? G / 2 : 1;  // heads per lane in the score phase
  static constexpr int CPL = DV / 32;             // value columns per lane
  // Shared memory map (bytes)
  static constexpr int OFF_Q = RING;
  static constexpr int OFF_P = OFF_Q + G * QPAD * 4;
  static constexpr int OFF_BAR = (OFF_P + kConsumerWarps * kTokPerWarp * G * 4 + 15) / 16 * 16;
  static constexpr int OFF_FLAG = OFF_BAR + 2 * NSTAGE * 8;
  static constexpr int SMEM = OFF_FLAG + 16;
  // Post-loop merge area, aliased onto the ring.
  static constexpr int M_O = 0;                                        // [4][G][DV]
  static constexpr int M_ML = M_O + kConsumerWarps * G * DV * 4;       // [4][G][2]
  static constexpr int M_W = M_ML + kConsumerWarps * G * 2 * 4;        // [kMaxSplit][G]
  static_assert(M_W + kMaxSplit * G * 4 <= RING, "merge area must fit in the ring");
  static_assert(STAGE % 16 == 0 && KB % 16 == 0 && VB % 16 == 0, "16-byte staging");
};

// Converts 8 cached key elements (16 bytes of bf16 or 8 bytes of int8) to fp32.
template <bool KI8>
__device__ __forceinline__ void load_k8(const unsigned char* p, float* f) {
  if constexpr (KI8) {
    uint2 w = *reinterpret_cast<const uint2*>(p);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[i] = static_cast<float>(static_cast<int8_t>((w.x >> (8 * i)) & 0xff));
      f[4 + i] = static_cast<float>(static_cast<int8_t>((w.y >> (8 * i)) & 0xff));
    }
  } else {
    uint4 w = *reinterpret_cast<const uint4*>(p);
    f[0] = bf16lo(w.x); f[1] = bf16hi(w.x); f[2] = bf16lo(w.y); f[3] = bf16hi(w.y);
    f[4] = bf16lo(w.z); f[5] = bf16hi(w.z); f[6] = bf16lo(w.w); f[7] = bf16hi(w.w);
  }
}

template <int R, int DV, int G, bool KI8>
__global__ void __launch_bounds__(kThreads)
decode_kernel(const DecodeParams p) {
  using C = Cfg<R, DV, G, KI8>;
  extern __shared__ __align__(128) unsigned char smem[];
  float* qs = reinterpret_cast<float*>(smem + C::OFF_Q);
  float* pw = reinterpret_cast<float*>(smem + C::OFF_P);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + C::OFF_BAR);
  uint64_t* empty = full + C::NSTAGE;
  int* flag = reinterpret_cast<int*>(smem + C::OFF_FLAG);

  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

  // ---- context length of this sequence (validated on the device)
  int L = p.seq_lens[b];
  int limit = p.max_seq_len;
  if (p.page_size == 0) limit = min(limit, p.capacity);
  else limit = min(limit, p.max_pages * p.page_size);
  if (L < 0 || L > limit) {
    if (tid == 0) record_error(p.err, TK_DEVERR_INDEX);
    L = L < 0 ? 0 : limit;
  }
  const int split_tokens = p.split_chunks * kChunk;
  const int nsplit_b = (L + split_tokens - 1) / split_tokens;
  const int h0 = g * G;  // first query head of the group

  if (split >= nsplit_b) {
    if (L == 0 && split == 0) {  // empty context: zero rows
      for (int i = tid; i < G * DV; i += kThreads) {
        size_t o = (static_cast<size_t>(b) * p.Hq + h0 + i / DV) * DV + (i % DV);
        if (p.out_f32) reinterpret_cast<float*>(p.out)[o] = 0.f;
        else reinterpret_cast<__nv_bfloat16*>(p.out)[o] = __float2bfloat16_rn(0.f);
      }
    }
    return;
  }
  const int tok_begin = split * split_tokens;
  const int tok_end = min(L, tok_begin + split_tokens);
  const int nchunks = (tok_end - tok_begin + kChunk - 1) / kChunk;

  if (tid == 0) {
    for (int s = 0; s < C::NSTAGE; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], kConsumerWarps);
    }
    fence_barrier_init();
  }
  __syncthreads();

  if (warp == kConsumerWarps) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      const uint64_t pol = l2_policy_evict_first();
      const unsigned char* kbase = static_cast<const unsigned char*>(p.k);
      const unsigned char* vbase = static_cast<const unsigned char*>(p.v);
      const unsigned char* sbase = reinterpret_cast<const unsigned char*>(p.k_scale);
      for (int i = 0; i < nchunks; ++i) {
        const int st = i % C::NSTAGE;
        if (i >= C::NSTAGE && !mbar_wait(&empty[st], ((i / C::NSTAGE) - 1) & 1, p.err)) break;
        const int t0 = tok_begin + i * kChunk;
        const int n = min(kChunk, tok_end - t0);
        unsigned char* sk = smem + st * C::STAGE;
        unsigned char* sv = sk + C::KB;
        unsigned char* ss = sv + C::VB;
        if (p.page_size == 0) {
          const size_t row = (static_cast<size_t>(b) * p.Hkv + g) * p.capacity + t0;
          const uint32_t sbytes = KI8 ? ((n + 3) & ~3) * 4 : 0;
          mbar_arrive_expect_tx(&full[st], n * (C::KROW + C::VROW) + sbytes);
          bulk_g2s_hint(sk, kbase + row * C::KROW, n * C::KROW, &full[st], pol);
          bulk_g2s_hint(sv, vbase + row * C::VROW, n * C::VROW, &full[st], pol);
          if (KI8) bulk_g2s_hint(ss, sbase + row * 4, sbytes, &full[st], pol);
        } else {
          // The chunk lies in one page (page_size >= 64) or spans 64/page_size pages.
          const int ps = p.page_size;
          uint32_t total = 0;
          for (int j = 0; j < n;) {
            const int nj = min(n - j, ps - ((t0 + j) & (ps - 1)));
            total += nj * (C::KROW + C::VROW) + (KI8 ? ((nj + 3) & ~3) * 4 : 0);
            j += nj;
          }
          mbar_arrive_expect_tx(&full[st], total);
          for (int j = 0; j < n;) {
            const int t = t0 + j;
            const int slot = t & (ps - 1);
            const int nj = min(n - j, ps - slot);
            int page = p.page_table[static_cast<size_t>(b) * p.max_pages + (t >> p.page_shift)];
            if (page < 0 || page >= p.num_pages) {
              record_error(p.err, TK_DEVERR_INDEX);
              page = 0;
            }
            const size_t row = (static_cast<size_t>(page) * p.Hkv + g) * ps + slot;
            bulk_g2s_hint(sk + j * C::KROW, kbase + row * C::KROW, nj * C::KROW, &full[st], pol);
            bulk_g2s_hint(sv + j * C::VROW, vbase + row * C::VROW, nj * C::VROW, &full[st], pol);
            if (KI8)
              bulk_g2s_hint(ss + j * 4, sbase + row * 4, ((nj + 3) & ~3) * 4, &full[st], pol);
            j += nj;
          }
        }
      }
    }
  } else {
    // ------------------------------------------------------------ consumers
    // Scaled query of the G heads, fp32 in shared memory.
    const __nv_bfloat16* qg =
        static_cast<const __nv_bfloat16*>(p.q) + (static_cast<size_t>(b) * p.Hq + h0) * R;
    for (int i = tid; i < G * R; i += 128)
      qs[(i / R) * C::QPAD + (i % R)] = __bfloat162float(qg[i]) * p.scale_log2;
    consumer_sync();

    const int tl = lane & 15;   // token within the warp's 16
    const int hs = lane >> 4;   // head half (score phase)
    float m[G], lsum[C::HPL];
    float2 acc[G][C::CPL / 2];
#pragma unroll
    for (int h = 0; h < G; ++h) {
      m[h] = -INFINITY;
#pragma unroll
      for (int c = 0; c < C::CPL / 2; ++c) acc[h][c] = make_float2(0.f, 0.f);
    }
#pragma unroll
    for (int j = 0; j < C::HPL; ++j) lsum[j] = 0.f;
    float* pwarp = pw + warp * kTokPerWarp * G;
    bool dead = false;

    for (int i = 0; i < nchunks; ++i) {
      const int st = i % C::NSTAGE;
      if (!dead && !mbar_wait(&full[st], (i / C::NSTAGE) & 1, p.err)) dead = true;
      if (dead) break;
      const int t0 = tok_begin + i * kChunk;
      const int nvalid = min(kTokPerWarp, tok_end - t0 - warp * kTokPerWarp);
      if (nvalid > 0) {
        const unsigned char* sk = smem + st * C::STAGE;
        const unsigned char* sv = sk + C::KB;
        const float* ss = reinterpret_cast<const float*>(sv + C::VB);
        const int tok = warp * kTokPerWarp + tl;  // token within the chunk
        // ---- scores s = (scale log2 e) q . k for this lane's token and heads
        constexpr int RL = (G == 1) ? R / 2 : R;
        const int r0 = (G == 1) ? hs * RL : 0;
        float2 s2[C::HPL];
#pragma unroll
        for (int j = 0; j < C::HPL; ++j) s2[j] = make_float2(0.f, 0.f);
        const unsigned char* krow = sk + tok * C::KROW + (KI8 ? r0 : 2 * r0);
#pragma unroll
        for (int c = 0; c < RL; c += 8) {
          float kf[8];
          load_k8<KI8>(krow + (KI8 ? c : 2 * c), kf);
#pragma unroll
          for (int j = 0; j < C::HPL; ++j) {
            const int h = (G == 1) ? 0 : hs * C::HPL + j;
            const float4 qa = *reinterpret_cast<const float4*>(qs + h * C::QPAD + r0 + c);
            const float4 qb = *reinterpret_cast<const float4*>(qs + h * C::QPAD + r0 + c + 4);
            s2[j] = ffma2(make_float2(qa.x, qa.y), make_float2(kf[0], kf[1]), s2[j]);
            s2[j] = ffma2(make_float2(qa.z, qa.w), make_float2(kf[2], kf[3]), s2[j]);
            s2[j] = ffma2(make_float2(qb.x, qb.y), make_float2(kf[4], kf[5]), s2[j]);
            s2[j] = ffma2(make_float2(qb.z, qb.w), make_float2(kf[6], kf[7]), s2[j]);
          }
        }
        float s[C::HPL];
#pragma unroll
        for (int j = 0; j < C::HPL; ++j) {
          s[j] = s2[j].x + s2[j].y;
          if (G == 1) s[j] += __shfl_xor_sync(0xffffffffu, s[j], 16);
          if (KI8) s[j] *= ss[tok];
          if (tl >= nvalid) s[j] = -INFINITY;
        }
        // ---- chunk max per head over the warp's 16 tokens, then broadcast all heads
        float cm[C::HPL];
#pragma unroll
        for (int j = 0; j < C::HPL; ++j) {
          cm[j] = s[j];
#pragma unroll
          for (int off = 8; off >= 1; off >>= 1)
            cm[j] = fmaxf(cm[j], __shfl_xor_sync(0xffffffffu, cm[j], off));
        }
        float alpha[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float c = __shfl_sync(0xffffffffu, cm[h % C::HPL], (G == 1) ? 0 : (h / C::HPL) * 16);
          const float mn = fmaxf(m[h], c);
          alpha[h] = fast_exp2(m[h] - mn);  // exp2(-inf) = 0 on the first chunk
          m[h] = mn;
        }
        // ---- weights of this chunk
#pragma unroll
        for (int j = 0; j < C::HPL; ++j) {
          const int h = (G == 1) ? 0 : hs * C::HPL + j;
          const float pj = fast_exp2(s[j] - m[h]);
          if (G > 1 || hs == 0) {
            lsum[j] = lsum[j] * alpha[h] + pj;
            pwarp[tl * G + h] = pj;
          }
        }
        __syncwarp();
        // ---- acc = alpha * acc + sum_t p_t v_t over this lane's value columns
#pragma unroll
        for (int h = 0; h < G; ++h) {
          const float2 a2 = make_float2(alpha[h], alpha[h]);
#pragma unroll
          for (int c = 0; c < C::CPL / 2; ++c) acc[h][c] = fmul2(acc[h][c], a2);
        }
        const unsigned char* vcol = sv + (warp * kTokPerWarp) * C::VROW + lane * C::CPL * 2;
#pragma unroll 4
        for (int t = 0; t < nvalid; ++t) {
          float2 vv[C::CPL / 2];
          if constexpr (C::CPL == 4) {
            const uint2 w = *reinterpret_cast<const uint2*>(vcol + t * C::VROW);
            vv[0] = make_float2(bf16lo(w.x), bf16hi(w.x));
            vv[1] = make_float2(bf16lo(w.y), bf16hi(w.y));
          } else {
            const uint32_t w = *reinterpret_cast<const uint32_t*>(vcol + t * C::VROW);
            vv[0] = make_float2(bf16lo(w), bf16hi(w));
          }
          float pt[G];
          if constexpr (G % 4 == 0) {
#pragma unroll
            for (int h = 0; h < G; h += 4) {
              const float4 x = *reinterpret_cast<const float4*>(pwarp + t * G + h);
              pt[h] = x.x; pt[h + 1] = x.y; pt[h + 2] = x.z; pt[h + 3] = x.w;
            }
          } else {
#pragma unroll
            for (int h = 0; h < G; ++h) pt[h] = pwarp[t * G + h];
          }
#pragma unroll
          for (int h = 0; h < G; ++h) {
            const float2 p2 = make_float2(pt[h], pt[h]);
#pragma unroll
            for (int c = 0; c < C::CPL / 2; ++c) acc[h][c] = ffma2(p2, vv[c], acc[h][c]);
          }
        }
        __syncwarp();
      }
      if (lane == 0) mbar_arrive(&empty[st]);
    }

    // ---- merge the four warps' states (merge area aliases the drained ring)
    consumer_sync();
    float* mo = reinterpret_cast<float*>(smem + C::M_O);
    float* mml = reinterpret_cast<float*>(smem + C::M_ML);
    float* wts = reinterpret_cast<float*>(smem + C::M_W);
#pragma unroll
    for (int j = 0; j < C::HPL; ++j) {
      float l = lsum[j];
#pragma unroll
      for (int off = 8; off >= 1; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
      const int h = (G == 1) ? 0 : hs * C::HPL + j;
      if (tl == 0 && (G > 1 || hs == 0)) {
        mml[(warp * G + h) * 2 + 0] = m[h];
        mml[(warp * G + h) * 2 + 1] = l;
      }
    }
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
      for (int c = 0; c < C::CPL / 2; ++c)
        *reinterpret_cast<float2*>(mo + (warp * G + h) * DV + lane * C::CPL + 2 * c) = acc[h][c];
    consumer_sync();

    const size_t pair = static_cast<size_t>(b) * p.Hkv + g;
    for (int i = tid; i < G * DV; i += 128) {
      const int h = i / DV, d = i % DV;
      float M = -INFINITY;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) M = fmaxf(M, mml[(w * G + h) * 2]);
      float O = 0.f, Lw = 0.f;
#pragma unroll
      for (int w = 0; w < kConsumerWarps; ++w) {
        const float f = fast_exp2(mml[(w * G + h) * 2] - M);
        O += f * mo[(w * G + h) * DV + d];
        Lw += f * mml[(w * G + h) * 2 + 1];
      }
      if (nsplit_b == 1) {
        const size_t o = (static_cast<size_t>(b) * p.Hq + h0 + h) * DV + d;
        if (p.out_f32) reinterpret_cast<float*>(p.out)[o] = O / Lw;
        else reinterpret_cast<__nv_bfloat16*>(p.out)[o] = __float2bfloat16_rn(O / Lw);
      } else {
        const size_t base = (pair * p.n_split + split) * G + h;
        p.part_o[base * DV + d] = O;
        if (d == 0) {
          p.part_ml[base * 2 + 0] = M;
          p.part_ml[base * 2 + 1] = Lw;
        }
      }
    }
    if (nsplit_b == 1) return;

    // ---- last CTA of the (b, g) group merges all splits
    __threadfence();
    consumer_sync();
    if (tid == 0) {
      const int old = atomicAdd(&p.counters[pair], 1);
      flag[0] = (old == nsplit_b - 1);
    }
    consumer_sync();
    if (!flag[0]) return;
    __threadfence();
    // warp w computes the split weights of heads w, w+4, ...
    for (int h = warp; h < G; h += kConsumerWarps) {
      float M = -INFINITY;
      for (int s = lane; s < nsplit_b; s += 32)
        M = fmaxf(M, __ldcg(p.part_ml + ((pair * p.n_split + s) * G + h) * 2));
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, off));
      float Lt = 0.f;
      for (int s = lane; s < nsplit_b; s += 32) {
        const size_t base = ((pair * p.n_split + s) * G + h) * 2;
        const float f = fast_exp2(__ldcg(p.part_ml + base) - M);
        wts[s * G + h] = f;
        Lt += f * __ldcg(p.part_ml + base + 1);
      }
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) Lt += __shfl_xor_sync(0xffffffffu, Lt, off);
      __syncwarp();
      const float inv = 1.f / Lt;
      for (int s = lane; s < nsplit_b; s += 32) wts[s * G + h] *= inv;
    }
    consumer_sync();
    for (int i = tid; i < G * DV; i += 128) {
      const int h = i / DV, d = i % DV;
      float O = 0.f;
      for (int s = 0; s < nsplit_b; ++s)
        O += wts[s * G + h] * __ldcg(p.part_o + ((pair * p.n_split + s) * G + h) * DV + d);
      const size_t o = (static_cast<size_t>(b) * p.Hq + h0 + h) * DV + d;
      if (p.out_f32) reinterpret_cast<float*>(p.out)[o] = O;
      else reinterpret_cast<__nv_bfloat16*>(p.out)[o] = __float2bfloat16_rn(O);
    }
    if (tid == 0) p.counters[pair] = 0;  // ready for the next launch
  }
}

template <int R, int DV, int G, bool KI8>
cudaError_t launch_t(const DecodeParams& p, cudaStream_t stream) {
  using C = Cfg<R, DV, G, KI8>;
  auto kern = decode_kernel<R, DV, G, KI8>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
  if (e != cudaSuccess) return e;
  dim3 grid(p.n_split, p.Hkv, p.B);
  kern<<<grid, kThreads, C::SMEM, stream>>>(p);
  return cudaGetLastError();
}

template <int R, int DV, bool KI8>
cudaError_t by_g(const DecodeParams& p, cudaStream_t s, int* uns) {
  switch (p.G) {
    case 1: return launch_t<R, DV, 1, KI8>(p, s);
    case 2: return launch_t<R, DV, 2, KI8>(p, s);
    case 4: return launch_t<R, DV, 4, KI8>(p, s);
    case 8: return launch_t<R, DV, 8, KI8>(p, s);
  }
  *uns = 1;
  return cudaSuccess;
}

template <int R, bool KI8>
cudaError_t by_dv(const DecodeParams& p, cudaStream_t s, int* uns) {
  switch (p.DV) {
    case 64: return by_g<R, 64, KI8>(p, s, uns);
    case 128: return by_g<R, 128, KI8>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

template <bool KI8>
cudaError_t by_r(const DecodeParams& p, cudaStream_t s, int* uns) {
  switch (p.R) {
    case 16: return by_dv<16, KI8>(p, s, uns);
    case 32: return by_dv<32, KI8>(p, s, uns);
    case 64: return by_dv<64, KI8>(p, s, uns);
    case 128: return by_dv<128, KI8>(p, s, uns);
  }
  *uns = 1;
  return cudaSuccess;
}

}  // namespace

DecodePlan plan_decode(int B, int Hq, int Hkv, int DV, int max_seq_len, int num_sms) {
  DecodePlan pl{};
  const int chunks = max(1, (max_seq_len + kChunk - 1) / kChunk);
  const long pairs = static_cast<long>(B) * Hkv;
  // Aim for about eight CTAs per SM over the launch so that the last wave is
  // short, with at least four chunks per split to amortise the pipeline fill.
  const long target = 8L * num_sms;
  int n = static_cast<int>((target + pairs - 1) / pairs);
  n = max(1, min(n, min(kMaxSplit, max(1, chunks / 4))));
  pl.split_chunks = (chunks + n - 1) / n;
  pl.n_split = (chunks + pl.split_chunks - 1) / pl.split_chunks;
  const int G = Hq / Hkv;
  auto align = [](size_t x) { return (x + 255) / 256 * 256; };
  pl.off_counters = 0;
  pl.off_ml = align(static_cast<size_t>(pairs) * 4);
  pl.off_o = pl.off_ml + align(static_cast<size_t>(pairs) * pl.n_split * G * 2 * 4);
  pl.bytes = pl.off_o + align(static_cast<size_t>(pairs) * pl.n_split * G * DV * 4);
  return pl;
}

cudaError_t launch_decode(const DecodeParams& p, cudaStream_t stream, int* unsupported) {
  *unsupported = 0;
  return p.k_int8 ? by_r<true>(p, stream, unsupported) : by_r<false>(p, stream, unsupported);
}

}  // namespace tk
