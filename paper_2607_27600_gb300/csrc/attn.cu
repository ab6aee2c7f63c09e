// attn.cu -- counter-causal flash attention on tcgen05 (Sec. 3.1: fresh
// queries, cached post-RoPE K/V reused, row i attends only slots j with
// i < j < n).  The same kernel, CAUSAL = true, runs the inference cycle's
// memory-augmented attention (Eq. 3 with the causal mask): the chunk's rows
// [row_lo, n) attend slots j <= i, i.e. every memory slot and the chunk
// causally; key tiles then run from the one holding the block's last row
// down to slot 0.
//
// One CTA = one work unit (sequence b, KV head g, block of P positions).
// The unit's query rows are the G = Hq/Hkv heads of group g at P
// consecutive positions, row r = position * G + head, so that P*G <= 256
// rows form two M=128 MMA tiles that share every K/V tile loaded (a GQA
// group is served by one K/V stream).  Key tiles of 128 slots run from the
// one holding slot n-1 down to the one holding slot p0+1: whole tiles at or
// below the diagonal are never loaded, and units running at the same time
// sweep the same keys in step (L2 reuse when K/V exceed L2).
//
//   warps 0..3, 4..7  softmax of M-half 0 / 1 (one row per thread): S from
//                     TMEM, mask, online softmax (log2 domain, lazy rescale),
//                     P (bf16) written back over S in TMEM, final O / l
//   warp 8            TMA producer (Q once; K and V tiles, 2 stages each);
//                     zeroes V rows past the sequence end in the last tile
//   warp 9            TMEM owner + tcgen05.mma issuer of M-half 0:
//                     S_h = Q_h K^T (SS),  O_h += P_h V (TS, P from TMEM)
//   warp 10           tcgen05.mma issuer of M-half 1
//   warp 11           idle (completes the third warpgroup)
//
// An e4m3 cache reaches this kernel as an exact bf16 copy of the layer's
// codes (made by the caller), its K scale folded into the softmax scale and
// its V scale into the output normalisation.
//
// SPLIT (the precise scoring pass over a bf16 cache): the queries arrive as
// bf16 pairs hi + lo (hi = bf16(q), lo = bf16(q - hi)), so S = Q_hi K^T +
// Q_lo K^T accumulates both products in TMEM, and P is handed to P V as the
// pair P_hi (TMEM columns [0, 64) of the S block) + P_lo (columns [64, 128)),
// two TS products into O.  K and V are exact bf16 inputs, so every operand of
// both contractions then carries about 16 significant bits.  The second Q
// tile costs 64 KB of shared memory at head_dim 128; the V ring then has one
// stage.
//
// F16 (the fp16 operand mode of the scoring pass): Q, K and V arrive as fp16
// (K and V as the caller's fp16 copy of the layer), P is written to TMEM as
// fp16 and O is stored as fp16; both products then run with fp16 operands
// (kind::f16 takes one type for A and B).  P <= 2^8 and |O| <= max |V|, so
// neither can leave the fp16 range.
//
// TMEM columns: S0 [0,128)  S1 [128,256)  O0 [256,256+DH)  O1 [256+DH, 256+2DH)
#include "attn.cuh"

namespace cc {

namespace {

constexpr int BKV = 128;        // keys per tile
constexpr int KST = 2;          // K and V pipeline stages
constexpr int kThreads = 384;   // 3 warpgroups: softmax 0, softmax 1, producer/MMA
// Register split after launch (setmaxnreg): the block is launched with 168
// registers per thread (64512 in all); the producer/MMA warpgroup gives some
// up and the two softmax warpgroups take them (224 / 56: the split at which
// the kernel compiles without spills, the split-operand variant with the
// fewest); 2 * 128 * softmax + 128 * producer <= 384 * 168.
constexpr int kRegsLaunch = 168;
struct RegSplit {
  static constexpr int softmax = 224, producer = 56;
  static_assert(2 * 128 * softmax + 128 * producer <= kThreads * kRegsLaunch,
                "register split exceeds the launch allocation");
};



// 2^x by the PTX ex2.approx instruction (2 ulp; 2^-inf = 0).
CC_DEV float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}


template <int DH, bool SPLIT = false>
struct AttnSmem {
  static constexpr int NH = DH / 64;                 // 64-element (128-byte) column halves
  static constexpr int Q_BYTES = NH * 256 * 128;     // 256 rows
  static constexpr int KV_BYTES = NH * BKV * 128;    // one K (or V) tile (2-byte elements)
  // V stages: one when the second (lo) Q tile of SPLIT leaves no room for two
  static constexpr int KSTV = (SPLIT && DH == 128) ? 1 : KST;
  static constexpr int OFF_Q = 0;
  static constexpr int OFF_QLO = OFF_Q + Q_BYTES;          // SPLIT: the lo tile of Q
  static constexpr int OFF_K = OFF_QLO + (SPLIT ? Q_BYTES : 0);
  static constexpr int OFF_V = OFF_K + KST * KV_BYTES;
  static constexpr int OFF_BAR = OFF_V + KSTV * KV_BYTES;
  static constexpr int BYTES = OFF_BAR + 256 + 1024;   // barriers + alignment slack
  static_assert(BYTES <= 232448, "shared memory of a CTA exceeds 227 KB");
};

// e4m3 pair (low 16 bits) -> f16 pair, exact (the decode kernel's e4m3 cache).
CC_DEV uint32_t e4m3x2_to_f16x2(uint32_t two) {
  uint32_t r;
  asm("cvt.rn.f16x2.e4m3x2 %0, %1;" : "=r"(r) : "h"((unsigned short)(two & 0xFFFFu)));
  return r;
}

// Work unit `unit_id` -> (sequence b, KV head g, positions p0..p_last).
// Counter-causal rows run over [row_lo, row_hi) when a range is given (keys
// still up to the sequence end); a row's result does not depend on the range
// (the extra key tiles of a unit that starts lower are fully masked for it
// and add exact zeros).
// Unit order: streams (sequence, KV head) in groups of streams_per_group;
// within a group, position blocks outermost (longest units first), the
// group's streams innermost.  The group size bounds how far apart in time
// two resident units of one stream read the same K/V tile (chosen so the
// K/V read in between stays well inside L2).  q_lo: first query slot
// (causal mode).  valid is false for a bad length (reported) or a block past
// the sequence end.
struct UnitInfo {
  int b, g, n, q_lo, p0, p_last;
  bool bad, valid;
};
CC_DEV UnitInfo decode_unit(const AttnParams &p, int unit_id, bool causal) {
  UnitInfo u{};
  const int blocks_per_stream = (p.q_span + p.P - 1) / p.P;
  const int n_streams = p.batch * p.n_kv_heads;
  const int per_group = p.streams_per_group * blocks_per_stream;
  const int grp = unit_id / per_group;
  const int s0 = grp * p.streams_per_group;
  const int gsz = min(p.streams_per_group, n_streams - s0);
  const int r = unit_id - grp * per_group;
  const int pb = r / gsz;
  const int stream = s0 + (r - pb * gsz);
  u.b = stream / p.n_kv_heads;
  u.g = stream - u.b * p.n_kv_heads;
  u.n = p.seq_len[u.b];
  u.q_lo = (causal || p.row_lo) ? p.row_lo[u.b] : 0;
  // query rows end: the sequence end, or a counter-causal row range's end
  const int q_hi = (!causal && p.row_hi) ? p.row_hi[u.b] : u.n;
  u.bad = u.n < 0 || u.n > p.cap || u.q_lo < 0 || u.q_lo > q_hi || q_hi > u.n;
  u.p0 = u.q_lo + pb * p.P;
  u.valid = !u.bad && u.p0 < q_hi;
  u.p_last = min(u.p0 + p.P, q_hi) - 1;
  return u;
}

template <int DH, bool CAUSAL, bool SPLIT, bool F16>
__global__ void __launch_bounds__(kThreads, 1)
    attn_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                const __grid_constant__ CUtensorMap tmV, const __grid_constant__ AttnParams p) {
  using L = AttnSmem<DH, SPLIT>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                              ~uintptr_t(1023));
  uint64_t *bars = reinterpret_cast<uint64_t *>(smem + L::OFF_BAR);
  uint64_t *q_full = bars + 0;
  uint64_t *k_full = bars + 1;             // [KST]
  uint64_t *k_empty = k_full + KST;        // [KST]
  uint64_t *v_full = k_empty + KST;        // [KST]
  uint64_t *v_empty = v_full + KST;        // [KST]
  uint64_t *v_fixed = v_empty + KST;       // tail tile: V rows past n zeroed
  uint64_t *s_ready = v_fixed + 1;         // [2]
  uint64_t *p_ready = s_ready + 2;         // [2] (keys 0..63 of P when split)
  uint64_t *o_done = p_ready + 2;          // [2]
  uint64_t *turn = o_done + 2;             // [2] two issuers: issuer h may issue its next burst
  uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(turn + 2);
  volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.group, P = p.P;
  // Key splits (few units): the splits of a unit are consecutive CTAs.
  const int S = p.kv_splits > 1 ? p.kv_splits : 1;
  const int unit_id = blockIdx.x / S, split = blockIdx.x - unit_id * S;
  const UnitInfo u = decode_unit(p, unit_id, CAUSAL);
  if (u.bad) {
    if (threadIdx.x == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    return;
  }
  if (!u.valid) return;                      // the whole block lies past the sequence end
  const int b = u.b, g = u.g, n = u.n, p0 = u.p0, p_last = u.p_last;
  // counter-causal: key tiles holding slots p0+1 .. n-1; causal: slots 0 .. p_last
  const int t0 = CAUSAL ? 0 : (p0 + 1) / BKV;
  const int t1 = CAUSAL ? p_last / BKV : (n - 1) / BKV;
  const int ntiles_unit = t1 - t0 + 1;
  const size_t row_base = (size_t)b * p.cap;
  // this CTA's share of the unit's key tiles (all of them without splits):
  // local iteration `it` handles tile t_hi - it; the tail tile is t_top
  const int t_top = t1;
  const int it_off = S > 1 ? split * max(ntiles_unit, 0) / S : 0;
  const int ntiles = S > 1 ? (split + 1) * max(ntiles_unit, 0) / S - it_off : ntiles_unit;
  const int t_hi = t1 - it_off;
  const size_t part_slot = ((size_t)unit_id * S + split) * 256;
  // pool row of key tile t (paged) or b*cap + 128 t; a bad page reads zeros
  // (a coordinate past the maps) and is reported
  auto tile_row = [&](int t) -> int {
    if (p.pg.head_major) return 0;   // coordinates (slot, b*Hkv + g) instead
    const long long r = kv_row(p.pg, p.cap, b, t * BKV);
    if (r < 0) {
      set_status(p.status, CC_ERR_DEVICE_ARG);
      return p.kv_rows;
    }
    return (int)r;
  };

  if (S > 1 && ntiles <= 0) {   // nothing for this split: an empty partial
    for (int R = threadIdx.x; R < 256; R += blockDim.x)
      p.part_ml[part_slot + R] = make_float2(-INFINITY, 0.f);
    return;
  }
  if (ntiles <= 0) {   // no slot after the block: every row attends nothing -> 0
    for (int idx = threadIdx.x; idx < (p_last - p0 + 1) * G; idx += blockDim.x) {
      int pos = p0 + idx / G, hl = idx % G;
      __nv_bfloat16 *o = p.out + (row_base + pos) * p.out_ld + (size_t)(g * G + hl) * DH;
      for (int v = 0; v < DH / 8; ++v) reinterpret_cast<uint4 *>(o)[v] = make_uint4(0, 0, 0, 0);
      if (p.out_lo > 0)
        for (int v = 0; v < DH / 8; ++v)
          reinterpret_cast<uint4 *>(o + p.out_lo)[v] = make_uint4(0, 0, 0, 0);
    }
    return;
  }

  // The producer warp initialises the barriers and issues the Q load before
  // the CTA-wide barrier, so the load's latency overlaps the TMEM allocation
  // and the barrier.
  if (warp == 8 && lane == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < KST; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 2);   // one commit per MMA issuer
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 2);
    }
    mbar_init(v_fixed, 1);
    for (int h = 0; h < 2; ++h) {
      mbar_init(&turn[h], 1);
      mbar_init(&s_ready[h], 1);
      mbar_init(&p_ready[h], 128);
      mbar_init(&o_done[h], 1);
    }
    *abort_flag = 0;
    fence_barrier_init();
    tma_prefetch_desc(&tmQ);
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    mbar_arrive_expect_tx(q_full, (SPLIT ? 2 : 1) * L::NH * 128 * G * P);
    for (int hh = 0; hh < L::NH; ++hh)
      tma_load_3d(smem + L::OFF_Q + hh * 256 * 128, &tmQ, q_full, hh * 64, g * G,
                  (int)row_base + p0);
    if constexpr (SPLIT)   // lo heads follow the hi heads in each row
      for (int hh = 0; hh < L::NH; ++hh)
        tma_load_3d(smem + L::OFF_QLO + hh * 256 * 128, &tmQ, q_full, hh * 64,
                    p.n_q_heads + g * G, (int)row_base + p0);
  }
  // Rows P*G..255 of the Q tile exist when G does not divide 256: zero them
  // (the Q load does not write them) so their S rows are exact zeros (finite,
  // never NaN) and the softmax can treat every row of a tile alike (no
  // per-row mask path); visible to the tensor cores after the barrier below.
  if (warp == 8 && G * P < 256) {
    for (int qt = 0; qt < (SPLIT ? 2 : 1); ++qt)
      for (int hh = 0; hh < L::NH; ++hh)
        for (int idx = G * P * 8 + lane; idx < 256 * 8; idx += 32)
          reinterpret_cast<uint4 *>(smem + L::OFF_Q + qt * L::Q_BYTES + hh * 256 * 128)[idx] =
              make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
  }
  if (warp == 9) tmem_alloc(tmem_slot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  if (warp >= 8) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(RegSplit::producer));
    if (warp == 8) {
    // ------------------------------------------------------------ producer
    // (the Q tile was requested before the CTA-wide barrier)
    {
      for (int it = 0; it < ntiles; ++it) {
        const int t = t_hi - it, s = it % KST;   // key tiles from the sequence end downwards
        const uint32_t ph = (it / KST) & 1;
        const int sv = it % L::KSTV;             // V stage (one stage with SPLIT, head_dim 128)
        const uint32_t phv = (it / L::KSTV) & 1;
        const int krow = tile_row(t);
        // TMA coordinates after the head_dim one: (KV head, row), or head-major (slot, b*Hkv + g)
        const int kc1 = p.pg.head_major ? t * BKV : g;
        const int kc2 = p.pg.head_major ? b * p.n_kv_heads + g : krow;
        int ok = 1;
        if (lane == 0) {
          ok = mbar_wait(&k_empty[s], ph ^ 1, abort_flag, p.status);
          if (ok) {
            mbar_arrive_expect_tx(&k_full[s], L::KV_BYTES);
            for (int hh = 0; hh < L::NH; ++hh)
              tma_load_3d(smem + L::OFF_K + s * L::KV_BYTES + hh * BKV * 128, &tmK, &k_full[s],
                          hh * 64, kc1, kc2);
            ok = mbar_wait(&v_empty[sv], phv ^ 1, abort_flag, p.status);
          }
          if (ok) {
            mbar_arrive_expect_tx(&v_full[sv], L::KV_BYTES);
            for (int hh = 0; hh < L::NH; ++hh)
              tma_load_3d(smem + L::OFF_V + sv * L::KV_BYTES + hh * BKV * 128, &tmV, &v_full[sv],
                          hh * 64, kc1, kc2);
          }
        }
        ok = __shfl_sync(0xFFFFFFFFu, ok, 0);
        if (!ok) break;
        if (t == t_top && n - t * BKV < BKV) {
          // rows past the sequence end may hold any bits; P is 0 there, but
          // 0 * NaN would still poison O, so zero them before the PV product
          if (!mbar_wait(&v_full[sv], phv, abort_flag, p.status)) break;
          const int first = n - t * BKV;
          uint8_t *vs = smem + L::OFF_V + sv * L::KV_BYTES;
          for (int hh = 0; hh < L::NH; ++hh)
            for (int idx = first * 8 + lane; idx < BKV * 8; idx += 32)
              reinterpret_cast<uint4 *>(vs + hh * BKV * 128)[idx] = make_uint4(0, 0, 0, 0);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(v_fixed);
        }
      }
    }
    } else if (warp == 9 || warp == 10) {
    // ------------------------------------------------------------ MMA issuers
    // One issuing thread per M-half (warp 9: half 0, warp 10: half 1).  An
    // issuing thread blocks while the tensor pipe's short queue is full, so a
    // lone issuer leaves the pipe idle during its own barrier waits between
    // bursts.  Two issuers take turns: a burst is one half's products for
    // one key tile (PV(t, h) then QK(t+1, h)), bursts alternate half 0,
    // half 1, half 0, ... (so the halves' softmaxes stay out of phase and
    // each overlaps the other half's products), and each issuer does its own
    // waits (P ready, K/V tiles) while the other one's burst runs; only the
    // hand-over of the turn lies between bursts, covered by the products
    // still queued.  Each half's products stay in one thread's program order
    // (PV(t) before QK(t+1): P lives in S's columns), so every result is
    // deterministic.
    if (lane == 0) {
      const int h_lo = warp - 9, h_hi = warp - 9;   // this issuer's M-half
      // every operand bf16 (fp16 with F16)
      constexpr uint32_t idesc_qk = F16 ? make_idesc_f16(128, BKV, 0, 0) : make_idesc_bf16(128, BKV, 0, 0);
      constexpr uint32_t idesc_pv = F16 ? make_idesc_f16(128, DH, 0, 1) : make_idesc_bf16(128, DH, 0, 1);
      // Shared-memory descriptors built once; a K step only advances the
      // start-address field (16-byte units): +2 per 16 columns of a 128-byte
      // row (Q, K), +128 per 16 keys of V.
      constexpr int NQ = SPLIT ? 2 : 1;   // Q tiles: hi (and lo)
      uint64_t qd[NQ][2][L::NH], kd[KST][L::NH], vd[L::KSTV];
#pragma unroll
      for (int qt = 0; qt < NQ; ++qt)
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int hh = 0; hh < L::NH; ++hh)
            qd[qt][h][hh] = make_sdesc_sw128(smem_u32(smem + L::OFF_Q + qt * L::Q_BYTES) +
                                                 hh * 256 * 128 + h * 128 * 128,
                                             16, 1024);
#pragma unroll
      for (int st = 0; st < KST; ++st)
#pragma unroll
        for (int hh = 0; hh < L::NH; ++hh)
          kd[st][hh] = make_sdesc_sw128(smem_u32(smem + L::OFF_K + st * L::KV_BYTES) + hh * BKV * 128,
                                        16, 1024);
#pragma unroll
      for (int st = 0; st < L::KSTV; ++st)
        vd[st] = make_sdesc_sw128(smem_u32(smem + L::OFF_V + st * L::KV_BYTES), BKV * 128, 1024);
      // pass_at >= 0: hand the turn over once that many products of the
      // burst remain to be issued (the other issuer's wake-up then overlaps
      // the products still queued)
      auto issue_qk = [&](int it, int h, auto &&pass, int pass_at) {
        const int st = it % KST;
        constexpr int kN = NQ * (DH / 16);
#pragma unroll
        for (int qt = 0; qt < NQ; ++qt)   // SPLIT: S = Q_hi K^T + Q_lo K^T
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            const int hh = kk >> 2, ko = (kk & 3) * 2;
            if (kN - (qt * (DH / 16) + kk) == pass_at) pass();
            umma_ss(tmem + h * 128, qd[qt][h][hh] + ko, kd[st][hh] + ko, idesc_qk,
                    (qt > 0 || kk > 0) ? 1u : 0u);
          }
      };
      constexpr int kPassAt = 2;   // products left in a burst when the turn is handed over (1-3 measured alike; 6 and 8 slower)
      // turns: this issuer's burst kb follows the other issuer's previous
      // burst (half 0 opens; half 1's burst kb follows half 0's burst kb)
      int kb = 0;
      auto take_turn = [&]() -> bool {
        if (h_lo == 0) return kb == 0 || mbar_wait(&turn[0], (kb - 1) & 1, abort_flag, p.status);
        return mbar_wait(&turn[1], kb & 1, abort_flag, p.status);
      };
      auto pass_turn = [&]() {
        mbar_arrive(&turn[1 - h_lo]);
        ++kb;
      };
      bool ok = mbar_wait(q_full, 0, abort_flag, p.status);
      if (ok) ok = mbar_wait(&k_full[0], 0, abort_flag, p.status);
      if (ok) ok = take_turn();
      if (ok) {
        tc_fence_after();
        for (int h = h_lo; h <= h_hi; ++h) {
          issue_qk(0, h, pass_turn, h == h_hi ? kPassAt : -1);
          umma_commit(&s_ready[h]);
        }
        umma_commit(&k_empty[0]);   // one arrival per issuer
      }
      for (int it = 0; ok && it < ntiles; ++it) {
        const int t = t_hi - it, s = it % L::KSTV;   // V stage
        const uint32_t ph = (it / L::KSTV) & 1;
        if (!(ok = mbar_wait(&v_full[s], ph, abort_flag, p.status))) break;
        if (t == t_top && n - t * BKV < BKV)
          if (!(ok = mbar_wait(v_fixed, 0, abort_flag, p.status))) break;
        for (int h = h_lo; h <= h_hi; ++h) {
          if (!(ok = mbar_wait(&p_ready[h], it & 1, abort_flag, p.status))) break;
          const int s2 = (it + 1) % KST;   // the next key tile's stage
          if (it + 1 < ntiles && h == h_lo)   // waited before the burst, not inside it
            if (!(ok = mbar_wait(&k_full[s2], ((it + 1) / KST) & 1, abort_flag, p.status))) break;
          if (!(ok = take_turn())) break;
          tc_fence_after();
#pragma unroll
          for (int pt = 0; pt < NQ; ++pt)   // SPLIT: O += P_hi V + P_lo V
#pragma unroll
            for (int kk = 0; kk < BKV / 16; ++kk) {
              // B = V tile, MN-major: 64-column halves 16 KB apart (LBO),
              // 8-key groups 1024 B apart (SBO); A = P_h, bf16 pairs in TMEM
              // (P_lo 64 columns after P_hi).
              umma_ts(tmem + 256 + h * DH, tmem + h * 128 + pt * 64 + kk * 8, vd[s] + kk * 128,
                      idesc_pv, (it > 0 || kk > 0 || pt > 0) ? 1u : 0u);
            }
          if (h == h_hi) umma_commit(&v_empty[s]);   // one arrival per issuer
          if (it + 1 < ntiles) {
            issue_qk(it + 1, h, pass_turn, kPassAt);
            umma_commit(&s_ready[h]);
            if (h == h_hi) umma_commit(&k_empty[s2]);
          } else {
            umma_commit(&o_done[h]);
            pass_turn();
          }
        }
      }
    }
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(RegSplit::softmax));
    // ------------------------------------------------------------ softmax
    const int h = warp >> 2, q = warp & 3;
    const int R = h * 128 + q * 32 + lane;              // unit row
    const bool row_used = R < P * G;
    const int pos = row_used ? p0 + R / G : 0x7FFFFFFF; // slot index of this row
    const int hl = row_used ? R % G : 0;
    const uint32_t lane_off = uint32_t(q * 32) << 16;
    const uint32_t s_t = tmem + lane_off + h * 128;
    const uint32_t o_t = tmem + lane_off + 256 + h * DH;
    const float sl2 = p.scale_log2;
    const float thr = 8.0f / sl2;   // lazy-rescale threshold: 2^8 in exp2 space, in raw units
    const float2 sl2v = make_float2(sl2, sl2);
    float m_used = -INFINITY, l = 0.f;   // m_used: reference max of the raw scores
    bool ok = true;
    for (int it = 0; it < ntiles; ++it) {
      const int j0 = (t_hi - it) * BKV;
      if (!(ok = mbar_wait(&s_ready[h], it & 1, abort_flag, p.status))) break;
      tc_fence_after();
      uint32_t sr[128];
      tmem_ld32(s_t + 0, *reinterpret_cast<uint32_t(*)[32]>(&sr[0]));
      tmem_ld32(s_t + 32, *reinterpret_cast<uint32_t(*)[32]>(&sr[32]));
      tmem_ld32(s_t + 64, *reinterpret_cast<uint32_t(*)[32]>(&sr[64]));
      tmem_ld32(s_t + 96, *reinterpret_cast<uint32_t(*)[32]>(&sr[96]));
      tmem_ld_wait();
      // row max with 8 independent partial maxima (a short dependency chain)
      float mp[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) mp[u] = -INFINITY;
      // uniform over the CTA: rows past P*G have zero queries and need no mask
      const bool need_mask = CAUSAL ? (j0 + BKV - 1 > p0) : ((j0 <= p0 + P - 1) || (j0 + BKV > n));
      if (need_mask) {
        // counter-causal: key j kept iff pos < j < n; causal: iff j <= min(pos, n - 1)
        const int lo = CAUSAL ? -1 : pos - j0;                    // keep c > lo
        const int hi = CAUSAL ? min(pos, n - 1) - j0 + 1 : n - j0;   // keep c < hi
#pragma unroll
        for (int c = 0; c < 128; ++c) {
          float x = (c > lo && c < hi) ? __uint_as_float(sr[c]) : -INFINITY;
          sr[c] = __float_as_uint(x);
          mp[c & 7] = fmaxf(mp[c & 7], x);
        }
      } else {
#pragma unroll
        for (int c = 0; c < 128; ++c) mp[c & 7] = fmaxf(mp[c & 7], __uint_as_float(sr[c]));
      }
      const float mt = fmaxf(fmaxf(fmaxf(mp[0], mp[1]), fmaxf(mp[2], mp[3])),
                             fmaxf(fmaxf(mp[4], mp[5]), fmaxf(mp[6], mp[7])));
      // lazy rescaling: move the reference max only when it grows by more
      // than 2^8 in exp2 space, so p <= 256 and O is rarely touched
      const float m_new = fmaxf(m_used, mt);
      const bool bump = m_new > m_used + thr;          // also true for -inf -> finite
      const bool rescale_o = bump && it > 0 && l > 0.f;
      float factor = 1.f;
      if (bump) {
        factor = fast_exp2((m_used - m_new) * sl2);   // 0 when m_used = -inf
        l *= factor;
        m_used = m_new;
      }
      // O still holds the previous tiles' sum (S_ready implies the last PV is
      // done); it must be rescaled before any PV of this tile accumulates.
      auto rescale = [&]() {
        if (__any_sync(0xFFFFFFFFu, rescale_o)) {
          const float f = rescale_o ? factor : 1.f;
#pragma unroll 1
          for (int c = 0; c < DH; c += 32) {
            uint32_t o[32];
            tmem_ld32(o_t + c, o);
            tmem_ld_wait();
#pragma unroll
            for (int k = 0; k < 32; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * f);
            tmem_st32(o_t + c, o);
          }
        }
      };
      // p = 2^(s*sl2 - m*sl2): one packed FMA per pair, bf16 P into TMEM over S,
      // the row sum l in fp32
      const float nm = (m_used == -INFINITY) ? 0.f : -m_used * sl2;
      const float2 nmv = make_float2(nm, nm);
      float2 lsum = make_float2(0.f, 0.f);
#pragma unroll
      for (int c0 = 0; c0 < 128; c0 += 32) {
        uint32_t pk[16];
        [[maybe_unused]] uint32_t pl[16];
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          const float2 y = __ffma2_rn(make_float2(__uint_as_float(sr[c0 + k]),
                                                  __uint_as_float(sr[c0 + k + 1])), sl2v, nmv);
          const float2 e = make_float2(fast_exp2(y.x), fast_exp2(y.y));
          pk[k / 2] = F16 ? pack_f16x2(e.x, e.y) : pack_bf16x2(e.x, e.y);
          if constexpr (SPLIT)   // P_lo = bf16(p - P_hi)
            pl[k / 2] = pack_bf16x2(e.x - bf16_lo(pk[k / 2]), e.y - bf16_hi(pk[k / 2]));
          lsum = __fadd2_rn(lsum, e);
        }
        tmem_st16(s_t + c0 / 2, pk);
        if constexpr (SPLIT) tmem_st16(s_t + 64 + c0 / 2, pl);
      }
      l += lsum.x + lsum.y;
      rescale();   // after P is written: S registers free for the O rows
      tmem_st_wait();
      tc_fence_before();
      mbar_arrive(&p_ready[h]);
    }
    // ---- epilogue: O / l -> bf16 -> out[row_base + pos][g*G + hl][:]
    if (ok) ok = mbar_wait(&o_done[h], 0, abort_flag, p.status);
    if (ok && S > 1) {   // key split: this CTA's unnormalised O and (max, sum) per row
      tc_fence_after();
      float *po = p.part_o + (part_slot + R) * DH;
#pragma unroll 1
      for (int c = 0; c < DH; c += 32) {
        uint32_t o[32];
        tmem_ld32(o_t + c, o);
        tmem_ld_wait();
#pragma unroll
        for (int v = 0; v < 8; ++v)
          reinterpret_cast<float4 *>(po + c)[v] =
              make_float4(__uint_as_float(o[v * 4]), __uint_as_float(o[v * 4 + 1]),
                          __uint_as_float(o[v * 4 + 2]), __uint_as_float(o[v * 4 + 3]));
      }
      p.part_ml[part_slot + R] = make_float2(m_used, l);
    } else if (ok) {
      tc_fence_after();
      const bool store = row_used && pos <= p_last;
      const float inv = l > 0.f ? p.v_scale / l : 0.f;   // V scale: e4m3 cache (else 1)
      __nv_bfloat16 *dst =
          p.out + (row_base + (store ? pos : 0)) * p.out_ld + (size_t)(g * G + hl) * DH;
#pragma unroll 1
      for (int c = 0; c < DH; c += 32) {
        uint32_t o[32];
        tmem_ld32(o_t + c, o);
        tmem_ld_wait();
        uint32_t pk[16];
#pragma unroll
        for (int k = 0; k < 32; k += 2)
          pk[k / 2] = F16 ? pack_f16x2(__uint_as_float(o[k]) * inv, __uint_as_float(o[k + 1]) * inv)
                          : pack_bf16x2(__uint_as_float(o[k]) * inv, __uint_as_float(o[k + 1]) * inv);
        if (store) {
          uint4 *d = reinterpret_cast<uint4 *>(dst + c);
#pragma unroll
          for (int v = 0; v < 4; ++v) d[v] = make_uint4(pk[v * 4], pk[v * 4 + 1], pk[v * 4 + 2], pk[v * 4 + 3]);
          if (p.out_lo > 0) {   // lo = bf16(o - hi)
            uint32_t lo[16];
#pragma unroll
            for (int k = 0; k < 32; k += 2)
              lo[k / 2] = pack_bf16x2(__uint_as_float(o[k]) * inv - bf16_lo(pk[k / 2]),
                                      __uint_as_float(o[k + 1]) * inv - bf16_hi(pk[k / 2]));
            uint4 *dl = reinterpret_cast<uint4 *>(dst + p.out_lo + c);
#pragma unroll
            for (int v = 0; v < 4; ++v)
              dl[v] = make_uint4(lo[v * 4], lo[v * 4 + 1], lo[v * 4 + 2], lo[v * 4 + 3]);
          }
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) __nanosleep(1000000);   // let copies still in flight land
  if (warp == 9) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// Key splits: out = sum_s 2^((m_s - m*) c) O_s / sum_s 2^((m_s - m*) c) l_s
// per row (m* the largest reference max, c = log2(e)/sqrt(dh)), splits in
// order; bf16 (and lo) stores as the kernel's own epilogue.  Block = one row
// of one unit, a thread per head_dim element: the splits' (max, sum) pairs
// are loaded in parallel and weighted once in shared memory, then every
// thread sums its element over the splits with eight loads in flight.
constexpr int kCombineMaxSplits = 256;

template <bool CAUSAL>
__global__ void attn_combine_kernel(const __grid_constant__ AttnParams p) {
  __shared__ float wgt[kCombineMaxSplits];
  __shared__ float lsum[kCombineMaxSplits];
  __shared__ float red[4];
  pdl_trigger();
  pdl_wait();
  const int R = blockIdx.x, unit_id = blockIdx.y, d = threadIdx.x;
  const UnitInfo u = decode_unit(p, unit_id, CAUSAL);
  const int G = p.group;
  if (!u.valid || R >= p.P * G) return;
  const int pos = u.p0 + R / G, hl = R % G;
  if (pos > u.p_last) return;
  const int S = p.kv_splits;
  const float c = p.scale_log2;
  const size_t base = (size_t)unit_id * S * 256 + R;   // split s's row: base + s * 256
  // reference max over the splits that saw keys
  float m = -INFINITY;
  for (int s = d; s < S; s += blockDim.x) {
    const float2 ml = p.part_ml[base + (size_t)s * 256];
    wgt[s] = ml.x;
    lsum[s] = ml.y;
    if (ml.y > 0.f) m = fmaxf(m, ml.x);
  }
  m = warp_max(m);
  if ((d & 31) == 0) red[d >> 5] = m;
  __syncthreads();
  m = red[0];
  for (int w = 1; w < (int)(blockDim.x >> 5); ++w) m = fmaxf(m, red[w]);
  for (int s = d; s < S; s += blockDim.x)
    wgt[s] = lsum[s] > 0.f ? exp2f((wgt[s] - m) * c) : 0.f;
  __syncthreads();
  float l = 0.f;
  for (int s = 0; s < S; ++s) l += wgt[s] * lsum[s];
  float o = 0.f;
  int s = 0;
  for (; s + 8 <= S; s += 8) {
    float v[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) v[k] = p.part_o[(base + (size_t)(s + k) * 256) * p.head_dim + d];
#pragma unroll
    for (int k = 0; k < 8; ++k) o += wgt[s + k] * v[k];
  }
  for (; s < S; ++s) o += wgt[s] * p.part_o[(base + (size_t)s * 256) * p.head_dim + d];
  const float v = l > 0.f ? o * p.v_scale / l : 0.f;
  __nv_bfloat16 *dst = p.out + ((size_t)u.b * p.cap + pos) * p.out_ld +
                       (size_t)(u.g * G + hl) * p.head_dim + d;
  if (p.f16) {   // fp16 operand mode: O as fp16 (the same 2 bytes)
    const __half hf = __float2half_rn(v);
    *dst = *reinterpret_cast<const __nv_bfloat16 *>(&hf);
    return;
  }
  const __nv_bfloat16 hi = __float2bfloat16_rn(v);
  *dst = hi;
  if (p.out_lo > 0) dst[p.out_lo] = __float2bfloat16_rn(v - __bfloat162float(hi));
}

template <int DH, bool CAUSAL, bool SPLIT = false, bool F16 = false>
cudaError_t launch_dh(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v,
                      const AttnParams &p, cudaStream_t stream) {
  using L = AttnSmem<DH, SPLIT>;
  auto kern = attn_kernel<DH, CAUSAL, SPLIT, F16>;
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         L::BYTES);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  const long long units = attn_units(p);
  if (units <= 0) return cudaSuccess;
  // Resident units of one stream start about T / (SMs / streams) apart (T a
  // unit's run time), so between two reads of a K/V tile the resident units
  // read about streams^2 * cap * (K+V bytes per slot) / SMs bytes.  Pick the
  // largest stream group keeping that under kReuseBytes.  The bound is set
  // from timings, far below the L2 size: Llama-3-8B at 8k slots and Qwen2.5
  // at 32k slots run fastest with all streams in one group (their K/V fit in
  // L2 whatever the order), four 32k Llama sequences and a 131k Qwen sequence
  // with groups of a few streams.
  static int sms[64] = {};
  if (dev < 64 && !sms[dev]) cudaDeviceGetAttribute(&sms[dev], cudaDevAttrMultiProcessorCount, dev);
  const double kReuseBytes = 2.0 * (1 << 20);
  const double per_stream2 = (double)p.cap * 4.0 * DH / (dev < 64 && sms[dev] ? sms[dev] : 148);
  const int n_streams = p.batch * p.n_kv_heads;
  AttnParams pp = p;
  pp.streams_per_group = (int)fmax(1.0, fmin((double)n_streams, floor(sqrt(kReuseBytes / per_stream2))));
  const int S = pp.kv_splits > 1 ? pp.kv_splits : 1;
  if (S > 1 && (!pp.part_o || !pp.part_ml)) return cudaErrorInvalidValue;
  kern<<<(unsigned)(units * S), kThreads, L::BYTES, stream>>>(q, k, v, pp);
  if (S > 1) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    attn_combine_kernel<CAUSAL><<<dim3(256, (unsigned)units), DH, 0, stream>>>(pp);
  }
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Decode attention: one query row per sequence (q_span == 1), at most
// kDecMaxG query heads per KV head.  For a single query row the products are
// a few hundred FMAs per key, so CUDA cores in fp32 suffice and the K/V bytes
// bound the time: CTA = (unit, key split); chunks of 128 keys are copied to
// shared memory with cp.async (double-buffered; K rows padded by 16 bytes so
// the score pass's column reads are conflict-free); per chunk the scores, an
// online softmax (log2 domain, reference max in raw units as the tile kernel
// keeps it) and P V; each CTA writes the partial (O, max, sum) rows that
// attn_combine_kernel merges.
// ---------------------------------------------------------------------------
constexpr int kDecChunk = 128;
constexpr int kDecThreads = 256;   // = 2 * kDecChunk: the score pass takes a key and half its dims

// K rows padded so the score pass's column reads are conflict-free: bf16
// rows +16 bytes (16-byte reads), e4m3 rows +8 bytes (8-byte reads).
template <int DH, bool FP8>
struct DecSmem {
  static constexpr int EB = FP8 ? 1 : 2;   // bytes per cached element
  static constexpr int K_ROW = DH * EB + (FP8 ? 8 : 16);
  static constexpr int V_ROW = DH * EB;
  static constexpr int K_BYTES = kDecChunk * K_ROW;
  static constexpr int V_BYTES = kDecChunk * V_ROW;
  static constexpr int BUF = K_BYTES + V_BYTES;
  static constexpr int OFF_Q = 2 * BUF;                                 // fp32 [G][DH]
  static constexpr int OFF_S = OFF_Q + kDecMaxG * DH * 4;               // fp32 [2][G][chunk]
  static constexpr int OFF_P = OFF_S + 2 * kDecMaxG * kDecChunk * 4;    // fp32 [G][chunk]
  static constexpr int OFF_F = OFF_P + kDecMaxG * kDecChunk * 4;        // fp32 [G]
  static constexpr int BYTES = OFF_F + kDecMaxG * 4;
};

CC_DEV void cp_async16(void *dst, const void *src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}
CC_DEV void cp_async8(void *dst, const void *src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(smem_u32(dst)), "l"(src)
               : "memory");
}
CC_DEV void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }

// 8 cached elements -> float: bf16 (16 bytes) or e4m3 codes (8 bytes, via f16)
template <bool FP8>
CC_DEV void load8_kv(const uint8_t *src, float *f) {
  if constexpr (FP8) {
    const uint2 x = *reinterpret_cast<const uint2 *>(src);
    const uint32_t h[4] = {e4m3x2_to_f16x2(x.x), e4m3x2_to_f16x2(x.x >> 16),
                           e4m3x2_to_f16x2(x.y), e4m3x2_to_f16x2(x.y >> 16)};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&h[i]));
      f[2 * i] = v.x;
      f[2 * i + 1] = v.y;
    }
  } else {
    const uint4 x = *reinterpret_cast<const uint4 *>(src);
    f[0] = bf16_lo(x.x); f[1] = bf16_hi(x.x); f[2] = bf16_lo(x.y); f[3] = bf16_hi(x.y);
    f[4] = bf16_lo(x.z); f[5] = bf16_hi(x.z); f[6] = bf16_lo(x.w); f[7] = bf16_hi(x.w);
  }
}
template <int N>
CC_DEV void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

template <int DH, bool FP8>
__global__ void __launch_bounds__(kDecThreads) attn_decode_kernel(const __grid_constant__ AttnParams p) {
  using L = DecSmem<DH, FP8>;
  extern __shared__ __align__(128) uint8_t smem[];
  pdl_trigger();   // the combine may launch (it waits for this grid before reading)
  pdl_wait();      // q and the new token's K/V come from the projection just before
  const int S = p.kv_splits;
  const int unit_id = blockIdx.x / S, split = blockIdx.x - unit_id * S;
  const UnitInfo u = decode_unit(p, unit_id, true);
  if (u.bad) {
    if (threadIdx.x == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    return;
  }
  if (!u.valid) return;
  const int G = p.group, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int pos = u.p0;            // the unit's one query slot
  const int n_keys = pos + 1;      // causal: keys 0 .. pos
  const int nch = (n_keys + kDecChunk - 1) / kDecChunk;
  const int c_lo = split * nch / S, c_hi = (split + 1) * nch / S;
  const size_t slot = ((size_t)unit_id * S + split) * 256;
  if (c_lo >= c_hi) {   // nothing for this split: an empty partial
    if (tid < G) p.part_ml[slot + tid] = make_float2(-INFINITY, 0.f);
    return;
  }
  float *qs = reinterpret_cast<float *>(smem + L::OFF_Q);
  float *sbuf = reinterpret_cast<float *>(smem + L::OFF_S);
  float *pbuf = reinterpret_cast<float *>(smem + L::OFF_P);
  float *fbuf = reinterpret_cast<float *>(smem + L::OFF_F);
  const size_t row_base = (size_t)u.b * p.cap;
  const int Hkv = p.n_kv_heads;

  const uint8_t *kg = reinterpret_cast<const uint8_t *>(p.k);
  const uint8_t *vg = reinterpret_cast<const uint8_t *>(p.v);
  auto issue = [&](int c, int buf) {
    uint8_t *kb = smem + buf * L::BUF, *vb = kb + L::K_BYTES;
    // K in DH/8 pieces per row (16 bytes bf16, 8 bytes e4m3), V in 16-byte pieces
    constexpr int KP = DH / 8, KPB = 8 * L::EB, VP = DH * L::EB / 16;
    // vector index of the chunk's first key (a chunk lies in one page; head-major:
    // consecutive slots are consecutive vectors, else Hkv apart); -1: bad page
    const long long cbase = kv_vec(p.pg, p.cap, u.b, u.g, c * kDecChunk);
    const int vstep = p.pg.head_major ? 1 : Hkv;
    if (cbase < 0 && tid == 0) set_status(p.status, CC_ERR_DEVICE_ARG);
    for (int i = tid; i < kDecChunk * KP; i += kDecThreads) {
      const int r = i / KP, e = i - r * KP;
      const int j = c * kDecChunk + r;
      uint8_t *kd = kb + r * L::K_ROW + e * KPB;
      if (j < n_keys && cbase >= 0) {
        const uint8_t *src = kg + ((size_t)(cbase + (long long)r * vstep) * DH) * L::EB + e * KPB;
        if constexpr (FP8) cp_async8(kd, src);
        else cp_async16(kd, src);
      } else if constexpr (FP8) {
        *reinterpret_cast<uint2 *>(kd) = make_uint2(0, 0);
      } else {
        *reinterpret_cast<uint4 *>(kd) = make_uint4(0, 0, 0, 0);
      }
    }
    for (int i = tid; i < kDecChunk * VP; i += kDecThreads) {
      const int r = i / VP, e = i - r * VP;
      const int j = c * kDecChunk + r;
      uint8_t *vd = vb + r * L::V_ROW + e * 16;
      if (j < n_keys && cbase >= 0)   // past the last key: zeros (P is 0 there, V must be finite)
        cp_async16(vd, vg + ((size_t)(cbase + (long long)r * vstep) * DH) * L::EB + e * 16);
      else
        *reinterpret_cast<uint4 *>(vd) = make_uint4(0, 0, 0, 0);
    }
    cp_async_commit();
  };
  issue(c_lo, 0);
  for (int i = tid; i < G * DH; i += kDecThreads) {
    const int h = i / DH, d = i - h * DH;
    qs[i] = __bfloat162float(
        p.q[(row_base + pos) * (size_t)p.n_q_heads * DH + (size_t)(u.g * G + h) * DH + d]);
  }

  constexpr int DPT = DH / 32;   // P V: warp h < G owns head h, lane the dims lane*DPT..
  float m_h = -INFINITY, l_h = 0.f;
  float o[DPT];
#pragma unroll
  for (int i = 0; i < DPT; ++i) o[i] = 0.f;
  const float c2 = p.scale_log2;
  for (int c = c_lo; c < c_hi; ++c) {
    const int buf = (c - c_lo) & 1;
    if (c + 1 < c_hi) {
      issue(c + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint8_t *kb = smem + buf * L::BUF, *vb = kb + L::K_BYTES;
    {   // scores: thread = (key j, half of the dims)
      const int j = tid & (kDecChunk - 1), half = tid / kDecChunk;
      const uint8_t *kr = kb + j * L::K_ROW + half * (DH / 2) * L::EB;
      float sc[kDecMaxG];
#pragma unroll
      for (int h = 0; h < kDecMaxG; ++h) sc[h] = 0.f;
#pragma unroll
      for (int d8 = 0; d8 < DH / 16; ++d8) {
        float kf[8];
        load8_kv<FP8>(kr + d8 * 8 * L::EB, kf);
        const int d0 = half * (DH / 2) + d8 * 8;
#pragma unroll
        for (int h = 0; h < kDecMaxG; ++h) {
          if (h < G) {
            const float4 qa = *reinterpret_cast<const float4 *>(qs + h * DH + d0);
            const float4 qb = *reinterpret_cast<const float4 *>(qs + h * DH + d0 + 4);
            float a = sc[h];
            a = fmaf(kf[0], qa.x, a); a = fmaf(kf[1], qa.y, a);
            a = fmaf(kf[2], qa.z, a); a = fmaf(kf[3], qa.w, a);
            a = fmaf(kf[4], qb.x, a); a = fmaf(kf[5], qb.y, a);
            a = fmaf(kf[6], qb.z, a); a = fmaf(kf[7], qb.w, a);
            sc[h] = a;
          }
        }
      }
#pragma unroll
      for (int h = 0; h < kDecMaxG; ++h)
        if (h < G) sbuf[(half * kDecMaxG + h) * kDecChunk + j] = sc[h];
    }
    __syncthreads();
    if (warp < G) {   // online softmax of head h = warp over the chunk
      const int h = warp;
      float sv[kDecChunk / 32];
      float cm = -INFINITY;
#pragma unroll
      for (int q = 0; q < kDecChunk / 32; ++q) {
        const int j = lane + 32 * q;
        float v = sbuf[h * kDecChunk + j] + sbuf[(kDecMaxG + h) * kDecChunk + j];
        if (c * kDecChunk + j >= n_keys) v = -INFINITY;
        sv[q] = v;
        cm = fmaxf(cm, v);
      }
      cm = warp_max(cm);
      const float m_new = fmaxf(m_h, cm);
      const bool any = m_new != -INFINITY;
      const float factor = any ? fast_exp2((m_h - m_new) * c2) : 1.f;   // 0 when m_h = -inf
      float ls = 0.f;
#pragma unroll
      for (int q = 0; q < kDecChunk / 32; ++q) {
        const float pv = any ? fast_exp2((sv[q] - m_new) * c2) : 0.f;
        pbuf[h * kDecChunk + lane + 32 * q] = pv;
        ls += pv;
      }
      ls = warp_sum(ls);
      l_h = l_h * factor + ls;
      m_h = m_new;
      if (lane == 0) fbuf[h] = factor;
    }
    __syncthreads();
    if (warp < G) {   // O = O * factor + P V
      const int h = warp;
      const float f = fbuf[h];
#pragma unroll
      for (int i = 0; i < DPT; ++i) o[i] *= f;
      const float *ph = pbuf + h * kDecChunk;
#pragma unroll 4
      for (int j = 0; j < kDecChunk; ++j) {
        const float pj = ph[j];
        const uint8_t *vr = vb + j * L::V_ROW + lane * DPT * L::EB;
        if constexpr (FP8) {
#pragma unroll
          for (int i = 0; i < DPT; i += 2) {
            const uint32_t hv = e4m3x2_to_f16x2(*reinterpret_cast<const uint16_t *>(vr + i));
            const float2 v = __half22float2(*reinterpret_cast<const __half2 *>(&hv));
            o[i] = fmaf(pj, v.x, o[i]);
            o[i + 1] = fmaf(pj, v.y, o[i + 1]);
          }
        } else if constexpr (DPT == 4) {
          const uint2 v = *reinterpret_cast<const uint2 *>(vr);
          o[0] = fmaf(pj, bf16_lo(v.x), o[0]);
          o[1] = fmaf(pj, bf16_hi(v.x), o[1]);
          o[2] = fmaf(pj, bf16_lo(v.y), o[2]);
          o[3] = fmaf(pj, bf16_hi(v.y), o[3]);
        } else {
          const uint32_t v = *reinterpret_cast<const uint32_t *>(vr);
          o[0] = fmaf(pj, bf16_lo(v), o[0]);
          o[1] = fmaf(pj, bf16_hi(v), o[1]);
        }
      }
    }
    __syncthreads();
  }
  if (warp < G) {   // partial row R = head warp of the unit's one position
    float *po = p.part_o + (slot + warp) * DH + lane * DPT;
#pragma unroll
    for (int i = 0; i < DPT; ++i) po[i] = o[i];
    if (lane == 0) p.part_ml[slot + warp] = make_float2(m_h, l_h);
  }
}

template <int DH, bool FP8>
cudaError_t launch_decode_dh(const AttnParams &p, cudaStream_t stream) {
  static bool attr_set[64] = {};
  int dev = 0;
  cudaGetDevice(&dev);
  if (dev < 64 && !attr_set[dev]) {
    cudaError_t e = cudaFuncSetAttribute(attn_decode_kernel<DH, FP8>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         DecSmem<DH, FP8>::BYTES);
    if (e != cudaSuccess) return e;
    attr_set[dev] = true;
  }
  const long long units = attn_units(p);
  if (units <= 0) return cudaSuccess;
  AttnParams pp = p;
  pp.streams_per_group = p.batch * p.n_kv_heads;
  cudaError_t e = launch_pdl(attn_decode_kernel<DH, FP8>, dim3((unsigned)(units * pp.kv_splits)),
                             dim3(kDecThreads), DecSmem<DH, FP8>::BYTES, stream, pp);
  if (e != cudaSuccess) return e;
  return launch_pdl(attn_combine_kernel<true>, dim3((unsigned)p.group, (unsigned)units), dim3(DH),
                    0, stream, pp);
}

}  // namespace

int attn_positions_per_unit(int group) { return 256 / group; }

long long attn_units(const AttnParams &p) {
  return (long long)p.batch * p.n_kv_heads * ((p.q_span + p.P - 1) / p.P);
}


cudaError_t launch_attention_decode(const AttnParams &p, cudaStream_t stream) {
  if (!p.causal || p.q_span != 1 || p.group > kDecMaxG || p.kv_splits < 1 || !p.q || !p.k ||
      !p.v || !p.part_o || !p.part_ml)
    return cudaErrorInvalidValue;
  const bool f8 = p.kv_fp8 != 0;
  if (p.head_dim == 128)
    return f8 ? launch_decode_dh<128, true>(p, stream) : launch_decode_dh<128, false>(p, stream);
  if (p.head_dim == 64)
    return f8 ? launch_decode_dh<64, true>(p, stream) : launch_decode_dh<64, false>(p, stream);
  return cudaErrorInvalidValue;
}

cudaError_t launch_attention(const CUtensorMap &q, const CUtensorMap &k, const CUtensorMap &v,
                             const AttnParams &p, cudaStream_t stream) {
  // an e4m3 cache reaches the tile kernel as a bf16 (or fp16) copy (the caller's)
  if (p.kv_fp8) return cudaErrorInvalidValue;
  if (p.f16) {   // the fp16 operand scoring pass: counter-causal, single operands
    if (p.causal || p.q_split || p.out_lo > 0) return cudaErrorInvalidValue;
    if (p.head_dim == 128) return launch_dh<128, false, false, true>(q, k, v, p, stream);
    if (p.head_dim == 64) return launch_dh<64, false, false, true>(q, k, v, p, stream);
    return cudaErrorInvalidValue;
  }
  if (p.causal) {
    if (p.head_dim == 128) return launch_dh<128, true>(q, k, v, p, stream);
    if (p.head_dim == 64) return launch_dh<64, true>(q, k, v, p, stream);
  } else if (p.q_split) {   // the precise scoring pass
    if (p.head_dim == 128) return launch_dh<128, false, true>(q, k, v, p, stream);
    if (p.head_dim == 64) return launch_dh<64, false, true>(q, k, v, p, stream);
  } else {
    if (p.head_dim == 128) return launch_dh<128, false>(q, k, v, p, stream);
    if (p.head_dim == 64) return launch_dh<64, false>(q, k, v, p, stream);
  }
  return cudaErrorInvalidValue;
}

}  // namespace cc
