// Support checks of the tensor-core (tcgen05) path for bf16 inputs, and the
// chunking of the RACE key kernel. Every bf16 shape these accept runs the
// persistent block kernel of tc_ws.cu (its limits, gamma >= 4 or r <= 128,
// cover every shape with r <= 256 whose table halves fit 32 projection
// columns each).
#include "device_common.cuh"
#include "tc_common.cuh"
#include "tc_race.cuh"

namespace elsaa {

namespace {

constexpr int kSmemPerSM = 233472;  // 228 KB of shared memory per SM

}  // namespace

bool tc_supported(const Plan &P) {
    if (P.dtype != ELSAA_BF16) return false;
    if (P.d != 64 && P.d != 128) return false;
    if (!(P.b == 32 || P.b == 64 || P.b == 128 || P.b == 256)) return false;
    if (P.gamma > 6 || P.L * P.gamma > 64) return false;
    if (P.r % 16 != 0 || P.r > 256) return false;
    // each half of a row's tables must fit in 32 projection columns
    const int split = tc::table_split(P.L, P.gamma);
    if (split * P.gamma > 32 || (P.L - split) * P.gamma > 32) return false;
    return true;
}

int tc_race_chunks(const Plan &P, int *chunk) {
    // CTAs per SM from the TMEM and shared memory of the key kernel; one
    // wave of chunks over all heads.
    const uint32_t cols = race_keys_ws_cols(P);
    int per_sm = 512 / (int)cols;
    const size_t smem = race_keys_ws_smem(P);
    int by_smem = (int)(kSmemPerSM / (smem + 1024));
    if (by_smem < per_sm) per_sm = by_smem;
    if (per_sm < 1) per_sm = 1;
    long slots = 152L * per_sm;
    int tiles = (P.N + 127) / 128;
    int S = (int)(slots / P.BH);
    if (S < 1) S = 1;
    if (S > tiles) S = tiles;
    int tiles_per = (tiles + S - 1) / S;
    *chunk = tiles_per * 128;
    return (P.N + *chunk - 1) / *chunk;
}

}  // namespace elsaa
