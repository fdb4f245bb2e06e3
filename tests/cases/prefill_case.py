"""One 4096-token Q4_0 call (hidden 2048, 128 experts, top-8, inter 768), 1 layer, from a cold
cache, twice.  Argument: slots per layer (default 128: every expert resident, one wave)."""
import sys
sys.path[:0] = [".", "tests"]
import torch, synth
from mfharness import Ctx, Shape
import paper_2607_09686_gb300 as mf
cfg = synth.CONFIGS["l48e128q4"]
T = 4096
shape = Shape(1, cfg.hidden, cfg.n_experts, cfg.top_k, cfg.inter, cfg.qtype)
slots = int(sys.argv[1]) if len(sys.argv) > 1 else 128
ctx = Ctx(shape, slots, max_tokens=T, workers=16)
r = synth.routes(0, 0, 0, 128, 8, T, 1.2, 0.0)
x = torch.from_numpy(synth.activations(0, 0, 0, 0, T, cfg.hidden)).cuda()
b = torch.from_numpy(synth.plant_bias(r, 128)).cuda()
y = torch.empty(T, cfg.hidden, device="cuda")
mf.mf_prefill_threshold(ctx.h, 2)
for rep in range(2):
    mf.mf_reset(ctx.h)
    mf.mf_moe_forward(ctx.h, 0, x, ctx.wr[0], b, T, y)
torch.cuda.synchronize()
assert mf.mf_check(ctx.h) == 0
print("ok")
ctx.close()
