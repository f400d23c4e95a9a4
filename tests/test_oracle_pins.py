"""The fp64 oracle against its pins (CPU only)."""
import pytest

from oracle import ec2moe_oracle as orc
from tests import pins


@pytest.mark.parametrize("pin", pins.ALL_PINS, ids=lambda p: p.__name__)
def test_pin(pin):
    pin(orc)
